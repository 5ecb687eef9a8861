// SDCC support (§5, self-distillation for conditioning consistency).
//
// Diverging rows. A row diverges when its live prefix differs from its prefix
// on the final compressed walk (App. B Def. "trajectory tree"): some key it
// saw is evicted by a later edit, i.e. there is j <= r with
// r < omega(j) < never. With F(r) = max{omega(j) : j <= r, omega(j) finite}
// (or -1), row r diverges iff F(r) > r: one prefix-max scan of the lifetimes
// per trajectory. These are the rows where SDCC places its KL term.
//
// Forward KL over the vocabulary (Eq. "soft_loss"), on CUDA cores with
// float32 arithmetic (hidden size d <= 256), no logits stored. For pair m the
// teacher row HT[rows_T[m]] and the student row HS[rows_S[m]] give
// zT = hT W^T, zS = hS W^T, and
//   KL_m = sum_v pT (log pT - log pS) = E_pT[zT - zS] - lse(zT) + lse(zS),
// computed online over vocabulary columns: the teacher's (max, sum of
// exp(zT - max), sum of exp(zT - max) (zT - zS)) and the student's (max, sum).
// Backward (teacher stop-gradient): dzS = c (pS - pT), c = lambda * dloss,
// dHS = dzS W (row-stationary), dW = dzS^T HS (vocabulary-stationary).

#include <math.h>

#include "common.cuh"

namespace mw {
namespace {

constexpr int DIV_NT = 1024;

// One block per trajectory: chunks of 1024 rows, warp max-scans, carry.
__global__ void __launch_bounds__(DIV_NT) k_diverging_rows(VisView v, uint8_t* __restrict__ out) {
    __shared__ int wmax[DIV_NT / 32];
    __shared__ int carry_s;
    const int b = blockIdx.x;
    const int64_t tok0 = v.traj_tok[b];
    const int T = v.traj_tok[b + 1] - (int)tok0;
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    if (t == 0) carry_s = -1;
    __syncthreads();
    for (int c0 = 0; c0 < T; c0 += DIV_NT) {
        const int r = c0 + t;
        int x = -1;
        if (r < T) {
            const int om = v.omega[tok0 + r];
            x = om < INT32_MAX ? om : -1;
        }
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x = max(x, y);
        }
        if (lane == 31) wmax[w] = x;
        __syncthreads();
        int f = carry_s;
        for (int q = 0; q < w; ++q) f = max(f, wmax[q]);
        f = max(f, x);
        if (r < T) out[tok0 + r] = f > r ? 1 : 0;
        __syncthreads();
        if (t == DIV_NT - 1) carry_s = f;
        __syncthreads();
    }
}

// Final compressed walk of every trajectory: the never-evicted positions in
// order (omega = never). One inclusive prefix count of survivors per
// trajectory gives each token's walk index (or -1), each row's student row
// (the walk index of the last survivor <= r, i.e. count - 1, -1 when none)
// and the walk length.
__global__ void __launch_bounds__(DIV_NT) k_final_walk(VisView v, int32_t* __restrict__ walk_index,
                                                       int32_t* __restrict__ student_row,
                                                       int32_t* __restrict__ walk_len) {
    __shared__ int wsum[DIV_NT / 32];
    __shared__ int carry_s;
    const int b = blockIdx.x;
    const int64_t tok0 = v.traj_tok[b];
    const int T = v.traj_tok[b + 1] - (int)tok0;
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    if (t == 0) carry_s = 0;
    __syncthreads();
    for (int c0 = 0; c0 < T; c0 += DIV_NT) {
        const int r = c0 + t;
        const int alive = (r < T && v.omega[tok0 + r] == INT32_MAX) ? 1 : 0;
        int x = alive;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) wsum[w] = x;
        __syncthreads();
        int incl = carry_s + x;
        for (int q = 0; q < w; ++q) incl += wsum[q];
        if (r < T) {
            walk_index[tok0 + r] = alive ? incl - 1 : -1;
            student_row[tok0 + r] = incl - 1;
        }
        __syncthreads();
        if (t == DIV_NT - 1) carry_s = incl;
        __syncthreads();
    }
    if (t == 0) walk_len[b] = carry_s;
}

// ---------------------------------------------------------------- forward KL

constexpr int KR = 8;    // pairs per forward block
constexpr int KH = 16;   // pairs per dHS block
constexpr int KWV = 32;  // vocabulary rows per dW block
constexpr int KWR = 32;  // pairs per dW step

// Online (max, sum) of exp, and the teacher's weighted sum a = sum exp(z - max) x.
struct TStat {
    float m, l, a;
};
__device__ __forceinline__ void tstat_merge(TStat& s, float m2, float l2, float a2) {
    const float mn = fmaxf(s.m, m2);
    if (mn == -INFINITY) return;
    const float e1 = expf(s.m - mn), e2 = expf(m2 - mn);
    s.l = s.l * e1 + l2 * e2;
    s.a = s.a * e1 + a2 * e2;
    s.m = mn;
}
__device__ __forceinline__ void smerge(float& m, float& l, float m2, float l2) {
    const float mn = fmaxf(m, m2);
    if (mn == -INFINITY) return;
    l = l * expf(m - mn) + l2 * expf(m2 - mn);
    m = mn;
}

// Stage the rows of up to n pairs into shared memory: zero past M, and zero
// for a row index outside [0, N), which raises the bounds flag.
template <typename Tin>
__device__ __forceinline__ void stage_rows(float* dst, const Tin* __restrict__ H, const int32_t* __restrict__ rows,
                                           int m0, int n, int M, int N, int d, int32_t* status) {
    for (int x = threadIdx.x; x < n * d; x += blockDim.x) {
        const int r = x / d, k = x % d;
        const int t = m0 + r < M ? checked_index(rows[m0 + r], N) : 0;
        if (t < 0 && k == 0) flag_bounds(status);
        dst[x] = (m0 + r < M && t >= 0) ? ld_f(H + (int64_t)t * d + k) : 0.f;
    }
}

// grid ceil(M / KR), block 256; writes kl[m], lseT[m], lseS[m].
template <typename Tin>
__global__ void __launch_bounds__(256) k_kl_fwd_simt(int M, int N_T, int N_S, int d, int Vocab,
                                                    const Tin* __restrict__ HT, const int32_t* __restrict__ rowsT,
                                                    const Tin* __restrict__ HS, const int32_t* __restrict__ rowsS,
                                                    const Tin* __restrict__ W, float* __restrict__ kl,
                                                    float* __restrict__ lseT, float* __restrict__ lseS,
                                                    int32_t* __restrict__ status) {
    extern __shared__ float sh[];
    float* ht = sh;            // [KR][d]
    float* hs = sh + KR * d;   // [KR][d]
    __shared__ float red[KR][8][5];
    const int m0 = blockIdx.x * KR;
    stage_rows(ht, HT, rowsT, m0, KR, M, N_T, d, status);
    stage_rows(hs, HS, rowsS, m0, KR, M, N_S, d, status);
    __syncthreads();
    TStat t[KR];
    float ms[KR], ls[KR];
#pragma unroll
    for (int r = 0; r < KR; ++r) {
        t[r].m = -INFINITY; t[r].l = 0.f; t[r].a = 0.f;
        ms[r] = -INFINITY; ls[r] = 0.f;
    }
    for (int v = threadIdx.x; v < Vocab; v += blockDim.x) {
        float zt[KR], zs[KR];
#pragma unroll
        for (int r = 0; r < KR; ++r) zt[r] = zs[r] = 0.f;
        const Tin* wrow = W + (int64_t)v * d;
        for (int k = 0; k < d; ++k) {
            const float w = ld_f(wrow + k);
#pragma unroll
            for (int r = 0; r < KR; ++r) {
                zt[r] = fmaf(ht[r * d + k], w, zt[r]);
                zs[r] = fmaf(hs[r * d + k], w, zs[r]);
            }
        }
#pragma unroll
        for (int r = 0; r < KR; ++r) {
            tstat_merge(t[r], zt[r], 1.f, zt[r] - zs[r]);
            smerge(ms[r], ls[r], zs[r], 1.f);
        }
    }
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
    for (int r = 0; r < KR; ++r) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float m2 = __shfl_xor_sync(0xffffffffu, t[r].m, o), l2 = __shfl_xor_sync(0xffffffffu, t[r].l, o),
                        a2 = __shfl_xor_sync(0xffffffffu, t[r].a, o);
            tstat_merge(t[r], m2, l2, a2);
            const float n2 = __shfl_xor_sync(0xffffffffu, ms[r], o), k2 = __shfl_xor_sync(0xffffffffu, ls[r], o);
            smerge(ms[r], ls[r], n2, k2);
        }
        if (lane == 0) {
            red[r][w][0] = t[r].m; red[r][w][1] = t[r].l; red[r][w][2] = t[r].a;
            red[r][w][3] = ms[r]; red[r][w][4] = ls[r];
        }
    }
    __syncthreads();
    if (threadIdx.x < KR && m0 + threadIdx.x < M) {
        const int r = threadIdx.x;
        TStat s{-INFINITY, 0.f, 0.f};
        float mm = -INFINITY, ll = 0.f;
        for (int q = 0; q < 8; ++q) {
            tstat_merge(s, red[r][q][0], red[r][q][1], red[r][q][2]);
            smerge(mm, ll, red[r][q][3], red[r][q][4]);
        }
        const float lt = s.m + logf(s.l), lsv = mm + logf(ll);
        lseT[m0 + r] = lt;
        lseS[m0 + r] = lsv;
        kl[m0 + r] = s.a / s.l - lt + lsv;
    }
}

// loss = lambda * sum_m kl[m], one block of 1024 threads in a fixed order.
__global__ void k_kl_loss(int M, const float* __restrict__ kl, float lam, float* __restrict__ loss) {
    __shared__ float red[32];
    float part = 0.f;
    for (int m = threadIdx.x; m < M; m += blockDim.x) part += kl[m];
    part = warp_sum(part);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = part;
    __syncthreads();
    if (threadIdx.x < 32) {
        float x = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
        x = warp_sum(x);
        if (threadIdx.x == 0) *loss = lam * x;
    }
}

// dHS: grid ceil(M / KH), block 256 (d <= 256); vocabulary tiles of 256.
template <typename Tin>
__global__ void __launch_bounds__(256) k_kl_dh_simt(int M, int N_T, int N_S, int d, int Vocab,
                                                   const Tin* __restrict__ HT, const int32_t* __restrict__ rowsT,
                                                   const Tin* __restrict__ HS, const int32_t* __restrict__ rowsS,
                                                   const Tin* __restrict__ W, const float* __restrict__ lseT,
                                                   const float* __restrict__ lseS, float c, int accumulate,
                                                   Tin* __restrict__ dHS, int32_t* __restrict__ status) {
    extern __shared__ float sh[];
    float* ht = sh;                // [KH][d]
    float* hs = sh + KH * d;       // [KH][d]
    float* dzs = hs + KH * d;      // [KH][256]
    __shared__ float slt[KH], sls[KH], sc[KH];
    const int m0 = blockIdx.x * KH;
    stage_rows(ht, HT, rowsT, m0, KH, M, N_T, d, status);
    stage_rows(hs, HS, rowsS, m0, KH, M, N_S, d, status);
    if (threadIdx.x < KH) {
        const bool ok = m0 + threadIdx.x < M;
        slt[threadIdx.x] = ok ? lseT[m0 + threadIdx.x] : 0.f;
        sls[threadIdx.x] = ok ? lseS[m0 + threadIdx.x] : 0.f;
        sc[threadIdx.x] = ok ? c : 0.f;
    }
    __syncthreads();
    float acc[KH];
#pragma unroll
    for (int r = 0; r < KH; ++r) acc[r] = 0.f;
    for (int v0 = 0; v0 < Vocab; v0 += 256) {
        const int v = v0 + threadIdx.x;
        if (v < Vocab) {
            float zt[KH], zs[KH];
#pragma unroll
            for (int r = 0; r < KH; ++r) zt[r] = zs[r] = 0.f;
            const Tin* wrow = W + (int64_t)v * d;
            for (int k = 0; k < d; ++k) {
                const float w = ld_f(wrow + k);
#pragma unroll
                for (int r = 0; r < KH; ++r) {
                    zt[r] = fmaf(ht[r * d + k], w, zt[r]);
                    zs[r] = fmaf(hs[r * d + k], w, zs[r]);
                }
            }
#pragma unroll
            for (int r = 0; r < KH; ++r)
                dzs[r * 256 + threadIdx.x] = sc[r] * (expf(zs[r] - sls[r]) - expf(zt[r] - slt[r]));
        } else {
#pragma unroll
            for (int r = 0; r < KH; ++r) dzs[r * 256 + threadIdx.x] = 0.f;
        }
        __syncthreads();
        const int k = threadIdx.x;
        if (k < d) {
            const int nv = min(256, Vocab - v0);
            for (int vv = 0; vv < nv; ++vv) {
                const float w = ld_f(W + (int64_t)(v0 + vv) * d + k);
#pragma unroll
                for (int r = 0; r < KH; ++r) acc[r] = fmaf(dzs[r * 256 + vv], w, acc[r]);
            }
        }
        __syncthreads();
    }
    if (threadIdx.x < d) {
#pragma unroll
        for (int r = 0; r < KH; ++r)
            if (m0 + r < M && checked_index(rowsS[m0 + r], N_S) >= 0) {
                Tin* dst = dHS + (int64_t)rowsS[m0 + r] * d + threadIdx.x;
                st_f(dst, accumulate ? ld_f(dst) + acc[r] : acc[r]);
            }
    }
}

// dW: grid ceil(Vocab / KWV), block 256 (d <= 256).
template <typename Tin>
__global__ void __launch_bounds__(256) k_kl_dw_simt(int M, int N_T, int N_S, int d, int Vocab,
                                                   const Tin* __restrict__ HT, const int32_t* __restrict__ rowsT,
                                                   const Tin* __restrict__ HS, const int32_t* __restrict__ rowsS,
                                                   const Tin* __restrict__ W, const float* __restrict__ lseT,
                                                   const float* __restrict__ lseS, float c, int accumulate,
                                                   float* __restrict__ dW, int32_t* __restrict__ status) {
    extern __shared__ float sh[];
    float* ws = sh;                 // [KWV][d]
    float* ht = sh + KWV * d;       // [KWR][d]
    float* hs = ht + KWR * d;       // [KWR][d]
    float* dzs = hs + KWR * d;      // [KWR][KWV]
    __shared__ float slt[KWR], sls[KWR], sc[KWR];
    const int v0 = blockIdx.x * KWV;
    for (int x = threadIdx.x; x < KWV * d; x += blockDim.x) {
        const int r = x / d, k = x % d;
        ws[x] = (v0 + r < Vocab) ? ld_f(W + (int64_t)(v0 + r) * d + k) : 0.f;
    }
    float acc[KWV];
#pragma unroll
    for (int q = 0; q < KWV; ++q) acc[q] = 0.f;
    for (int m0 = 0; m0 < M; m0 += KWR) {
        __syncthreads();
        stage_rows(ht, HT, rowsT, m0, KWR, M, N_T, d, status);
        stage_rows(hs, HS, rowsS, m0, KWR, M, N_S, d, status);
        if (threadIdx.x < KWR) {
            const bool ok = m0 + threadIdx.x < M;
            slt[threadIdx.x] = ok ? lseT[m0 + threadIdx.x] : 0.f;
            sls[threadIdx.x] = ok ? lseS[m0 + threadIdx.x] : 0.f;
            sc[threadIdx.x] = ok ? c : 0.f;
        }
        __syncthreads();
        {   // 32 x 32 logits of both: thread -> (pair r, 4 vocabulary columns)
            const int r = threadIdx.x >> 3, c0 = (threadIdx.x & 7) * 4;
            float zt[4] = {0.f, 0.f, 0.f, 0.f}, zs[4] = {0.f, 0.f, 0.f, 0.f};
            for (int k = 0; k < d; ++k) {
                const float tv = ht[r * d + k], sv = hs[r * d + k];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float wv = ws[(c0 + q) * d + k];
                    zt[q] = fmaf(tv, wv, zt[q]);
                    zs[q] = fmaf(sv, wv, zs[q]);
                }
            }
#pragma unroll
            for (int q = 0; q < 4; ++q)
                dzs[r * KWV + c0 + q] = sc[r] * (expf(zs[q] - sls[r]) - expf(zt[q] - slt[r]));
        }
        __syncthreads();
        const int k = threadIdx.x;
        if (k < d) {
            for (int r = 0; r < KWR; ++r) {
                const float hv = hs[r * d + k];
#pragma unroll
                for (int q = 0; q < KWV; ++q) acc[q] = fmaf(dzs[r * KWV + q], hv, acc[q]);
            }
        }
    }
    if (threadIdx.x < d) {
#pragma unroll
        for (int q = 0; q < KWV; ++q)
            if (v0 + q < Vocab) {
                float* dst = dW + (int64_t)(v0 + q) * d + threadIdx.x;
                *dst = accumulate ? *dst + acc[q] : acc[q];
            }
    }
}

template <typename Tin>
mw_status kl_fwd_t(const void* HT, const int32_t* rowsT, const void* HS, const int32_t* rowsS, int M,
                   const void* W, int N_T, int N_S, int d, int Vocab, float lam, float* kl, float* loss, float* lseT,
                   float* lseS, int32_t* status, cudaStream_t s) {
    const size_t smem = sizeof(float) * 2 * KR * d;
    mw_status st = cuda_status(
        cudaFuncSetAttribute(k_kl_fwd_simt<Tin>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    if (st != MW_OK) return st;
    count_launches(1);
    k_kl_fwd_simt<Tin><<<(unsigned)ceil_div(M, KR), 256, smem, s>>>(M, N_T, N_S, d, Vocab, (const Tin*)HT, rowsT,
                                                                    (const Tin*)HS, rowsS, (const Tin*)W, kl,
                                                                    lseT, lseS, status);
    if ((st = launch_status()) != MW_OK) return st;
    count_launches(1);
    k_kl_loss<<<1, 1024, 0, s>>>(M, kl, lam, loss);
    return launch_status();
}

template <typename Tin>
mw_status kl_bwd_t(const void* HT, const int32_t* rowsT, const void* HS, const int32_t* rowsS, int M,
                   const void* W, int N_T, int N_S, int d, int Vocab, float c, const float* lseT, const float* lseS,
                   int accumulate, void* dHS, float* dW, int32_t* status, cudaStream_t s) {
    mw_status st = MW_OK;
    if (!accumulate && (st = cuda_status(cudaMemsetAsync(dHS, 0, sizeof(Tin) * (size_t)N_S * d, s))) != MW_OK)
        return st;
    if (M == 0)
        return accumulate ? MW_OK : cuda_status(cudaMemsetAsync(dW, 0, sizeof(float) * (size_t)Vocab * d, s));
    const size_t smem_h = sizeof(float) * (2 * KH * d + KH * 256);
    const size_t smem_w = sizeof(float) * (KWV * d + 2 * KWR * d + KWR * KWV);
    if ((st = cuda_status(cudaFuncSetAttribute(k_kl_dh_simt<Tin>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)smem_h))) != MW_OK)
        return st;
    if ((st = cuda_status(cudaFuncSetAttribute(k_kl_dw_simt<Tin>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)smem_w))) != MW_OK)
        return st;
    count_launches(2);
    k_kl_dh_simt<Tin><<<(unsigned)ceil_div(M, KH), 256, smem_h, s>>>(M, N_T, N_S, d, Vocab, (const Tin*)HT, rowsT,
                                                                     (const Tin*)HS, rowsS, (const Tin*)W, lseT,
                                                                     lseS, c, accumulate, (Tin*)dHS, status);
    k_kl_dw_simt<Tin><<<(unsigned)ceil_div(Vocab, KWV), 256, smem_w, s>>>(M, N_T, N_S, d, Vocab, (const Tin*)HT,
                                                                          rowsT, (const Tin*)HS, rowsS,
                                                                          (const Tin*)W, lseT, lseS, c, accumulate,
                                                                          dW, status);
    return launch_status();
}

}  // namespace
}  // namespace mw

using namespace mw;

extern "C" mw_status mw_final_walk(const mw_vis_layout* L, const void* vis, int32_t* walk_index,
                                   int32_t* student_row, int32_t* walk_len, void* stream) {
    if (L && L->kind != MW_VIEWS_EDITS) return MW_ESHAPE;   // needs single-interval lifetimes
    if (!L) return MW_EINVAL;
    if (L->n_traj == 0) return MW_OK;
    if (!vis || !walk_len || (L->total_tokens > 0 && (!walk_index || !student_row))) return MW_EINVAL;
    count_launches(1);
    k_final_walk<<<(unsigned)L->n_traj, DIV_NT, 0, (cudaStream_t)stream>>>(make_view(L, vis), walk_index,
                                                                          student_row, walk_len);
    return launch_status();
}

namespace mw {
bool lm_bwd_tc_supported(int d);
int64_t kl_tc_ws(int M, int d);
mw_status kl_fwd_tc(const void*, const int32_t*, const void*, const int32_t*, int, const void*, int, int, int, int,
                    float*, void*, cudaStream_t);
mw_status kl_bwd_tc(const int32_t*, int, const void*, int, int, int, float, void*, int, void*, float*,
                    cudaStream_t);
int32_t* kl_tc_status(int M, int d, void* ws);
}  // namespace mw

// bf16 with a hidden size the LM head's CTA groups can split runs on the
// tensor cores; fp32 (and bf16 with other d <= 256) on CUDA cores.
static bool kl_tc(int d, int dtype) { return dtype == MW_BF16 && lm_bwd_tc_supported(d); }

static mw_status kl_args(int M, int N_T, int N_S, int d, int Vocab, int dtype) {
    if (M < 0 || N_T < 0 || N_S < 0 || d <= 0 || Vocab <= 0) return MW_ESHAPE;
    if (M > N_S) return MW_ESHAPE;        // student rows are distinct; teacher rows may repeat
    if (M > 0 && N_T == 0) return MW_ESHAPE;
    if (dtype != MW_F32 && dtype != MW_BF16) return MW_EDTYPE;
    if (!kl_tc(d, dtype) && d > 256) return MW_ESHAPE;
    return MW_OK;
}

// Workspace: CUDA cores, lse of the teacher and of the student per pair and
// the status words; tensor cores, the fused passes' arrays (see kl_tc_ws).
static int32_t* kl_simt_status(int M, void* ws) { return at<int32_t>(ws, 2 * align256(4 * (int64_t)M)); }

extern "C" mw_status mw_forward_kl_ws(int M, int d, int Vocab, int dtype, size_t* bytes) {
    if (!bytes) return MW_EINVAL;
    mw_status st = kl_args(M, M, M, d, Vocab, dtype);
    if (st != MW_OK) return st;
    *bytes = kl_tc(d, dtype) ? (size_t)kl_tc_ws(M, d) : (size_t)(2 * align256(4 * (int64_t)M) + 256);
    return MW_OK;
}

extern "C" mw_status mw_forward_kl_check_status(int M, int d, int Vocab, int dtype, void* ws, void* stream) {
    mw_status st = kl_args(M, M, M, d, Vocab, dtype);
    if (st != MW_OK) return st;
    if (!ws) return MW_EINVAL;
    int32_t h[8];
    if ((st = cuda_status(cudaMemcpyAsync(h, kl_tc(d, dtype) ? kl_tc_status(M, d, ws) : kl_simt_status(M, ws),
                                          sizeof(h), cudaMemcpyDeviceToHost, (cudaStream_t)stream))) != MW_OK)
        return st;
    if ((st = cuda_status(cudaStreamSynchronize((cudaStream_t)stream))) != MW_OK) return st;
    return h[1] ? MW_ETIMEOUT : h[0] ? MW_EDEVICE : MW_OK;
}

extern "C" mw_status mw_forward_kl_fwd(const void* HT, const int32_t* rows_T, const void* HS, const int32_t* rows_S,
                                       int M, const void* W, int N_T, int N_S, int d, int Vocab, int dtype,
                                       float lam, float* kl, float* loss, void* ws, void* stream) {
    mw_status st = kl_args(M, N_T, N_S, d, Vocab, dtype);
    if (st != MW_OK) return st;
    if (!(lam >= 0.f) || !isfinite(lam)) return MW_EINVAL;
    if (!loss || !ws) return MW_EINVAL;
    if (M > 0 && (!HT || !rows_T || !HS || !rows_S || !W || !kl)) return MW_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    float* lseT = at<float>(ws, 0);
    float* lseS = at<float>(ws, align256(4 * (int64_t)M));
    int32_t* status = kl_tc(d, dtype) ? kl_tc_status(M, d, ws) : kl_simt_status(M, ws);
    if ((st = cuda_status(cudaMemsetAsync(status, 0, 32, s))) != MW_OK) return st;
    if (M == 0) {
        count_launches(1);
        k_kl_loss<<<1, 1024, 0, s>>>(0, kl, lam, loss);
        return launch_status();
    }
    if (kl_tc(d, dtype)) {
        if ((st = kl_fwd_tc(HT, rows_T, HS, rows_S, M, W, N_T, N_S, d, Vocab, kl, ws, s)) != MW_OK) return st;
        count_launches(1);
        k_kl_loss<<<1, 1024, 0, s>>>(M, kl, lam, loss);
        return launch_status();
    }
    return dtype == MW_F32 ? kl_fwd_t<float>(HT, rows_T, HS, rows_S, M, W, N_T, N_S, d, Vocab, lam, kl, loss, lseT,
                                             lseS, status, s)
                           : kl_fwd_t<__nv_bfloat16>(HT, rows_T, HS, rows_S, M, W, N_T, N_S, d, Vocab, lam, kl, loss,
                                                     lseT, lseS, status, s);
}

extern "C" mw_status mw_forward_kl_bwd(const void* HT, const int32_t* rows_T, const void* HS, const int32_t* rows_S,
                                       int M, const void* W, int N_T, int N_S, int d, int Vocab, int dtype,
                                       float lam, float dloss, int accumulate, void* ws, void* dHS, float* dW,
                                       void* stream) {
    mw_status st = kl_args(M, N_T, N_S, d, Vocab, dtype);
    if (st != MW_OK) return st;
    if (!(lam >= 0.f) || !isfinite(lam) || !isfinite(dloss)) return MW_EINVAL;
    if (!ws || !dW || (N_S > 0 && !dHS)) return MW_EINVAL;
    if (M > 0 && (!HT || !rows_T || !HS || !rows_S || !W)) return MW_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    const float* lseT = at<float>(ws, 0);
    const float* lseS = at<float>(ws, align256(4 * (int64_t)M));
    const float c = lam * dloss;
    if (kl_tc(d, dtype)) return kl_bwd_tc(rows_S, M, W, N_S, d, Vocab, c, ws, accumulate, dHS, dW, s);
    int32_t* status = kl_simt_status(M, ws);   // reset by the forward; the backward adds to it
    return dtype == MW_F32
               ? kl_bwd_t<float>(HT, rows_T, HS, rows_S, M, W, N_T, N_S, d, Vocab, c, lseT, lseS, accumulate, dHS,
                                 dW, status, s)
               : kl_bwd_t<__nv_bfloat16>(HT, rows_T, HS, rows_S, M, W, N_T, N_S, d, Vocab, c, lseT, lseS,
                                         accumulate, dHS, dW, status, s);
}

extern "C" mw_status mw_diverging_rows(const mw_vis_layout* L, const void* vis, uint8_t* out, void* stream) {
    if (L && L->kind != MW_VIEWS_EDITS) return MW_ESHAPE;   // needs single-interval lifetimes
    if (!L) return MW_EINVAL;
    if (L->total_tokens == 0) return MW_OK;
    if (!vis || !out) return MW_EINVAL;
    count_launches(1);
    k_diverging_rows<<<(unsigned)L->n_traj, DIV_NT, 0, (cudaStream_t)stream>>>(make_view(L, vis), out);
    return launch_status();
}
