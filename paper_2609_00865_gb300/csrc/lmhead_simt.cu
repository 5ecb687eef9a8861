// Fused LM-head log-prob and clipped policy loss on CUDA cores, float32
// arithmetic (the float32 path; hidden size d <= 256). No logits tensor is
// stored: logits are recomputed tile by tile in every pass.
//
// Forward:  per loss row m, lse_m = log sum_v exp(H_t . W_v), lp_m = z_tgt - lse_m.
// Loss:     ratio, PPO/GRPO clipped surrogate, mean over loss rows, g = dL/dlp
//           (App. B.4 "Pitfall A, RL view"; App. F.1 clip range).
// Backward: dz = g (onehot - softmax); dH = dz W (row-stationary pass),
//           dW = dz^T H (vocab-stationary pass).

#include <math.h>

#include "common.cuh"

namespace mw {

// Shared by both LM-head paths: ratio, clipped surrogate, g, mean loss.
// With lp_ref (may be null) each loss row also adds beta times the
// low-variance KL estimate to the reference policy (App. F.1),
//   k3 = exp(d) - d - 1 = expm1(d) - d,  d = lp_ref - lp,  dk3/dlp = -expm1(d).
// One block of 1024 threads; the mean is reduced in a fixed order.
__global__ void k_loss_epilogue(int M, const float* __restrict__ lp, const float* __restrict__ lp_old,
                                const float* __restrict__ adv, float eps_lo, float eps_hi,
                                const float* __restrict__ lp_ref, float beta, float* __restrict__ ratio,
                                float* __restrict__ gsave, float* __restrict__ loss) {
    __shared__ float red[32];
    float part = 0.f;
    const float invM = M > 0 ? 1.f / (float)M : 0.f;
    for (int m = threadIdx.x; m < M; m += blockDim.x) {
        const float r = expf(lp[m] - lp_old[m]);
        const float A = adv[m];
        const float unclipped = r * A;
        const float clipped = fminf(fmaxf(r, 1.f - eps_lo), 1.f + eps_hi) * A;
        float g = (clipped < unclipped) ? 0.f : -A * r * invM;
        part += -fminf(unclipped, clipped);
        if (lp_ref) {
            const float d = lp_ref[m] - lp[m];
            const float em1 = expm1f(d);
            part += beta * (em1 - d);
            g -= beta * em1 * invM;
        }
        ratio[m] = r;
        gsave[m] = g;
    }
    part = warp_sum(part);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = part;
    __syncthreads();
    if (threadIdx.x < 32) {
        float x = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
        x = warp_sum(x);
        if (threadIdx.x == 0) *loss = x * invM;
    }
}

// Eq. "logdiff": mean_m |lp_train[m] - lp_rollout[m]|, one block of 1024
// threads in a fixed order (0 for M = 0).
__global__ void k_logdiff(int M, const float* __restrict__ a, const float* __restrict__ b, float* __restrict__ out) {
    __shared__ float red[32];
    float part = 0.f;
    for (int m = threadIdx.x; m < M; m += blockDim.x) part += fabsf(a[m] - b[m]);
    part = warp_sum(part);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = part;
    __syncthreads();
    if (threadIdx.x < 32) {
        float x = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
        x = warp_sum(x);
        if (threadIdx.x == 0) *out = M > 0 ? x / (float)M : 0.f;
    }
}

namespace {

constexpr int FR = 16;  // loss rows per block (forward / dH)

// Online (max, sum-exp) merge.
__device__ __forceinline__ void lse_merge(float& m, float& l, float m2, float l2) {
    const float mn = fmaxf(m, m2);
    if (mn == -INFINITY) return;
    l = l * expf(m - mn) + l2 * expf(m2 - mn);
    m = mn;
}

// Physical rows and targets of loss rows m0 .. m0 + n - 1 into shared memory:
// -1 past M; a row outside [0, N) or a target outside [0, Vocab) also gives
// row and target -1 and raises the bounds flag: the row then reads as zero
// and its dH row is not written.
__device__ __forceinline__ void stage_index(int* srow, int* stg, const int32_t* __restrict__ rows,
                                            const int32_t* __restrict__ targets, int m0, int n, int M, int N,
                                            int Vocab, int32_t* status) {
    if (threadIdx.x < n) {
        const int m = m0 + threadIdx.x;
        int r = -1, t = -1;
        if (m < M) {
            r = checked_index(rows[m], N);
            if (r >= 0) t = checked_index(targets[r], Vocab);
            if (t < 0) {
                flag_bounds(status);
                r = -1;
            }
        }
        srow[threadIdx.x] = r;
        stg[threadIdx.x] = t;
    }
}

template <typename Tin>
__device__ __forceinline__ void stage_hidden(float* hs, const Tin* __restrict__ H, const int* srow, int n, int d) {
    for (int x = threadIdx.x; x < n * d; x += blockDim.x) {
        const int r = x / d, k = x % d;
        hs[x] = srow[r] >= 0 ? ld_f(H + (int64_t)srow[r] * d + k) : 0.f;
    }
}

template <typename Tin>
__device__ __forceinline__ void row_logits(const float* __restrict__ hs, int d, const Tin* __restrict__ wrow,
                                           float* z) {
#pragma unroll
    for (int r = 0; r < FR; ++r) z[r] = 0.f;
    for (int k = 0; k < d; ++k) {
        const float w = ld_f(wrow + k);
#pragma unroll
        for (int r = 0; r < FR; ++r) z[r] = fmaf(hs[r * d + k], w, z[r]);
    }
}

// grid: ceil(M / FR); block 256. Writes lse[m] and zt[m] (target logit).
template <typename Tin>
__global__ void __launch_bounds__(256) k_lm_fwd_simt(int M, int N, int d, int Vocab, const Tin* __restrict__ H,
                                                    const Tin* __restrict__ W, const int32_t* __restrict__ targets,
                                                    const int32_t* __restrict__ rows, float* __restrict__ lse,
                                                    float* __restrict__ zt, int32_t* __restrict__ status) {
    extern __shared__ float hs[];  // [FR][d]
    __shared__ float sm[FR][8], sl[FR][8];
    __shared__ int tg[FR], srow[FR];
    const int m0 = blockIdx.x * FR;
    stage_index(srow, tg, rows, targets, m0, FR, M, N, Vocab, status);
    __syncthreads();
    stage_hidden(hs, H, srow, FR, d);
    __syncthreads();
    float m[FR], l[FR], z[FR];
#pragma unroll
    for (int r = 0; r < FR; ++r) { m[r] = -INFINITY; l[r] = 0.f; }
    for (int v = threadIdx.x; v < Vocab; v += blockDim.x) {
        row_logits<Tin>(hs, d, W + (int64_t)v * d, z);
#pragma unroll
        for (int r = 0; r < FR; ++r) {
            lse_merge(m[r], l[r], z[r], 1.f);
            if (v == tg[r]) zt[m0 + r] = z[r];
        }
    }
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
    for (int r = 0; r < FR; ++r) {
        float mm = m[r], ll = l[r];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float m2 = __shfl_xor_sync(0xffffffffu, mm, o), l2 = __shfl_xor_sync(0xffffffffu, ll, o);
            lse_merge(mm, ll, m2, l2);
        }
        if (lane == 0) { sm[r][w] = mm; sl[r][w] = ll; }
    }
    __syncthreads();
    if (threadIdx.x < FR && m0 + threadIdx.x < M) {
        float mm = -INFINITY, ll = 0.f;
        for (int q = 0; q < 8; ++q) lse_merge(mm, ll, sm[threadIdx.x][q], sl[threadIdx.x][q]);
        lse[m0 + threadIdx.x] = mm + logf(ll);
    }
}

__global__ void k_lp_from_zt(int M, const float* __restrict__ zt, const float* __restrict__ lse,
                             float* __restrict__ lp) {
    const int m = blockIdx.x * blockDim.x + threadIdx.x;
    if (m < M) lp[m] = zt[m] - lse[m];
}

// dH: grid ceil(M / FR), block 256 (d <= 256). Vocab tiles of 256 columns.
template <typename Tin>
__global__ void __launch_bounds__(256) k_lm_dh_simt(int M, int N, int d, int Vocab, const Tin* __restrict__ H,
                                                   const Tin* __restrict__ W, const int32_t* __restrict__ targets,
                                                   const int32_t* __restrict__ rows, const float* __restrict__ lse,
                                                   const float* __restrict__ g, float dloss, Tin* __restrict__ dH,
                                                   int32_t* __restrict__ status) {
    extern __shared__ float sh[];
    float* hs = sh;               // [FR][d]
    float* dzs = sh + FR * d;     // [FR][256]
    __shared__ int tg[FR], srow[FR];
    __shared__ float slse[FR], sg[FR];
    const int m0 = blockIdx.x * FR;
    stage_index(srow, tg, rows, targets, m0, FR, M, N, Vocab, status);
    if (threadIdx.x < FR) {
        const bool ok = m0 + threadIdx.x < M;
        slse[threadIdx.x] = ok ? lse[m0 + threadIdx.x] : 0.f;
        sg[threadIdx.x] = ok ? g[m0 + threadIdx.x] * dloss : 0.f;
    }
    __syncthreads();
    stage_hidden(hs, H, srow, FR, d);
    __syncthreads();
    float acc[FR], z[FR];
#pragma unroll
    for (int r = 0; r < FR; ++r) acc[r] = 0.f;
    for (int v0 = 0; v0 < Vocab; v0 += 256) {
        const int v = v0 + threadIdx.x;
        if (v < Vocab) {
            row_logits<Tin>(hs, d, W + (int64_t)v * d, z);
#pragma unroll
            for (int r = 0; r < FR; ++r)
                dzs[r * 256 + threadIdx.x] = sg[r] * ((v == tg[r] ? 1.f : 0.f) - expf(z[r] - slse[r]));
        } else {
#pragma unroll
            for (int r = 0; r < FR; ++r) dzs[r * 256 + threadIdx.x] = 0.f;
        }
        __syncthreads();
        const int k = threadIdx.x;
        if (k < d) {
            const int nv = min(256, Vocab - v0);
            for (int vv = 0; vv < nv; ++vv) {
                const float w = ld_f(W + (int64_t)(v0 + vv) * d + k);
#pragma unroll
                for (int r = 0; r < FR; ++r) acc[r] = fmaf(dzs[r * 256 + vv], w, acc[r]);
            }
        }
        __syncthreads();
    }
    if (threadIdx.x < d) {
#pragma unroll
        for (int r = 0; r < FR; ++r)
            if (srow[r] >= 0) st_f(dH + (int64_t)srow[r] * d + threadIdx.x, acc[r]);
    }
}

constexpr int WV = 32;  // vocab rows per dW block
constexpr int WR = 32;  // loss rows per dW step

// dW: grid ceil(Vocab / WV), block 256 (d <= 256).
template <typename Tin>
__global__ void __launch_bounds__(256) k_lm_dw_simt(int M, int N, int d, int Vocab, const Tin* __restrict__ H,
                                                   const Tin* __restrict__ W, const int32_t* __restrict__ targets,
                                                   const int32_t* __restrict__ rows, const float* __restrict__ lse,
                                                   const float* __restrict__ g, float dloss, float* __restrict__ dW,
                                                   int32_t* __restrict__ status) {
    extern __shared__ float sh[];
    float* ws = sh;                // [WV][d]
    float* hs = sh + WV * d;       // [WR][d]
    float* dzs = hs + WR * d;      // [WR][WV]
    __shared__ int tg[WR], srow[WR];
    __shared__ float slse[WR], sg[WR];
    const int v0 = blockIdx.x * WV;
    for (int x = threadIdx.x; x < WV * d; x += blockDim.x) {
        const int r = x / d, k = x % d;
        ws[x] = (v0 + r < Vocab) ? ld_f(W + (int64_t)(v0 + r) * d + k) : 0.f;
    }
    float acc[WV];
#pragma unroll
    for (int q = 0; q < WV; ++q) acc[q] = 0.f;
    for (int m0 = 0; m0 < M; m0 += WR) {
        __syncthreads();
        stage_index(srow, tg, rows, targets, m0, WR, M, N, Vocab, status);
        if (threadIdx.x < WR) {
            const bool ok = m0 + threadIdx.x < M;
            slse[threadIdx.x] = ok ? lse[m0 + threadIdx.x] : 0.f;
            sg[threadIdx.x] = ok ? g[m0 + threadIdx.x] * dloss : 0.f;
        }
        __syncthreads();
        stage_hidden(hs, H, srow, WR, d);
        __syncthreads();
        {   // 32 x 32 logits: thread -> (row r, 4 vocab columns)
            const int r = threadIdx.x >> 3, c0 = (threadIdx.x & 7) * 4;
            float z[4] = {0.f, 0.f, 0.f, 0.f};
            for (int k = 0; k < d; ++k) {
                const float hv = hs[r * d + k];
#pragma unroll
                for (int q = 0; q < 4; ++q) z[q] = fmaf(hv, ws[(c0 + q) * d + k], z[q]);
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int v = v0 + c0 + q;
                dzs[r * WV + c0 + q] = sg[r] * ((v == tg[r] ? 1.f : 0.f) - expf(z[q] - slse[r]));
            }
        }
        __syncthreads();
        const int k = threadIdx.x;
        if (k < d) {
            for (int r = 0; r < WR; ++r) {
                const float hv = hs[r * d + k];
#pragma unroll
                for (int q = 0; q < WV; ++q) acc[q] = fmaf(dzs[r * WV + q], hv, acc[q]);
            }
        }
    }
    if (threadIdx.x < d) {
#pragma unroll
        for (int q = 0; q < WV; ++q)
            if (v0 + q < Vocab) dW[(int64_t)(v0 + q) * d + threadIdx.x] = acc[q];
    }
}

template <typename Tin>
mw_status fwd_t(const void* H, const void* W, const int32_t* targets, const int32_t* rows, int M, int N, int d,
                int Vocab, float* lse, float* zt, float* lp, int32_t* status, cudaStream_t s) {
    const size_t smem = sizeof(float) * FR * d;
    count_launches(2);
    cudaFuncSetAttribute(k_lm_fwd_simt<Tin>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    k_lm_fwd_simt<Tin><<<(unsigned)ceil_div(M, FR), 256, smem, s>>>(M, N, d, Vocab, (const Tin*)H, (const Tin*)W,
                                                                    targets, rows, lse, zt, status);
    k_lp_from_zt<<<(unsigned)ceil_div(M, 256), 256, 0, s>>>(M, zt, lse, lp);
    return launch_status();
}

template <typename Tin>
mw_status bwd_t(const void* H, const void* W, const int32_t* targets, const int32_t* rows, int M, int N, int d,
                int Vocab, const float* lse, const float* g, float dloss, void* dH, float* dW, int32_t* status,
                cudaStream_t s) {
    mw_status st = cuda_status(cudaMemsetAsync(dH, 0, sizeof(Tin) * (size_t)N * d, s));
    if (st != MW_OK) return st;
    if (M == 0) return cuda_status(cudaMemsetAsync(dW, 0, sizeof(float) * (size_t)Vocab * d, s));
    count_launches(2);
    const size_t smem_h = sizeof(float) * (FR * d + FR * 256);
    cudaFuncSetAttribute(k_lm_dh_simt<Tin>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_h);
    k_lm_dh_simt<Tin><<<(unsigned)ceil_div(M, FR), 256, smem_h, s>>>(M, N, d, Vocab, (const Tin*)H, (const Tin*)W,
                                                                     targets, rows, lse, g, dloss, (Tin*)dH, status);
    const size_t smem_w = sizeof(float) * (WV * d + WR * d + WR * WV);
    cudaFuncSetAttribute(k_lm_dw_simt<Tin>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_w);
    k_lm_dw_simt<Tin><<<(unsigned)ceil_div(Vocab, WV), 256, smem_w, s>>>(M, N, d, Vocab, (const Tin*)H,
                                                                         (const Tin*)W, targets, rows, lse, g, dloss,
                                                                         dW, status);
    return launch_status();
}

}  // namespace

mw_status lm_fwd_simt(const void* H, const void* W, const int32_t* targets, const int32_t* rows, int M, int N, int d,
                      int Vocab, int dtype, float* lse, float* zt, float* lp, int32_t* status, cudaStream_t s) {
    if (M == 0) return MW_OK;
    return dtype == MW_F32 ? fwd_t<float>(H, W, targets, rows, M, N, d, Vocab, lse, zt, lp, status, s)
                           : fwd_t<__nv_bfloat16>(H, W, targets, rows, M, N, d, Vocab, lse, zt, lp, status, s);
}

mw_status lm_bwd_simt(const void* H, const void* W, const int32_t* targets, const int32_t* rows, int M, int N,
                      int d, int Vocab, int dtype, const float* lse, const float* g, float dloss, void* dH,
                      float* dW, int32_t* status, cudaStream_t s) {
    return dtype == MW_F32
               ? bwd_t<float>(H, W, targets, rows, M, N, d, Vocab, lse, g, dloss, dH, dW, status, s)
               : bwd_t<__nv_bfloat16>(H, W, targets, rows, M, N, d, Vocab, lse, g, dloss, dH, dW, status, s);
}

}  // namespace mw
