// Tensor-core LM-head row maxima over a vocabulary range (bf16 in, fp32
// accumulate): the reference prepass of the fused forward. No logits tensor
// is stored.
//
//   gather   Hg[m] = H[rows[m]] (bf16, zero-padded to a multiple of 128 rows),
//            tg[m] = targets[rows[m]]
//   partials persistent CTAs over (vocab chunk, 128-row tile) items; per item
//            the chunk's 256-wide vocab tiles are computed as
//            Z = Hg_tile W_tile^T with tcgen05.mma into one of two TMEM
//            accumulators (128 x 256 fp32 each) fed by a 4-stage TMA ring, while
//            four epilogue warps fold the previous tile into a running
//            (max, sum 2^(z log2 e - max)) per row and pick out the target
//            logit. Each item writes one (max, sum) partial per row.
//   k_lm_ref the row's reference: the largest of its partial maxima.
// Concurrent CTAs work on the same vocab chunk, so each W tile is read from
// HBM about once per wave and shared through L2.
//
// The training path runs this only over the first kRefVocab vocabulary
// entries (lm_ref_tc): the row maxima there are the fixed per-row references
// of the fused forward in lmhead_bwd_tc.cu, which computes the log-softmax
// over the whole vocabulary.

#include <math.h>

#include "common.cuh"
#include "tc.cuh"
#include "tmap.cuh"

namespace mw {

namespace {

using namespace tc;

constexpr int NT = 192;
constexpr int BM = 128, BN = 256, BK = 64;
constexpr uint32_t A_B = BM * BK * 2;   // 16 KB
constexpr uint32_t B_B = BN * BK * 2;   // 32 KB
constexpr uint32_t ST_B = A_B + B_B;
constexpr int NSTAGE = 4;
constexpr uint32_t SMEM_LMF = NSTAGE * ST_B + 1024;
constexpr float LOG2E_F = 1.4426950408889634f;
// vocabulary entries whose row maxima serve as the fused forward's references
constexpr int kRefVocab = 2048;

struct LmFwdParams {
    int M, M_pad, d, V;
    int R, NV, C, NVC;        // row tiles, vocab tiles, chunks, vocab tiles per chunk
    int GR;                   // row tiles per item group
    const int32_t* tg;        // [M_pad]
    float2* part;             // [C][M_pad] (max2, sum)
    float* zt;                // [M]
    int32_t* status;
};

// Item w -> (vocab chunk c, row tile r). Items run in groups of GR row tiles:
// within a group chunk-major, rows fastest. The CTAs resident at one time then
// cover at most GR row tiles, whose hidden-state tiles stay in L2 (GR is sized
// from d on the host), and the W tiles of their chunks are shared in step.
__device__ __forceinline__ void item_rc(int w, int R, int C, int GR, int& c, int& r) {
    const int rg = w / (GR * C);
    const int rem = w - rg * (GR * C);
    const int gr = min(GR, R - rg * GR);   // rows in this (possibly ragged last) group
    c = rem / gr;
    r = rg * GR + rem % gr;
}

__global__ void __launch_bounds__(NT, 1)
    k_lm_fwd_tc(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, LmFwdParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t full[NSTAGE], empty[NSTAGE], acc_full[2], acc_empty[2];
    __shared__ uint32_t tmem_base;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_items = p.R * p.C;
    const int KC = p.d / BK;
    if (threadIdx.x == 0) {
        for (int s = 0; s < NSTAGE; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&acc_full[s], 1);
            mbar_init(&acc_empty[s], 128);
        }
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&tmem_base, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base;

    if (warp == 0) {
        if (lane == 0) {
            prefetch_tmap(&tmA);
            prefetch_tmap(&tmB);
            uint32_t it = 0;
            bool ok = true;
            for (int w = blockIdx.x; ok && w < n_items; w += gridDim.x) {
                int c, r;
                item_rc(w, p.R, p.C, p.GR, c, r);
                const int v0 = c * p.NVC, v1 = min(v0 + p.NVC, p.NV);
                for (int vt = v0; ok && vt < v1; ++vt)
                    for (int kc = 0; kc < KC; ++kc, ++it) {
                        const int s = it % NSTAGE;
                        if (it >= NSTAGE && !mbar_wait(&empty[s], ((it / NSTAGE) - 1) & 1, p.status, 401)) {
                            ok = false;
                            break;
                        }
                        mbar_expect_tx(&full[s], ST_B);
                        tma_load_2d(sm + s * ST_B, &tmA, &full[s], kc * BK, r * BM);
                        tma_load_2d(sm + s * ST_B + A_B, &tmB, &full[s], kc * BK, vt * BN);
                    }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(BM, BN, 0, 0);
            const uint32_t base = smem_u32(sm);
            uint32_t it = 0, tile = 0;
            bool ok = true;
            for (int w = blockIdx.x; ok && w < n_items; w += gridDim.x) {
                int c, r_unused;
                item_rc(w, p.R, p.C, p.GR, c, r_unused);
                const int v0 = c * p.NVC, v1 = min(v0 + p.NVC, p.NV);
                for (int vt = v0; ok && vt < v1; ++vt, ++tile) {
                    const int ab = tile & 1;
                    if (tile >= 2 && !mbar_wait(&acc_empty[ab], ((tile >> 1) - 1) & 1, p.status, 402)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    for (int kc = 0; kc < KC; ++kc, ++it) {
                        const int s = it % NSTAGE;
                        if (!mbar_wait(&full[s], (it / NSTAGE) & 1, p.status, 403)) { ok = false; break; }
                        tc_fence_after();
                        const uint32_t a = base + s * ST_B, b = a + A_B;
#pragma unroll
                        for (int ks = 0; ks < 4; ++ks)
                            mma_ss(tmem + ab * BN, sdesc_sw128(a + ks * 32, 16, 1024), sdesc_sw128(b + ks * 32, 16, 1024),
                                   idesc, (kc | ks) != 0);
                        mma_commit(&empty[s]);
                    }
                    if (ok) mma_commit(&acc_full[ab]);
                }
            }
        }
    } else {
        const int qw = warp & 3;
        const int rl = qw * 32 + lane;
        const uint32_t lane_base = tmem + ((uint32_t)(qw * 32) << 16);
        uint32_t tile = 0;
        bool ok = true;
        for (int w = blockIdx.x; ok && w < n_items; w += gridDim.x) {
            int c, r;
            item_rc(w, p.R, p.C, p.GR, c, r);
            const int v0 = c * p.NVC, v1 = min(v0 + p.NVC, p.NV);
            const int m = r * BM + rl;
            const int tgt = p.tg[m];
            float mx = -INFINITY, l = 0.f;
            for (int vt = v0; vt < v1; ++vt, ++tile) {
                const int ab = tile & 1;
                if (!mbar_wait(&acc_full[ab], (tile >> 1) & 1, p.status, 404)) { ok = false; break; }
                tc_fence_after();
#pragma unroll 1
                for (int cc = 0; cc < BN / 32; ++cc) {
                    uint32_t z[32];
                    tmem_ld32(lane_base + ab * BN + cc * 32, z);
                    tmem_wait_ld();
                    const int vb = vt * BN + cc * 32;
                    const int nvalid = min(32, p.V - vb);
                    if (tgt >= vb && tgt < vb + 32 && m < p.M) {
#pragma unroll
                        for (int x = 0; x < 32; ++x)
                            if (tgt == vb + x) p.zt[m] = __uint_as_float(z[x]);
                    }
                    float cm = -INFINITY;
#pragma unroll
                    for (int x = 0; x < 32; ++x)
                        if (x < nvalid) cm = fmaxf(cm, __uint_as_float(z[x]));
                    const float cm2 = cm * LOG2E_F;
                    if (cm2 > mx) {
                        l *= ex2f_approx(mx - cm2);
                        mx = cm2;
                    }
                    float s = 0.f;
#pragma unroll
                    for (int x = 0; x < 32; ++x)
                        if (x < nvalid) s += ex2f_approx(fmaf(__uint_as_float(z[x]), LOG2E_F, -mx));
                    l += s;
                }
                tc_fence_before();
                mbar_arrive(&acc_empty[ab]);
            }
            if (ok) p.part[(int64_t)c * p.M_pad + m] = make_float2(mx, l);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// Hg[m] = H[rows[m]], tg[m] = targets[rows[m]] (-1 without targets); padded
// rows (m >= M) are zero with target -1. A row outside [0, N) or a target
// outside [0, V) is neither read nor used (zero row, target -1) and raises the
// bounds flag.
__global__ void k_lm_gather(int M, int M_pad, int d, int N, int V, const __nv_bfloat16* __restrict__ H,
                            const int32_t* __restrict__ targets, const int32_t* __restrict__ rows,
                            __nv_bfloat16* __restrict__ Hg, int32_t* __restrict__ tg, int32_t* __restrict__ status) {
    const int vec = d / 8;   // 16-byte vectors per row
    const int64_t total = (int64_t)M_pad * vec;
    for (int64_t x = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; x < total; x += (int64_t)gridDim.x * blockDim.x) {
        const int m = (int)(x / vec), k = (int)(x % vec);
        const int r = m < M ? checked_index(rows[m], N) : -1;
        uint4 val = make_uint4(0, 0, 0, 0);
        if (r >= 0) val = reinterpret_cast<const uint4*>(H + (int64_t)r * d)[k];
        reinterpret_cast<uint4*>(Hg + (int64_t)m * d)[k] = val;
        if (k == 0) {
            const int t = r >= 0 && targets ? checked_index(targets[r], V) : -1;
            if (m < M && (r < 0 || (targets && t < 0))) flag_bounds(status);
            tg[m] = t;
        }
    }
}

// par[m] = (0, ref, target bits, 0): ref = the row's largest logit over the
// vocabulary subset, in log2 units (max over the chunk partials); padded rows
// (m >= M) get ref 0 and target -1.
__global__ void k_lm_ref(int M, int M_pad, int C, const float2* __restrict__ part, const int32_t* __restrict__ tg,
                         float4* __restrict__ par) {
    const int m = blockIdx.x * blockDim.x + threadIdx.x;
    if (m >= M_pad) return;
    float mx = 0.f;
    if (m < M) {
        mx = -INFINITY;
        for (int c = 0; c < C; ++c) mx = fmaxf(mx, part[(int64_t)c * M_pad + m].x);
    }
    par[m] = make_float4(0.f, mx, __int_as_float(m < M ? tg[m] : -1), 0.f);
}

}  // namespace

// Shapes of the bf16 LM-head work split, shared with the workspace layout.
struct LmPlan {
    int M_pad, R, NV, C, NVC, grid;
};

static int num_sms() {
    int dev = 0, n = 152;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n > 0 ? n : 152;
}

LmPlan lm_plan(int M, int V) {
    LmPlan q;
    q.M_pad = (int)ceil_div(M, BM) * BM;
    q.R = q.M_pad / BM;
    q.NV = (int)ceil_div(V, BN);
    const int G = num_sms();
    // choose the number of vocab chunks C minimising waves x tiles-per-item
    long best = -1;
    q.C = 1;
    for (int C = 1; C <= 64; ++C) {
        const long items = (long)q.R * C;
        const long waves = (items + G - 1) / G;
        const long cost = waves * ceil_div(q.NV, C);
        if (best < 0 || cost < best) { best = cost; q.C = C; }
    }
    q.NVC = (int)ceil_div(q.NV, q.C);
    q.C = (int)ceil_div(q.NV, q.NVC);
    q.grid = (int)std::min<long>((long)q.R * q.C, G);
    return q;
}

// Forward partials of the loss rows against vocabulary entries [0, V): the
// gathered rows (Hg, tg) must already be in place.
static mw_status lm_partials(const void* W, int M, int d, int V, const void* Hg, const int32_t* tg, float2* part,
                             float* zt, int32_t* status, cudaStream_t s, LmPlan& q) {
    q = lm_plan(M, V);
    CUtensorMap ta, tb;
    if (!tmap_bf16_2d(&ta, Hg, q.M_pad, d, d, BM, BK) || !tmap_bf16_2d(&tb, W, V, d, d, BN, BK)) return MW_ECUDA;
    LmFwdParams p;
    p.M = M;
    p.M_pad = q.M_pad;
    p.d = d;
    p.V = V;
    p.R = q.R;
    p.NV = q.NV;
    p.C = q.C;
    p.NVC = q.NVC;
    // row tiles whose bf16 hidden-state tiles fill about 30 MB of L2 (32 at d = 3584)
    p.GR = (int)std::max<int64_t>(8, std::min<int64_t>(q.R, (30ll << 20) / ((int64_t)BM * d * 2)));
    p.tg = tg;
    p.part = part;
    p.zt = zt;
    p.status = status;
    mw_status st = cuda_status(cudaFuncSetAttribute(k_lm_fwd_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                    (int)SMEM_LMF));
    if (st != MW_OK) return st;
    count_launches(1);
    k_lm_fwd_tc<<<q.grid, NT, SMEM_LMF, s>>>(ta, tb, p);
    return launch_status();
}

static mw_status lm_gather(const void* H, const int32_t* targets, const int32_t* rows, int M, int N, int d, int V,
                           void* Hg, int32_t* tg, int32_t* status, cudaStream_t s) {
    const int64_t M_pad = ceil_div(M, BM) * BM;
    const int64_t vec = M_pad * (d / 8);
    count_launches(1);
    k_lm_gather<<<(unsigned)std::min<int64_t>(ceil_div(vec, 256), 152 * 32), 256, 0, s>>>(
        M, (int)M_pad, d, N, V, (const __nv_bfloat16*)H, targets, rows, (__nv_bfloat16*)Hg, tg, status);
    return launch_status();
}

int lm_ref_vocab(int V) { return std::min(V, kRefVocab); }

mw_status lm_ref_tc(const void* H, const void* W, const int32_t* targets, const int32_t* rows, int M, int N, int d,
                    int V, void* Hg, int32_t* tg, float2* part, float* zt, float4* par, int32_t* status,
                    cudaStream_t s) {
    if (M == 0) return MW_OK;
    mw_status st = lm_gather(H, targets, rows, M, N, d, V, Hg, tg, status, s);
    LmPlan q;
    if (st == MW_OK) st = lm_partials(W, M, d, lm_ref_vocab(V), Hg, tg, part, zt, status, s, q);
    if (st != MW_OK) return st;
    count_launches(1);
    k_lm_ref<<<(unsigned)ceil_div(q.M_pad, 256), 256, 0, s>>>(M, q.M_pad, q.C, part, tg, par);
    return launch_status();
}

}  // namespace mw
