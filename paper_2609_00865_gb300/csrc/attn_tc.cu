// Tensor-core masked GQA attention, bf16 in / fp32 accumulate, head dim 128.
//
// Mask (§4.2): key j is visible to row i iff j <= i < omega(j). A tile's
// class comes from the visibility builder: EMPTY tiles are never listed,
// FULL tiles run unmasked, PARTIAL and diagonal tiles apply the row's
// per-(segment, k-tile) view bits (and causality on the diagonal). For a row
// of segment s, "omega(j) > i" is the same as "j is in view_s", because every
// lifetime ends at a junction; so one 128-bit word per (segment, k-tile)
// replaces 128 lifetime compares.
//
// Forward kernel (one CTA per (q-tile, q-head), heaviest q-tiles first):
//   warp 0      TMA producer: Q once, then K_j / V_j of each listed k-tile
//               (2-stage rings, 128-byte swizzle)
//   warp 1      TMEM allocator + single-thread tcgen05.mma issuer:
//               S_j = Q K_j^T into one of two TMEM S buffers, then
//               O += P_{j-1} V_{j-1} once the softmax has written P_{j-1}
//   warps 2..5  softmax / epilogue, one query row per thread: online softmax
//               in the exp2 domain with lazy rescaling of O (only when the
//               running max grows by more than 2^8), P written as bf16 into
//               shared memory, O / l and the log-sum-exp written at the end.
// All waits are bounded (tc::mbar_wait); a timeout ends the CTA and is
// reported through the visibility status word.

#include <math.h>

#include "common.cuh"
#include "tc.cuh"
#include "tmap.cuh"

namespace mw {
namespace {

using namespace tc;

constexpr int DH = 128;
constexpr uint32_t TILE_B = 128 * DH * 2;  // one 128 x 128 bf16 tile: two [128][64] swizzled halves
constexpr uint32_t HALF_B = TILE_B / 2;
constexpr int NTHREADS = 192;
constexpr float LOG2E = 1.4426950408889634f;
constexpr float RESCALE_T = 8.0f;          // lazy-rescale threshold (log2 units)

// dynamic shared memory map (bytes from the 1024-aligned base)
constexpr uint32_t SM_Q = 0;
constexpr uint32_t SM_K = SM_Q + TILE_B;
constexpr uint32_t SM_V = SM_K + 2 * TILE_B;
constexpr uint32_t SM_P = SM_V + 2 * TILE_B;
constexpr uint32_t SM_TOTAL = SM_P + TILE_B;
constexpr uint32_t SMEM_FWD = SM_TOTAL + 1024;

// TMEM columns
constexpr uint32_t TM_S0 = 0, TM_O = 256;

struct FwdParams {
    VisView v;
    int64_t total;
    int n_traj, max_tiles, Hq, Hkv;
    float scale_log2;
    __nv_bfloat16* O;
    float* LSE;
};

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ void load_tile(uint8_t* dst, const CUtensorMap* map, uint64_t* bar, int head, int row) {
    tma_load_3d(dst, map, bar, 0, head, row);
    tma_load_3d(dst + HALF_B, map, bar, 64, head, row);
}

// K-major operand descriptor for k-step ks (16 elements) of a [128][128] tile.
__device__ __forceinline__ uint64_t kmaj(uint32_t base, int ks) {
    return sdesc_sw128(base + (ks >> 2) * HALF_B + (ks & 3) * 32, 16, 1024);
}
// MN-major operand descriptor (rows = K dim, 128 contiguous N elements split in
// two 64-wide halves) for k-step ks.
__device__ __forceinline__ uint64_t mnmaj(uint32_t base, int ks) {
    return sdesc_sw128(base + ks * 2048, HALF_B, 1024);
}

__global__ void __launch_bounds__(NTHREADS, 1)
    k_attn_fwd_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                  const __grid_constant__ CUtensorMap tmV, FwdParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t q_full, k_full[2], k_empty[2], v_full[2], v_empty[2], s_full[2], s_free[2],
        p_full, o_done;
    __shared__ uint32_t tmem_base;
    __shared__ int abort_flag;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // item -> (local q-tile, trajectory, head); heaviest (largest qt) first,
    // query heads of one KV group adjacent.
    const int h = blockIdx.x % p.Hq;
    const int r = blockIdx.x / p.Hq;
    const int qt = p.max_tiles - 1 - r / p.n_traj;
    const int b = r % p.n_traj;
    const VisView& v = p.v;
    const int nt = v.traj_tile[b + 1] - v.traj_tile[b];
    if (qt >= nt) return;
    const int64_t g = v.traj_tile[b] + qt;
    const int64_t tok0 = v.traj_tok[b];
    const int T = v.traj_tok[b + 1] - (int)tok0;
    const int kvh = h / (p.Hq / p.Hkv);
    const int p0 = v.fwd_ptr[g];
    const int n = v.fwd_ptr[g + 1] - p0;
    int32_t* status = v.status;

    if (threadIdx.x == 0) {
        mbar_init(&q_full, 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&k_empty[s], 1);
            mbar_init(&v_full[s], 1);
            mbar_init(&v_empty[s], 1);
            mbar_init(&s_full[s], 1);
            mbar_init(&s_free[s], 128);
        }
        mbar_init(&p_full, 128);
        mbar_init(&o_done, 1);
        abort_flag = 0;
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
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            prefetch_tmap(&tmQ);
            prefetch_tmap(&tmK);
            prefetch_tmap(&tmV);
            mbar_expect_tx(&q_full, TILE_B);
            load_tile(sm + SM_Q, &tmQ, &q_full, h, (int)(tok0 + qt * 128));
            for (int j = 0; j < n; ++j) {
                const int kt = v.fwd_idx[p0 + j] >> 2;
                const int s = j & 1;
                const int row = (int)(tok0 + kt * 128);
                if (j >= 2 && !mbar_wait(&k_empty[s], ((j - 2) >> 1) & 1, status, 101)) { abort_flag = 1; break; }
                mbar_expect_tx(&k_full[s], TILE_B);
                load_tile(sm + SM_K + s * TILE_B, &tmK, &k_full[s], kvh, row);
                if (j >= 2 && !mbar_wait(&v_empty[s], ((j - 2) >> 1) & 1, status, 102)) { abort_flag = 1; break; }
                mbar_expect_tx(&v_full[s], TILE_B);
                load_tile(sm + SM_V + s * TILE_B, &tmV, &v_full[s], kvh, row);
                if (*(volatile int*)&abort_flag) break;
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t iS = idesc_bf16(128, 128, 0, 0);   // S = Q K^T: both K-major
            const uint32_t iO = idesc_bf16(128, 128, 0, 1);   // O += P V: V is MN-major
            const uint32_t sq = smem_u32(sm + SM_Q), sk = smem_u32(sm + SM_K), sv = smem_u32(sm + SM_V),
                           sp = smem_u32(sm + SM_P);
            bool ok = mbar_wait(&q_full, 0, status, 201);
            auto pv = [&](int t) -> bool {
                if (!mbar_wait(&p_full, t & 1, status, 202)) return false;
                if (!mbar_wait(&v_full[t & 1], (t >> 1) & 1, status, 203)) return false;
                tc_fence_after();
                const uint32_t vb = sv + (t & 1) * TILE_B;
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) mma_ss(tmem + TM_O, kmaj(sp, ks), mnmaj(vb, ks), iO, (t > 0 || ks > 0));
                mma_commit(&v_empty[t & 1]);
                mma_commit(&o_done);
                return true;
            };
            for (int j = 0; ok && j < n; ++j) {
                const int s = j & 1;
                if (!mbar_wait(&k_full[s], (j >> 1) & 1, status, 204)) { ok = false; break; }
                if (j >= 2 && !mbar_wait(&s_free[s], ((j - 2) >> 1) & 1, status, 205)) { ok = false; break; }
                tc_fence_after();
                const uint32_t kb = sk + s * TILE_B;
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) mma_ss(tmem + TM_S0 + s * 128, kmaj(sq, ks), kmaj(kb, ks), iS, ks > 0);
                mma_commit(&k_empty[s]);
                mma_commit(&s_full[s]);
                if (j >= 1 && !pv(j - 1)) { ok = false; break; }
            }
            if (ok && n > 0) ok = pv(n - 1);
            if (!ok) abort_flag = 1;
        }
    } else {
        // ------------------------------------------------------------ softmax + epilogue
        const int qw = warp & 3;
        const int rl = qw * 32 + lane;          // row inside the q-tile = TMEM lane
        const int i = qt * 128 + rl;
        const int ie = min(i, T - 1);
        const int seg = v.seg[tok0 + ie];
        const uint4* km = reinterpret_cast<const uint4*>(v.keymask) + v.traj_km[b] + (int64_t)seg * nt;
        const uint32_t lane_base = tmem + ((uint32_t)(qw * 32) << 16);
        uint8_t* prow = sm + SM_P;
        float m = -INFINITY, l = 0.f;
        bool ok = true;
        for (int j = 0; j < n; ++j) {
            const int e = v.fwd_idx[p0 + j];
            const int kt = e >> 2, cls = e & 3;
            if (!mbar_wait(&s_full[j & 1], (j >> 1) & 1, status, 301)) { ok = false; break; }
            tc_fence_after();
            float s[128];
            {
                uint32_t rr[32];
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    tmem_ld32(lane_base + TM_S0 + (j & 1) * 128 + c * 32, rr);
                    tmem_wait_ld();
#pragma unroll
                    for (int x = 0; x < 32; ++x) s[c * 32 + x] = __uint_as_float(rr[x]);
                }
            }
            tc_fence_before();
            mbar_arrive(&s_free[j & 1]);
            if (cls != MW_TILE_FULL || kt == qt) {
                uint4 w = km[kt];
                uint32_t wd[4] = {w.x, w.y, w.z, w.w};
                if (kt == qt) {   // causal inside the diagonal tile: keys c <= ie - kt*128
                    const int lim = ie - kt * 128;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const int hi = lim - 32 * q;   // keep bits 0..hi
                        const uint32_t keep = hi >= 31 ? 0xffffffffu : (hi < 0 ? 0u : ((2u << hi) - 1u));
                        wd[q] &= keep;
                    }
                }
#pragma unroll
                for (int c = 0; c < 128; ++c)
                    if (!((wd[c >> 5] >> (c & 31)) & 1u)) s[c] = -INFINITY;
            }
            float mx = -INFINITY;
#pragma unroll
            for (int c = 0; c < 128; ++c) mx = fmaxf(mx, s[c]);
            const float mx2 = mx * p.scale_log2;
            float alpha = 1.f;
            if (mx2 > m + RESCALE_T) {
                alpha = ex2(m - mx2);   // 0 when m = -inf
                m = mx2;
            }
            const float mu = (m == -INFINITY) ? 0.f : m;
            float rs = 0.f;
#pragma unroll
            for (int c = 0; c < 128; ++c) {
                s[c] = ex2(fmaf(s[c], p.scale_log2, -mu));
                rs += s[c];
            }
            l = l * alpha + rs;
            // P_j overwrites P_{j-1}: wait for O += P_{j-1} V_{j-1} to finish
            if (j >= 1 && !mbar_wait(&o_done, (j - 1) & 1, status, 302)) { ok = false; break; }
            tc_fence_after();
#pragma unroll
            for (int c = 0; c < 16; ++c) {
                uint4 pk;
                pk.x = pack_bf16(s[8 * c + 0], s[8 * c + 1]);
                pk.y = pack_bf16(s[8 * c + 2], s[8 * c + 3]);
                pk.z = pack_bf16(s[8 * c + 4], s[8 * c + 5]);
                pk.w = pack_bf16(s[8 * c + 6], s[8 * c + 7]);
                *reinterpret_cast<uint4*>(prow + (c >> 3) * HALF_B + sw128_off(rl, c & 7)) = pk;
            }
            // O was last written by PV_{j-1}; rescale it when the max moved
            if (j >= 1 && __any_sync(0xffffffffu, alpha != 1.f)) {
                uint32_t o[32];
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    tmem_ld32(lane_base + TM_O + c * 32, o);
                    tmem_wait_ld();
#pragma unroll
                    for (int x = 0; x < 32; ++x) o[x] = __float_as_uint(__uint_as_float(o[x]) * alpha);
                    uint32_t lo[16], hi[16];
#pragma unroll
                    for (int x = 0; x < 16; ++x) { lo[x] = o[x]; hi[x] = o[16 + x]; }
                    tmem_st16(lane_base + TM_O + c * 32, lo);
                    tmem_st16(lane_base + TM_O + c * 32 + 16, hi);
                }
                tmem_wait_st();
            }
            fence_async_smem();
            tc_fence_before();
            mbar_arrive(&p_full);
        }
        // epilogue: O / l, LSE (natural log)
        if (ok && n > 0 && mbar_wait(&o_done, (n - 1) & 1, status, 303)) {
            tc_fence_after();
            const float inv = 1.f / l;
            __nv_bfloat16* orow = p.O + ((tok0 + ie) * p.Hq + h) * DH;
            uint32_t o[32];
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                tmem_ld32(lane_base + TM_O + c * 32, o);
                tmem_wait_ld();
                if (i < T) {
#pragma unroll
                    for (int x = 0; x < 4; ++x) {
                        uint4 pk;
                        pk.x = pack_bf16(__uint_as_float(o[8 * x + 0]) * inv, __uint_as_float(o[8 * x + 1]) * inv);
                        pk.y = pack_bf16(__uint_as_float(o[8 * x + 2]) * inv, __uint_as_float(o[8 * x + 3]) * inv);
                        pk.z = pack_bf16(__uint_as_float(o[8 * x + 4]) * inv, __uint_as_float(o[8 * x + 5]) * inv);
                        pk.w = pack_bf16(__uint_as_float(o[8 * x + 6]) * inv, __uint_as_float(o[8 * x + 7]) * inv);
                        *reinterpret_cast<uint4*>(orow + c * 32 + 8 * x) = pk;
                    }
                }
            }
            if (i < T) p.LSE[(int64_t)h * p.total + tok0 + i] = (m + __log2f(l)) * 0.6931471805599453f;
        } else {
            abort_flag = 1;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

}  // namespace

mw_status attn_fwd_tc(const mw_vis_layout* L, const void* vis, const void* Q, const void* K, const void* V,
                      void* O, float* LSE, int Hq, int Hkv, float scale, cudaStream_t s) {
    if (L->n_tiles == 0) return MW_OK;
    CUtensorMap tq, tk, tv;
    const uint64_t T = (uint64_t)L->total_tokens;
    if (!tmap_bf16_3d(&tq, Q, T, Hq, DH, 128, 64) || !tmap_bf16_3d(&tk, K, T, Hkv, DH, 128, 64) ||
        !tmap_bf16_3d(&tv, V, T, Hkv, DH, 128, 64))
        return MW_ECUDA;
    FwdParams p;
    p.v = make_view(L, vis);
    p.total = L->total_tokens;
    p.n_traj = L->n_traj;
    p.max_tiles = L->max_tiles;
    p.Hq = Hq;
    p.Hkv = Hkv;
    p.scale_log2 = scale * LOG2E;
    p.O = (__nv_bfloat16*)O;
    p.LSE = LSE;
    mw_status st = cuda_status(cudaFuncSetAttribute(k_attn_fwd_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                    (int)SMEM_FWD));
    if (st != MW_OK) return st;
    const unsigned grid = (unsigned)((int64_t)L->max_tiles * L->n_traj * Hq);
    count_launches(1);
    k_attn_fwd_tc<<<grid, NTHREADS, SMEM_FWD, s>>>(tq, tk, tv, p);
    return launch_status();
}

}  // namespace mw
