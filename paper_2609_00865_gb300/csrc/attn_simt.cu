// Masked GQA attention on CUDA cores with float32 arithmetic.
//
// This is the path for float32 inputs, where tensor-core tf32 could not hold
// 1e-4 relative agreement. It implements the same mask as the tensor-core
// path (§4.2: key j visible to row i iff j <= i < omega(j)), visiting only the
// non-EMPTY tiles of each q-tile's list in the forward.
//
// SEGK variants read keys from per-segment copies ("segment key rows": row
// (traj_km[b] + s nt_b) * 128 + j holds key j as seen by segment s, e.g.
// rotated to its logical position in view_s) instead of the physical rows;
// the dK/dV kernel then writes one float32 gradient row per (segment, key).
//
// Work mapping: one warp per query row (forward, dQ) or per key row (dK/dV).
// In the forward a lane owns one key of each 32-key chunk for the q.k dot and
// one slice of head dims for the P.V accumulation. In dK/dV the rows that see
// key j form the interval [j, min(omega(j), T)), so no tile list is needed.

#include <math.h>

#include "common.cuh"

namespace mw {
namespace {

constexpr float NEG_INF = -INFINITY;

template <typename Tin, int DH>
__device__ __forceinline__ float dot_row(const float* __restrict__ q_s, const Tin* __restrict__ row) {
    float acc = 0.f;
#pragma unroll 8
    for (int d = 0; d < DH; ++d) acc = fmaf(q_s[d], ld_f(row + d), acc);
    return acc;
}

template <typename Tin, int DH, bool SEGK>
__global__ void __launch_bounds__(128) k_attn_fwd_simt(VisView v, int64_t total, const Tin* __restrict__ Q,
                                                      const Tin* __restrict__ K, const Tin* __restrict__ V,
                                                      Tin* __restrict__ O, float* __restrict__ LSE, int Hq,
                                                      int Hkv, float scale) {
    constexpr int NC = DH / 32;
    __shared__ float qs[4][DH];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t g = blockIdx.x;
    const int h = blockIdx.y;
    const int b = v.tile_traj[g];
    const int qt = (int)(g - v.traj_tile[b]);
    const int64_t tok0 = v.traj_tok[b];
    const int T = v.traj_tok[b + 1] - (int)tok0;
    const int kvh = h / (Hq / Hkv);
    const int p0 = v.fwd_ptr[g], p1 = v.fwd_ptr[g + 1];
    const int nt = v.traj_tile[b + 1] - v.traj_tile[b];
    for (int r = warp; r < MW_TILE; r += 4) {
        const int i = qt * MW_TILE + r;
        if (i >= T) break;
        const int64_t gi = tok0 + i;
        const int64_t kb = SEGK ? (v.traj_km[b] + (int64_t)v.seg[gi] * nt) * MW_TILE : tok0;  // key row of j = 0
#pragma unroll
        for (int c = 0; c < NC; ++c) qs[warp][lane + 32 * c] = ld_f(Q + (gi * Hq + h) * DH + lane + 32 * c);
        __syncwarp();
        float m = NEG_INF, l = 0.f, o[NC];
#pragma unroll
        for (int c = 0; c < NC; ++c) o[c] = 0.f;
        for (int p = p0; p < p1; ++p) {
            const int e = v.fwd_idx[p];
            const int kt = e >> 4, cls = e & 3;
            const int jend = min(kt * MW_TILE + MW_TILE, i + 1);
            if (!MW_DBG_IN(kt, qt + 1, v.status, 211)) continue;
            for (int j0 = kt * MW_TILE; j0 < jend; j0 += 32) {
                const int j = j0 + lane;
                bool vis = j < jend;
                if (vis && cls != MW_TILE_FULL) vis = i < v.omega[tok0 + j];
                float s = NEG_INF;
                if (vis) s = dot_row<Tin, DH>(qs[warp], K + ((kb + j) * Hkv + kvh) * DH) * scale;
                const float cm = warp_max(s);
                if (cm == NEG_INF) continue;
                const float mn = fmaxf(m, cm);
                const float alpha = expf(m - mn);
                const float pj = vis ? expf(s - mn) : 0.f;
                l = l * alpha + warp_sum(pj);
#pragma unroll
                for (int c = 0; c < NC; ++c) o[c] *= alpha;
                const int nk = min(32, jend - j0);
                for (int jj = 0; jj < nk; ++jj) {
                    const float pb = __shfl_sync(0xffffffffu, pj, jj);
                    const Tin* vr = V + ((tok0 + j0 + jj) * Hkv + kvh) * DH;
#pragma unroll
                    for (int c = 0; c < NC; ++c) o[c] = fmaf(pb, ld_f(vr + lane + 32 * c), o[c]);
                }
                m = mn;
            }
        }
        const float inv = 1.f / l;
#pragma unroll
        for (int c = 0; c < NC; ++c) st_f(O + (gi * Hq + h) * DH + lane + 32 * c, o[c] * inv);
        if (lane == 0) LSE[(int64_t)h * total + gi] = m + logf(l);
        __syncwarp();
    }
}

// Delta_i = rowsum(dO_i * O_i) per (row, head); one warp each.
template <typename Tin, int DH>
__global__ void k_attn_delta(int64_t total, int Hq, const Tin* __restrict__ O, const Tin* __restrict__ dO,
                             float* __restrict__ delta) {
    const int lane = threadIdx.x & 31;
    const int64_t nw = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t w = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; w < total * Hq; w += nw) {
        const int64_t gi = w / Hq;
        const int h = (int)(w % Hq);
        float acc = 0.f;
        for (int d = lane; d < DH; d += 32) acc = fmaf(ld_f(O + w * DH + d), ld_f(dO + w * DH + d), acc);
        acc = warp_sum(acc);
        if (lane == 0) delta[(int64_t)h * total + gi] = acc;
    }
}

// dQ_i = scale * sum_j P_ij (dP_ij - Delta_i) k_j ; one warp per row.
template <typename Tin, int DH, bool SEGK>
__global__ void __launch_bounds__(128) k_attn_dq_simt(VisView v, int64_t total, const Tin* __restrict__ Q,
                                                     const Tin* __restrict__ K, const Tin* __restrict__ V,
                                                     const Tin* __restrict__ dO, const float* __restrict__ LSE,
                                                     const float* __restrict__ delta, Tin* __restrict__ dQ,
                                                     int Hq, int Hkv, float scale) {
    constexpr int NC = DH / 32;
    __shared__ float qs[4][DH];
    __shared__ float ds_[4][DH];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t g = blockIdx.x;
    const int h = blockIdx.y;
    const int b = v.tile_traj[g];
    const int qt = (int)(g - v.traj_tile[b]);
    const int64_t tok0 = v.traj_tok[b];
    const int T = v.traj_tok[b + 1] - (int)tok0;
    const int kvh = h / (Hq / Hkv);
    const int p0 = v.fwd_ptr[g], p1 = v.fwd_ptr[g + 1];
    const int nt = v.traj_tile[b + 1] - v.traj_tile[b];
    for (int r = warp; r < MW_TILE; r += 4) {
        const int i = qt * MW_TILE + r;
        if (i >= T) break;
        const int64_t gi = tok0 + i;
        const int64_t kb = SEGK ? (v.traj_km[b] + (int64_t)v.seg[gi] * nt) * MW_TILE : tok0;  // key row of j = 0
#pragma unroll
        for (int c = 0; c < NC; ++c) {
            qs[warp][lane + 32 * c] = ld_f(Q + (gi * Hq + h) * DH + lane + 32 * c);
            ds_[warp][lane + 32 * c] = ld_f(dO + (gi * Hq + h) * DH + lane + 32 * c);
        }
        __syncwarp();
        const float lse = LSE[(int64_t)h * total + gi];
        const float dl = delta[(int64_t)h * total + gi];
        float dq[NC];
#pragma unroll
        for (int c = 0; c < NC; ++c) dq[c] = 0.f;
        for (int p = p0; p < p1; ++p) {
            const int e = v.fwd_idx[p];
            const int kt = e >> 4, cls = e & 3;
            const int jend = min(kt * MW_TILE + MW_TILE, i + 1);
            if (!MW_DBG_IN(kt, qt + 1, v.status, 212)) continue;
            for (int j0 = kt * MW_TILE; j0 < jend; j0 += 32) {
                const int j = j0 + lane;
                bool vis = j < jend;
                if (vis && cls != MW_TILE_FULL) vis = i < v.omega[tok0 + j];
                float dsj = 0.f;
                if (vis) {
                    const float s = dot_row<Tin, DH>(qs[warp], K + ((kb + j) * Hkv + kvh) * DH) * scale;
                    const float pj = expf(s - lse);
                    const float dp = dot_row<Tin, DH>(ds_[warp], V + ((tok0 + j) * Hkv + kvh) * DH);
                    dsj = pj * (dp - dl);
                }
                const int nk = min(32, jend - j0);
                for (int jj = 0; jj < nk; ++jj) {
                    const float db = __shfl_sync(0xffffffffu, dsj, jj);
                    const Tin* kr = K + ((kb + j0 + jj) * Hkv + kvh) * DH;
#pragma unroll
                    for (int c = 0; c < NC; ++c) dq[c] = fmaf(db, ld_f(kr + lane + 32 * c), dq[c]);
                }
            }
        }
#pragma unroll
        for (int c = 0; c < NC; ++c) st_f(dQ + (gi * Hq + h) * DH + lane + 32 * c, dq[c] * scale);
        __syncwarp();
    }
}

// dK_j = scale * sum_{h in group} sum_{i in [j, omega_j)} dS_ij q_i ,
// dV_j = sum_{h in group} sum_i P_ij dO_i ; one warp per key row.
template <typename Tin, int DH>
__global__ void __launch_bounds__(128) k_attn_dkv_simt(VisView v, int64_t total, const Tin* __restrict__ Q,
                                                      const Tin* __restrict__ K, const Tin* __restrict__ V,
                                                      const Tin* __restrict__ dO, const float* __restrict__ LSE,
                                                      const float* __restrict__ delta, Tin* __restrict__ dK,
                                                      Tin* __restrict__ dV, int Hq, int Hkv, float scale) {
    constexpr int NC = DH / 32;
    __shared__ float ks[4][DH];
    __shared__ float vs[4][DH];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t g = blockIdx.x;
    const int kvh = blockIdx.y;
    const int grp = Hq / Hkv;
    const int b = v.tile_traj[g];
    const int kt = (int)(g - v.traj_tile[b]);
    const int64_t tok0 = v.traj_tok[b];
    const int T = v.traj_tok[b + 1] - (int)tok0;
    for (int r = warp; r < MW_TILE; r += 4) {
        const int j = kt * MW_TILE + r;
        if (j >= T) break;
        const int64_t gj = tok0 + j;
#pragma unroll
        for (int c = 0; c < NC; ++c) {
            ks[warp][lane + 32 * c] = ld_f(K + (gj * Hkv + kvh) * DH + lane + 32 * c);
            vs[warp][lane + 32 * c] = ld_f(V + (gj * Hkv + kvh) * DH + lane + 32 * c);
        }
        __syncwarp();
        const int iend = min(v.omega[gj], T);
        float dk[NC], dv[NC];
#pragma unroll
        for (int c = 0; c < NC; ++c) dk[c] = dv[c] = 0.f;
        for (int h = kvh * grp; h < (kvh + 1) * grp; ++h) {
            for (int i0 = j; i0 < iend; i0 += 32) {
                const int i = i0 + lane;
                float pi = 0.f, dsi = 0.f;
                if (i < iend) {
                    const int64_t gi = tok0 + i;
                    const float s = dot_row<Tin, DH>(ks[warp], Q + (gi * Hq + h) * DH) * scale;
                    pi = expf(s - LSE[(int64_t)h * total + gi]);
                    const float dp = dot_row<Tin, DH>(vs[warp], dO + (gi * Hq + h) * DH);
                    dsi = pi * (dp - delta[(int64_t)h * total + gi]);
                }
                const int ni = min(32, iend - i0);
                for (int ii = 0; ii < ni; ++ii) {
                    const float pb = __shfl_sync(0xffffffffu, pi, ii);
                    const float db = __shfl_sync(0xffffffffu, dsi, ii);
                    const int64_t row = ((tok0 + i0 + ii) * Hq + h) * DH;
#pragma unroll
                    for (int c = 0; c < NC; ++c) {
                        dv[c] = fmaf(pb, ld_f(dO + row + lane + 32 * c), dv[c]);
                        dk[c] = fmaf(db, ld_f(Q + row + lane + 32 * c), dk[c]);
                    }
                }
            }
        }
#pragma unroll
        for (int c = 0; c < NC; ++c) {
            st_f(dK + (gj * Hkv + kvh) * DH + lane + 32 * c, dk[c] * scale);
            st_f(dV + (gj * Hkv + kvh) * DH + lane + 32 * c, dv[c]);
        }
        __syncwarp();
    }
}

// dK/dV with segment key rows: the rows that see key j split by segment; for
// segment s (rows [max(j, J_s), min(omega_j, T, J_(s+1)))) the key row read is
// (kmb + s nt) 128 + j, and that row's gradient dKseg = scale * sum dS q is
// written in float32 (zero when no row of s sees j). dV sums over all rows.
template <typename Tin, int DH>
__global__ void __launch_bounds__(128) k_attn_dkv_segk_simt(VisView v, int64_t total, const Tin* __restrict__ Q,
                                                           const Tin* __restrict__ Kseg, const Tin* __restrict__ V,
                                                           const Tin* __restrict__ dO, const float* __restrict__ LSE,
                                                           const float* __restrict__ delta,
                                                           float* __restrict__ dKseg, Tin* __restrict__ dV, int Hq,
                                                           int Hkv, float scale) {
    constexpr int NC = DH / 32;
    __shared__ float ks[4][DH];
    __shared__ float vs[4][DH];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t g = blockIdx.x;
    const int kvh = blockIdx.y;
    const int grp = Hq / Hkv;
    const int b = v.tile_traj[g];
    const int kt = (int)(g - v.traj_tile[b]);
    const int64_t tok0 = v.traj_tok[b];
    const int T = v.traj_tok[b + 1] - (int)tok0;
    const int nt = v.traj_tile[b + 1] - v.traj_tile[b];
    const int nseg = v.traj_seg[b + 1] - v.traj_seg[b];
    const int32_t* sst = v.seg_start + v.traj_seg[b];
    for (int r = warp; r < MW_TILE; r += 4) {
        const int j = kt * MW_TILE + r;
        if (j >= T) break;
        const int64_t gj = tok0 + j;
#pragma unroll
        for (int c = 0; c < NC; ++c) vs[warp][lane + 32 * c] = ld_f(V + (gj * Hkv + kvh) * DH + lane + 32 * c);
        const int iend = min(v.omega[gj], T);
        float dv[NC];
#pragma unroll
        for (int c = 0; c < NC; ++c) dv[c] = 0.f;
        for (int s = 0; s < nseg; ++s) {
            const int64_t krow = (v.traj_km[b] + (int64_t)s * nt) * MW_TILE + j;
            const int rlo = max(j, sst[s]);
            const int rhi = min(iend, s + 1 < nseg ? sst[s + 1] : T);
            float dk[NC];
#pragma unroll
            for (int c = 0; c < NC; ++c) dk[c] = 0.f;
            if (rlo < rhi) {
                __syncwarp();
#pragma unroll
                for (int c = 0; c < NC; ++c)
                    ks[warp][lane + 32 * c] = ld_f(Kseg + (krow * Hkv + kvh) * DH + lane + 32 * c);
                __syncwarp();
                for (int h = kvh * grp; h < (kvh + 1) * grp; ++h) {
                    for (int i0 = rlo; i0 < rhi; i0 += 32) {
                        const int i = i0 + lane;
                        float pi = 0.f, dsi = 0.f;
                        if (i < rhi) {
                            const int64_t gi = tok0 + i;
                            const float sc = dot_row<Tin, DH>(ks[warp], Q + (gi * Hq + h) * DH) * scale;
                            pi = expf(sc - LSE[(int64_t)h * total + gi]);
                            const float dp = dot_row<Tin, DH>(vs[warp], dO + (gi * Hq + h) * DH);
                            dsi = pi * (dp - delta[(int64_t)h * total + gi]);
                        }
                        const int ni = min(32, rhi - i0);
                        for (int ii = 0; ii < ni; ++ii) {
                            const float pb = __shfl_sync(0xffffffffu, pi, ii);
                            const float db = __shfl_sync(0xffffffffu, dsi, ii);
                            const int64_t row = ((tok0 + i0 + ii) * Hq + h) * DH;
#pragma unroll
                            for (int c = 0; c < NC; ++c) {
                                dv[c] = fmaf(pb, ld_f(dO + row + lane + 32 * c), dv[c]);
                                dk[c] = fmaf(db, ld_f(Q + row + lane + 32 * c), dk[c]);
                            }
                        }
                    }
                }
            }
#pragma unroll
            for (int c = 0; c < NC; ++c) dKseg[(krow * Hkv + kvh) * DH + lane + 32 * c] = dk[c] * scale;
        }
#pragma unroll
        for (int c = 0; c < NC; ++c) st_f(dV + (gj * Hkv + kvh) * DH + lane + 32 * c, dv[c]);
        __syncwarp();
    }
}

template <typename Tin, int DH>
mw_status fwd_impl(const mw_vis_layout* L, const void* vis, const void* Q, const void* K, const void* V,
                   void* O, float* LSE, int Hq, int Hkv, float scale, cudaStream_t s) {
    if (L->n_tiles == 0 || Hq == 0) return MW_OK;
    VisView v = make_view(L, vis);
    dim3 grid((unsigned)L->n_tiles, (unsigned)Hq);
    count_launches(1);
    k_attn_fwd_simt<Tin, DH, false><<<grid, 128, 0, s>>>(v, L->total_tokens, (const Tin*)Q, (const Tin*)K,
                                                  (const Tin*)V, (Tin*)O, LSE, Hq, Hkv, scale);
    return launch_status();
}

template <typename Tin, int DH>
mw_status bwd_impl(const mw_vis_layout* L, const void* vis, const void* Q, const void* K, const void* V,
                   const void* O, const void* dO, const float* LSE, void* dQ, void* dK, void* dV, int Hq,
                   int Hkv, float scale, float* delta, cudaStream_t s) {
    if (L->n_tiles == 0 || Hq == 0) return MW_OK;
    VisView v = make_view(L, vis);
    const int64_t warps = L->total_tokens * Hq;
    count_launches(3);
    k_attn_delta<Tin, DH><<<(unsigned)std::min<int64_t>(ceil_div(warps, 8), 152 * 64), 256, 0, s>>>(
        L->total_tokens, Hq, (const Tin*)O, (const Tin*)dO, delta);
    dim3 gq((unsigned)L->n_tiles, (unsigned)Hq);
    k_attn_dq_simt<Tin, DH, false><<<gq, 128, 0, s>>>(v, L->total_tokens, (const Tin*)Q, (const Tin*)K, (const Tin*)V,
                                               (const Tin*)dO, LSE, delta, (Tin*)dQ, Hq, Hkv, scale);
    dim3 gk((unsigned)L->n_tiles, (unsigned)Hkv);
    k_attn_dkv_simt<Tin, DH><<<gk, 128, 0, s>>>(v, L->total_tokens, (const Tin*)Q, (const Tin*)K, (const Tin*)V,
                                                (const Tin*)dO, LSE, delta, (Tin*)dK, (Tin*)dV, Hq, Hkv, scale);
    return launch_status();
}

// Segment-key forward: as fwd_impl with keys from the segment key rows.
template <typename Tin, int DH>
mw_status fwd_segk_impl(const mw_vis_layout* L, const void* vis, const void* Q, const void* Kseg, const void* V,
                        void* O, float* LSE, int Hq, int Hkv, float scale, cudaStream_t s) {
    if (L->n_tiles == 0 || Hq == 0) return MW_OK;
    VisView v = make_view(L, vis);
    dim3 grid((unsigned)L->n_tiles, (unsigned)Hq);
    count_launches(1);
    k_attn_fwd_simt<Tin, DH, true><<<grid, 128, 0, s>>>(v, L->total_tokens, (const Tin*)Q, (const Tin*)Kseg,
                                                        (const Tin*)V, (Tin*)O, LSE, Hq, Hkv, scale);
    return launch_status();
}

// Segment-key backward after Delta: dQ (rotated space), dKseg (float32 per
// segment key row), dV.
template <typename Tin, int DH>
mw_status bwd_segk_impl(const mw_vis_layout* L, const void* vis, const void* Q, const void* Kseg, const void* V,
                        const void* dO, const float* LSE, const float* delta, void* dQ, float* dKseg, void* dV,
                        int Hq, int Hkv, float scale, cudaStream_t s) {
    if (L->n_tiles == 0 || Hq == 0) return MW_OK;
    VisView v = make_view(L, vis);
    count_launches(2);
    dim3 gq((unsigned)L->n_tiles, (unsigned)Hq);
    k_attn_dq_simt<Tin, DH, true><<<gq, 128, 0, s>>>(v, L->total_tokens, (const Tin*)Q, (const Tin*)Kseg,
                                                     (const Tin*)V, (const Tin*)dO, LSE, delta, (Tin*)dQ, Hq, Hkv,
                                                     scale);
    dim3 gk((unsigned)L->n_tiles, (unsigned)Hkv);
    k_attn_dkv_segk_simt<Tin, DH><<<gk, 128, 0, s>>>(v, L->total_tokens, (const Tin*)Q, (const Tin*)Kseg,
                                                     (const Tin*)V, (const Tin*)dO, LSE, delta, dKseg, (Tin*)dV, Hq,
                                                     Hkv, scale);
    return launch_status();
}

}  // namespace

// Delta_i = rowsum(dO_i * O_i) for every (row, head); HBM-bound, shared by
// both backward paths.
mw_status attn_delta(const mw_vis_layout* L, const void* O, const void* dO, int Hq, int Dh, int dtype, float* delta,
                     cudaStream_t s) {
    const int64_t warps = L->total_tokens * Hq;
    if (warps == 0) return MW_OK;
    const unsigned grid = (unsigned)std::min<int64_t>(ceil_div(warps, 8), 152 * 64);
    count_launches(1);
    if (dtype == MW_F32) {
        if (Dh == 64) k_attn_delta<float, 64><<<grid, 256, 0, s>>>(L->total_tokens, Hq, (const float*)O, (const float*)dO, delta);
        else k_attn_delta<float, 128><<<grid, 256, 0, s>>>(L->total_tokens, Hq, (const float*)O, (const float*)dO, delta);
    } else {
        if (Dh == 64)
            k_attn_delta<__nv_bfloat16, 64><<<grid, 256, 0, s>>>(L->total_tokens, Hq, (const __nv_bfloat16*)O,
                                                                 (const __nv_bfloat16*)dO, delta);
        else
            k_attn_delta<__nv_bfloat16, 128><<<grid, 256, 0, s>>>(L->total_tokens, Hq, (const __nv_bfloat16*)O,
                                                                  (const __nv_bfloat16*)dO, delta);
    }
    return launch_status();
}

mw_status attn_fwd_simt(const mw_vis_layout* L, const void* vis, const void* Q, const void* K, const void* V,
                        void* O, float* LSE, int Hq, int Hkv, int Dh, int dtype, float scale, cudaStream_t s) {
    if (dtype == MW_F32) {
        if (Dh == 64) return fwd_impl<float, 64>(L, vis, Q, K, V, O, LSE, Hq, Hkv, scale, s);
        if (Dh == 128) return fwd_impl<float, 128>(L, vis, Q, K, V, O, LSE, Hq, Hkv, scale, s);
    } else {
        if (Dh == 64) return fwd_impl<__nv_bfloat16, 64>(L, vis, Q, K, V, O, LSE, Hq, Hkv, scale, s);
        if (Dh == 128) return fwd_impl<__nv_bfloat16, 128>(L, vis, Q, K, V, O, LSE, Hq, Hkv, scale, s);
    }
    return MW_ESHAPE;
}

mw_status attn_bwd_simt(const mw_vis_layout* L, const void* vis, const void* Q, const void* K, const void* V,
                        const void* O, const void* dO, const float* LSE, void* dQ, void* dK, void* dV, int Hq,
                        int Hkv, int Dh, int dtype, float scale, float* delta, cudaStream_t s) {
    if (dtype == MW_F32) {
        if (Dh == 64) return bwd_impl<float, 64>(L, vis, Q, K, V, O, dO, LSE, dQ, dK, dV, Hq, Hkv, scale, delta, s);
        if (Dh == 128) return bwd_impl<float, 128>(L, vis, Q, K, V, O, dO, LSE, dQ, dK, dV, Hq, Hkv, scale, delta, s);
    } else {
        if (Dh == 64)
            return bwd_impl<__nv_bfloat16, 64>(L, vis, Q, K, V, O, dO, LSE, dQ, dK, dV, Hq, Hkv, scale, delta, s);
        if (Dh == 128)
            return bwd_impl<__nv_bfloat16, 128>(L, vis, Q, K, V, O, dO, LSE, dQ, dK, dV, Hq, Hkv, scale, delta, s);
    }
    return MW_ESHAPE;
}

mw_status attn_fwd_simt_segk(const mw_vis_layout* L, const void* vis, const void* Q, const void* Kseg,
                             const void* V, void* O, float* LSE, int Hq, int Hkv, int Dh, int dtype, float scale,
                             cudaStream_t s) {
    if (dtype == MW_F32) {
        if (Dh == 64) return fwd_segk_impl<float, 64>(L, vis, Q, Kseg, V, O, LSE, Hq, Hkv, scale, s);
        if (Dh == 128) return fwd_segk_impl<float, 128>(L, vis, Q, Kseg, V, O, LSE, Hq, Hkv, scale, s);
    } else {
        if (Dh == 64) return fwd_segk_impl<__nv_bfloat16, 64>(L, vis, Q, Kseg, V, O, LSE, Hq, Hkv, scale, s);
        if (Dh == 128) return fwd_segk_impl<__nv_bfloat16, 128>(L, vis, Q, Kseg, V, O, LSE, Hq, Hkv, scale, s);
    }
    return MW_ESHAPE;
}

mw_status attn_bwd_simt_segk(const mw_vis_layout* L, const void* vis, const void* Q, const void* Kseg,
                             const void* V, const void* dO, const float* LSE, const float* delta, void* dQ,
                             float* dKseg, void* dV, int Hq, int Hkv, int Dh, int dtype, float scale,
                             cudaStream_t s) {
    if (dtype == MW_F32) {
        if (Dh == 64)
            return bwd_segk_impl<float, 64>(L, vis, Q, Kseg, V, dO, LSE, delta, dQ, dKseg, dV, Hq, Hkv, scale, s);
        if (Dh == 128)
            return bwd_segk_impl<float, 128>(L, vis, Q, Kseg, V, dO, LSE, delta, dQ, dKseg, dV, Hq, Hkv, scale, s);
    } else {
        if (Dh == 64)
            return bwd_segk_impl<__nv_bfloat16, 64>(L, vis, Q, Kseg, V, dO, LSE, delta, dQ, dKseg, dV, Hq, Hkv,
                                                    scale, s);
        if (Dh == 128)
            return bwd_segk_impl<__nv_bfloat16, 128>(L, vis, Q, Kseg, V, dO, LSE, delta, dQ, dKseg, dV, Hq, Hkv,
                                                     scale, s);
    }
    return MW_ESHAPE;
}

}  // namespace mw
