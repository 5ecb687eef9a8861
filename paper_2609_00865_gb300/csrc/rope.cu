// Row-wise logical positions and rotary position embedding (§4.2).
//
// The paper reassigns position ids so that the keys each row sees form a
// gap-free sequence (condition (ii) of the 4D-mask equivalence proposition,
// App. C). In segment s the key at physical position j then sits at its rank
// in the segment's live view, p_s(j) = #{view members before j}. That rank is
// a prefix popcount of the per-(segment, k-tile) view bits the visibility
// builder already stores, so the positions cost one scan per segment.
//
// Rotary embedding (RoFormer, rotate-half pairing): feature f < Dh/2 is paired
// with f + Dh/2 and the pair is turned by p * theta^(-2f/Dh). A key's rotation
// depends on the segment of the row that reads it, so the attention reads
// keys from per-segment copies ("segment key rows"): row (traj_km[b] + s nt_b)
// * 128 + j holds key j of trajectory b rotated for segment s (zero where j
// is not in view_s). All kernels here are HBM-bound element-wise passes.

#include <math.h>

#include <algorithm>

#include "common.cuh"

namespace mw {
namespace {

struct TrajRef {
    int b, kt;
    int64_t tok0;
    int T, nt, nseg;
    int64_t kmb;
};

// Trajectory-local coordinates of global k-tile (or q-tile) g.
__device__ __forceinline__ TrajRef traj_of_tile(const VisView& v, int64_t g) {
    TrajRef r;
    r.b = v.tile_traj[g];
    r.kt = (int)(g - v.traj_tile[r.b]);
    r.tok0 = v.traj_tok[r.b];
    r.T = v.traj_tok[r.b + 1] - (int)r.tok0;
    r.nt = v.traj_tile[r.b + 1] - v.traj_tile[r.b];
    r.nseg = v.traj_seg[r.b + 1] - v.traj_seg[r.b];
    r.kmb = v.traj_km[r.b];
    return r;
}

// One block per global segment: exclusive prefix popcount of its view bits,
// tile by tile, then every key's rank (or -1) with coalesced stores.
__global__ void __launch_bounds__(256) k_logical_pos(VisView v, int n_traj, int32_t* __restrict__ pos) {
    __shared__ int tp[256];
    __shared__ int wsum[8];
    __shared__ int carry_s;
    const int sg = blockIdx.x;
    int lo = 0, hi = n_traj;  // largest b with traj_seg[b] <= sg
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (v.traj_seg[mid] <= sg) lo = mid; else hi = mid;
    }
    const int b = lo;
    const int s = sg - v.traj_seg[b];
    const int nt = v.traj_tile[b + 1] - v.traj_tile[b];
    const int64_t ent0 = v.traj_km[b] + (int64_t)s * nt;   // keymask entry of (s, kt = 0)
    const uint32_t* km = v.keymask + ent0 * 4;
    int32_t* out = pos + ent0 * MW_TILE;
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    if (t == 0) carry_s = 0;
    __syncthreads();
    for (int c0 = 0; c0 < nt; c0 += 256) {
        const int kt = c0 + t;
        int cnt = 0;
        if (kt < nt)
            cnt = __popc(km[4 * kt]) + __popc(km[4 * kt + 1]) + __popc(km[4 * kt + 2]) + __popc(km[4 * kt + 3]);
        int incl = cnt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) wsum[w] = incl;
        __syncthreads();
        int before = carry_s;
        for (int q = 0; q < w; ++q) before += wsum[q];
        tp[t] = before + incl - cnt;
        __syncthreads();
        const int ntc = min(256, nt - c0);
        for (int k = t; k < ntc * MW_TILE; k += 256) {
            const int tl = k >> 7, jj = k & 127, wd = jj >> 5, bit = jj & 31;
            const uint32_t* tw = km + 4 * (c0 + tl);
            const uint32_t word = tw[wd];
            int32_t r = -1;
            if ((word >> bit) & 1u) {
                r = tp[tl] + __popc(word & ((1u << bit) - 1u));
                for (int q = 0; q < wd; ++q) r += __popc(tw[q]);
            }
            out[(int64_t)(c0 + tl) * MW_TILE + jj] = r;
        }
        __syncthreads();
        if (t == 255) carry_s = tp[255] + cnt;
        __syncthreads();
    }
}

// table[p][f] = (cos, sin)(p theta^(-2f/Dh)), evaluated in double and rounded.
__global__ void k_rope_table(int64_t n, int half, int Dh, double theta, float2* __restrict__ table) {
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t p = i / half;
        const int f = (int)(i - p * half);
        const double a = (double)p * pow(theta, -2.0 * f / Dh);
        double sn, cs;
        sincos(a, &sn, &cs);
        table[i] = make_float2((float)cs, (float)sn);
    }
}

// Turn the pair (x0, x1) by the table angle of position p (sgn = -1: back).
__device__ __forceinline__ void rotate(float x0, float x1, float2 cs, float sgn, float& y0, float& y1) {
    const float sn = sgn * cs.y;
    y0 = fmaf(x0, cs.x, -x1 * sn);
    y1 = fmaf(x1, cs.x, x0 * sn);
}

// Bounds of a position against the table; a miss is recorded, not trapped.
__device__ __forceinline__ bool pos_ok(const VisView& v, int p, int n_pos) {
    if (p >= 0 && p < n_pos) return true;
    atomicExch(v.status + ST_BOUNDS, 1);
    return false;
}

// Y_i = R(+-p(seg(i), i)) X_i for every row; one block per q-tile. X may be Y.
template <typename T>
__global__ void __launch_bounds__(256) k_rope_rows(VisView v, const int32_t* __restrict__ pos,
                                                   const float2* __restrict__ table, int n_pos, const T* X, T* Y,
                                                   int H, int Dh, float sgn) {
    const TrajRef r = traj_of_tile(v, blockIdx.x);
    const int half = Dh >> 1;
    const int rows = min(MW_TILE, r.T - r.kt * MW_TILE);
    const int per_row = H * half;
    for (int e = threadIdx.x; e < rows * per_row; e += blockDim.x) {
        const int jj = e / per_row, rem = e - jj * per_row;
        const int h = rem / half, f = rem - h * half;
        const int i = r.kt * MW_TILE + jj;
        const int64_t gi = r.tok0 + i;
        const int s = v.seg[gi];
        const int p = pos[(r.kmb + (int64_t)s * r.nt) * MW_TILE + i];
        const int64_t o = (gi * H + h) * Dh + f;
        float y0 = 0.f, y1 = 0.f;
        if (pos_ok(v, p, n_pos)) rotate(ld_f(X + o), ld_f(X + o + half), table[(int64_t)p * half + f], sgn, y0, y1);
        st_f(Y + o, y0);
        st_f(Y + o + half, y1);
    }
}

// The same with 16-byte vectors: a thread turns VEC consecutive features of
// both halves of one (row, head), with the VEC table entries as float4 loads.
// Needs half a row (Dh / 2 elements) to be whole vectors and X, Y 16-byte
// aligned (checked by the launcher).
template <typename T>
__global__ void __launch_bounds__(256) k_rope_rows_vec(VisView v, const int32_t* __restrict__ pos,
                                                       const float2* __restrict__ table, int n_pos, const T* X, T* Y,
                                                       int H, int Dh, float sgn) {
    constexpr int VEC = 16 / sizeof(T);
    const TrajRef r = traj_of_tile(v, blockIdx.x);
    const int half = Dh >> 1;
    const int hv = half / VEC;   // vectors per half row
    const int rows = min(MW_TILE, r.T - r.kt * MW_TILE);
    const int per_row = H * hv;
    for (int e = threadIdx.x; e < rows * per_row; e += blockDim.x) {
        const int jj = e / per_row, rem = e - jj * per_row;
        const int h = rem / hv, f = (rem - h * hv) * VEC;
        const int i = r.kt * MW_TILE + jj;
        const int64_t gi = r.tok0 + i;
        const int s = v.seg[gi];
        const int p = pos[(r.kmb + (int64_t)s * r.nt) * MW_TILE + i];
        const int64_t o = (gi * H + h) * Dh + f;
        uint4 y0v = make_uint4(0u, 0u, 0u, 0u), y1v = y0v;
        if (pos_ok(v, p, n_pos)) {
            const uint4 x0v = *reinterpret_cast<const uint4*>(X + o), x1v = *reinterpret_cast<const uint4*>(X + o + half);
            const T* x0 = reinterpret_cast<const T*>(&x0v);
            const T* x1 = reinterpret_cast<const T*>(&x1v);
            T* y0 = reinterpret_cast<T*>(&y0v);
            T* y1 = reinterpret_cast<T*>(&y1v);
            const float4* tb = reinterpret_cast<const float4*>(table + (int64_t)p * half + f);
#pragma unroll
            for (int q = 0; q < VEC / 2; ++q) {
                const float4 cs = tb[q];
                float a0, a1, b0, b1;
                rotate(ld_f(x0 + 2 * q), ld_f(x1 + 2 * q), make_float2(cs.x, cs.y), sgn, a0, a1);
                rotate(ld_f(x0 + 2 * q + 1), ld_f(x1 + 2 * q + 1), make_float2(cs.z, cs.w), sgn, b0, b1);
                st_f(y0 + 2 * q, a0);
                st_f(y1 + 2 * q, a1);
                st_f(y0 + 2 * q + 1, b0);
                st_f(y1 + 2 * q + 1, b1);
            }
        }
        *reinterpret_cast<uint4*>(Y + o) = y0v;
        *reinterpret_cast<uint4*>(Y + o + half) = y1v;
    }
}

// Segment key rows: Y[(kmb + s nt) 128 + j] = R(p_s(j)) X[j], zero off-view.
template <typename T>
__global__ void __launch_bounds__(256) k_rope_segments(VisView v, const int32_t* __restrict__ pos,
                                                       const float2* __restrict__ table, int n_pos,
                                                       const T* __restrict__ X, T* __restrict__ Y, int H, int Dh) {
    const TrajRef r = traj_of_tile(v, blockIdx.x);
    const int half = Dh >> 1;
    const int per_row = H * half;
    for (int s = 0; s < r.nseg; ++s) {
        const int64_t row0 = (r.kmb + (int64_t)s * r.nt + r.kt) * MW_TILE;
        for (int e = threadIdx.x; e < MW_TILE * per_row; e += blockDim.x) {
            const int jj = e / per_row, rem = e - jj * per_row;
            const int h = rem / half, f = rem - h * half;
            const int p = pos[row0 + jj];
            float y0 = 0.f, y1 = 0.f;
            if (p >= 0 && pos_ok(v, p, n_pos)) {
                const int64_t xi = ((r.tok0 + r.kt * MW_TILE + jj) * H + h) * Dh + f;
                rotate(ld_f(X + xi), ld_f(X + xi + half), table[(int64_t)p * half + f], 1.f, y0, y1);
            }
            const int64_t yo = ((row0 + jj) * H + h) * Dh + f;
            st_f(Y + yo, y0);
            st_f(Y + yo + half, y1);
        }
    }
}

// Transpose of k_rope_segments: dX[j] = sum_{s: j in view_s} R(p_s(j))^T dY_s[j]
// (ROT = false: the plain sum over those segments, for values read unrotated).
template <typename T, bool ROT>
__global__ void __launch_bounds__(256) k_rope_segments_bwd(VisView v, const int32_t* __restrict__ pos,
                                                           const float2* __restrict__ table, int n_pos,
                                                           const float* __restrict__ dY, T* __restrict__ dX,
                                                           int H, int Dh) {
    const TrajRef r = traj_of_tile(v, blockIdx.x);
    const int half = Dh >> 1;
    const int per_row = H * half;
    const int rows = min(MW_TILE, r.T - r.kt * MW_TILE);
    for (int e = threadIdx.x; e < rows * per_row; e += blockDim.x) {
        const int jj = e / per_row, rem = e - jj * per_row;
        const int h = rem / half, f = rem - h * half;
        float a0 = 0.f, a1 = 0.f;
        for (int s = 0; s < r.nseg; ++s) {
            const int64_t row = (r.kmb + (int64_t)s * r.nt + r.kt) * MW_TILE + jj;
            const int p = pos[row];
            if (p < 0) continue;
            const int64_t yo = (row * H + h) * Dh + f;
            if (ROT) {
                if (!pos_ok(v, p, n_pos)) continue;
                float y0, y1;
                rotate(dY[yo], dY[yo + half], table[(int64_t)p * half + f], -1.f, y0, y1);
                a0 += y0;
                a1 += y1;
            } else {
                a0 += dY[yo];
                a1 += dY[yo + half];
            }
        }
        const int64_t xo = ((r.tok0 + r.kt * MW_TILE + jj) * H + h) * Dh + f;
        st_f(dX + xo, a0);
        st_f(dX + xo + half, a1);
    }
}

}  // namespace

mw_status logical_positions(const mw_vis_layout* L, const void* vis, int32_t* pos, cudaStream_t s) {
    if (L->n_segs == 0 || L->n_tiles == 0) return MW_OK;
    count_launches(1);
    k_logical_pos<<<(unsigned)L->n_segs, 256, 0, s>>>(make_view(L, vis), L->n_traj, pos);
    return launch_status();
}

mw_status rope_table(int n_pos, int Dh, double theta, float* table, cudaStream_t s) {
    const int64_t n = (int64_t)n_pos * (Dh / 2);
    if (n == 0) return MW_OK;
    count_launches(1);
    k_rope_table<<<(unsigned)std::min<int64_t>(ceil_div(n, 256), 152 * 16), 256, 0, s>>>(
        n, Dh / 2, Dh, theta, reinterpret_cast<float2*>(table));
    return launch_status();
}

mw_status rope_rows(const mw_vis_layout* L, const void* vis, const int32_t* pos, const float* table, int n_pos,
                    const void* X, void* Y, int H, int Dh, int dtype, bool inverse, cudaStream_t s) {
    if (L->n_tiles == 0 || H == 0) return MW_OK;
    VisView v = make_view(L, vis);
    const float2* tb = reinterpret_cast<const float2*>(table);
    const float sgn = inverse ? -1.f : 1.f;
    count_launches(1);
    const int esz = dtype == MW_F32 ? 4 : 2;
    const bool vec = ((Dh / 2) * esz) % 16 == 0 && ((uintptr_t)X | (uintptr_t)Y) % 16 == 0;
    if (dtype == MW_F32) {
        if (vec)
            k_rope_rows_vec<float><<<(unsigned)L->n_tiles, 256, 0, s>>>(v, pos, tb, n_pos, (const float*)X, (float*)Y,
                                                                        H, Dh, sgn);
        else
            k_rope_rows<float><<<(unsigned)L->n_tiles, 256, 0, s>>>(v, pos, tb, n_pos, (const float*)X, (float*)Y, H,
                                                                    Dh, sgn);
    } else {
        if (vec)
            k_rope_rows_vec<__nv_bfloat16><<<(unsigned)L->n_tiles, 256, 0, s>>>(
                v, pos, tb, n_pos, (const __nv_bfloat16*)X, (__nv_bfloat16*)Y, H, Dh, sgn);
        else
            k_rope_rows<__nv_bfloat16><<<(unsigned)L->n_tiles, 256, 0, s>>>(
                v, pos, tb, n_pos, (const __nv_bfloat16*)X, (__nv_bfloat16*)Y, H, Dh, sgn);
    }
    return launch_status();
}

mw_status rope_segments(const mw_vis_layout* L, const void* vis, const int32_t* pos, const float* table, int n_pos,
                        const void* X, void* Y, int H, int Dh, int dtype, cudaStream_t s) {
    if (L->n_tiles == 0 || H == 0) return MW_OK;
    VisView v = make_view(L, vis);
    const float2* tb = reinterpret_cast<const float2*>(table);
    count_launches(1);
    if (dtype == MW_F32)
        k_rope_segments<float><<<(unsigned)L->n_tiles, 256, 0, s>>>(v, pos, tb, n_pos, (const float*)X, (float*)Y,
                                                                    H, Dh);
    else
        k_rope_segments<__nv_bfloat16><<<(unsigned)L->n_tiles, 256, 0, s>>>(
            v, pos, tb, n_pos, (const __nv_bfloat16*)X, (__nv_bfloat16*)Y, H, Dh);
    return launch_status();
}

mw_status rope_segments_bwd(const mw_vis_layout* L, const void* vis, const int32_t* pos, const float* table,
                            int n_pos, const float* dY, void* dX, int H, int Dh, int dtype, bool rotate_back,
                            cudaStream_t s) {
    if (L->n_tiles == 0 || H == 0) return MW_OK;
    VisView v = make_view(L, vis);
    const float2* tb = reinterpret_cast<const float2*>(table);
    const unsigned grid = (unsigned)L->n_tiles;
    count_launches(1);
    if (dtype == MW_F32) {
        if (rotate_back)
            k_rope_segments_bwd<float, true><<<grid, 256, 0, s>>>(v, pos, tb, n_pos, dY, (float*)dX, H, Dh);
        else
            k_rope_segments_bwd<float, false><<<grid, 256, 0, s>>>(v, pos, tb, n_pos, dY, (float*)dX, H, Dh);
    } else {
        if (rotate_back)
            k_rope_segments_bwd<__nv_bfloat16, true><<<grid, 256, 0, s>>>(v, pos, tb, n_pos, dY, (__nv_bfloat16*)dX,
                                                                           H, Dh);
        else
            k_rope_segments_bwd<__nv_bfloat16, false><<<grid, 256, 0, s>>>(v, pos, tb, n_pos, dY, (__nv_bfloat16*)dX,
                                                                            H, Dh);
    }
    return launch_status();
}

}  // namespace mw
