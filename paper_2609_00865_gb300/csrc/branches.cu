// Branch-replicated packing for stacked layers (App. G).
//
// From the second layer on, a token's state differs between the branches
// (segments' live views) that hold it: inside branch s it was computed from
// the keys that survived to s. The exact multi-layer step therefore runs
// every branch's compact sequence -- its live view in order, as §4.1
// materialises it -- through all layers. These two kernels move per-token
// rows between the physical layout and the packed branches, using the
// visibility build's compact views (csrc, cpos, seg_len):
//   pack        Xp[off_g + c] = X[csrc_g(c)]   for c < |view_g|
//   unpack_add  dX[j] = sum over segments g holding j, in segment order, of
//               dXp[off_g + cpos_g(j)]
// with the branches back to back in global segment order, off_g the sum of
// the earlier segments' lengths. A row is `row_elems` elements of the dtype;
// both kernels copy 16-byte vectors.

#include "common.cuh"

namespace mw {
namespace {

// first packed row of global segment g: the earlier segments' lengths
__device__ __forceinline__ int64_t branch_off(const VisView& v, int g) {
    int64_t o = 0;
    for (int q = 0; q < g; ++q) o += v.seg_len[q];
    return o;
}

// One block per (segment, 128-row compact tile) entry with rows in it.
__global__ void __launch_bounds__(256) k_branch_pack(VisView v, int n_traj, int vec, const uint4* __restrict__ X,
                                                     uint4* __restrict__ Xp) {
    const int64_t e = blockIdx.x;
    int lo = 0, hi = n_traj;   // the trajectory holding entry e: largest b with traj_km[b] <= e
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (v.traj_km[mid] <= e) lo = mid; else hi = mid;
    }
    const int b = lo;
    const int nt = v.traj_tile[b + 1] - v.traj_tile[b];
    const int64_t rel = e - v.traj_km[b];
    const int s = (int)(rel / nt), kt = (int)(rel - (int64_t)s * nt);
    const int g = v.traj_seg[b] + s;
    const int len = v.seg_len[g];
    if (kt * MW_TILE >= len) return;
    __shared__ int64_t off;
    if (threadIdx.x == 0) off = branch_off(v, g);
    __syncthreads();
    const int64_t tok0 = v.traj_tok[b];
    const int rows = min(MW_TILE, len - kt * MW_TILE);
    for (int x = threadIdx.x; x < rows * vec; x += blockDim.x) {
        const int r = x / vec, k = x - r * vec;
        const int c = kt * MW_TILE + r;
        const int j = v.csrc[e * MW_TILE + r];
        if (MW_DBG_IN(j, v.traj_tok[b + 1] - tok0, v.status, 301)) Xp[(off + c) * vec + k] = X[(tok0 + j) * vec + k];
    }
}

// One block per key tile; a thread sums one 16-byte vector of one key's row
// over the segments holding the key (a key enters the views at its own
// segment), float32 accumulation. With at most SCH segments per trajectory
// the packed row of every (segment, key) of the tile is looked up once into
// shared memory first, so a thread's loads of the key's copies do not wait on
// one another's ranks. (Measured on the attention workload's packed branches:
// 0.61 -> 0.58 ms per call, about 0.42 of the copy bandwidth either way.)
constexpr int SCH = 16;
template <typename T>
__global__ void __launch_bounds__(256) k_branch_unpack_add(VisView v, int vec, const uint4* __restrict__ dXp,
                                                           uint4* __restrict__ dX) {
    constexpr int PER = 16 / sizeof(T);   // elements per vector
    __shared__ int64_t off[64];
    __shared__ int64_t prow[SCH][MW_TILE];   // packed row of key r in segment s, -1 if the view lacks it
    const int64_t g = blockIdx.x;
    const int b = v.tile_traj[g];
    const int nt = v.traj_tile[b + 1] - v.traj_tile[b];
    const int kt = (int)(g - v.traj_tile[b]);
    const int64_t tok0 = v.traj_tok[b];
    const int T_b = v.traj_tok[b + 1] - (int)tok0;
    const int g0 = v.traj_seg[b], nseg = v.traj_seg[b + 1] - g0;
    for (int s = threadIdx.x; s < nseg && s < 64; s += blockDim.x) off[s] = branch_off(v, g0 + s);
    __syncthreads();
    // the packed row of key j's copy in segment s (-1 if none)
    auto packed_row = [&](int s, int j) -> int64_t {
        const int c = v.cpos[(v.traj_km[b] + (int64_t)s * nt) * MW_TILE + j];
        if (c < 0 || !MW_DBG_IN(c, v.seg_len[g0 + s], v.status, 302)) return -1;
        return (s < 64 ? off[s] : branch_off(v, g0 + s)) + c;
    };
    const bool staged = nseg <= SCH;   // uniform over the block
    if (staged) {
        for (int e = threadIdx.x; e < SCH * MW_TILE; e += blockDim.x) {
            const int s = e / MW_TILE, r = e - s * MW_TILE;
            const int j = kt * MW_TILE + r;
            prow[s][r] = (s < nseg && j < T_b && s >= v.seg[tok0 + j]) ? packed_row(s, j) : -1;
        }
        __syncthreads();
    }
    // (key r, vector k) of x = r vec + k, advanced by the block size without a
    // division per step
    int r = threadIdx.x / vec, k = threadIdx.x - r * vec;
    const int rstep = blockDim.x / vec, kstep = blockDim.x - rstep * vec;
    for (; r < MW_TILE; r += rstep, k += kstep) {
        if (k >= vec) {
            k -= vec;
            ++r;
            if (r >= MW_TILE) break;
        }
        const int j = kt * MW_TILE + r;
        if (j >= T_b) break;   // later keys of the tile are past the trajectory too
        float acc[PER];
#pragma unroll
        for (int q = 0; q < PER; ++q) acc[q] = 0.f;
        auto add = [&](const uint4& u) {
            const T* t = reinterpret_cast<const T*>(&u);
#pragma unroll
            for (int q = 0; q < PER; ++q) acc[q] += ld_f(t + q);
        };
        if (staged) {
            // four copies' loads in flight at a time
            for (int s0 = 0; s0 < nseg; s0 += 4) {
                uint4 u[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int64_t pr = s0 + q < SCH ? prow[s0 + q][r] : -1;
                    u[q] = pr >= 0 ? __ldg(dXp + pr * vec + k) : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    if (s0 + q < SCH && prow[s0 + q][r] >= 0) add(u[q]);
            }
        } else {
            for (int s = v.seg[tok0 + j]; s < nseg; ++s) {
                const int64_t pr = packed_row(s, j);
                if (pr >= 0) add(dXp[pr * vec + k]);
            }
        }
        uint4 u;
        T* t = reinterpret_cast<T*>(&u);
#pragma unroll
        for (int q = 0; q < PER; ++q) st_f(t + q, acc[q]);
        dX[(tok0 + j) * vec + k] = u;
    }
}

}  // namespace
}  // namespace mw

using namespace mw;

static mw_status branch_args(const mw_vis_layout* L, const void* vis, int row_elems, int dtype) {
    if (!L || !vis) return MW_EINVAL;
    if (dtype != MW_F32 && dtype != MW_BF16) return MW_EDTYPE;
    const int esz = dtype == MW_F32 ? 4 : 2;
    if (row_elems <= 0 || (row_elems * esz) % 16) return MW_ESHAPE;
    return MW_OK;
}

extern "C" mw_status mw_branch_pack(const mw_vis_layout* L, const void* vis, const void* X, void* Xp, int row_elems,
                                    int dtype, void* stream) {
    mw_status st = branch_args(L, vis, row_elems, dtype);
    if (st != MW_OK) return st;
    if (L->n_keymask == 0) return MW_OK;
    if (!X || !Xp) return MW_EINVAL;
    const int vec = row_elems * (dtype == MW_F32 ? 4 : 2) / 16;
    count_launches(1);
    k_branch_pack<<<(unsigned)L->n_keymask, 256, 0, (cudaStream_t)stream>>>(
        make_view(L, vis), L->n_traj, vec, (const uint4*)X, (uint4*)Xp);
    return launch_status();
}

extern "C" mw_status mw_branch_unpack_add(const mw_vis_layout* L, const void* vis, const void* dXp, void* dX,
                                          int row_elems, int dtype, void* stream) {
    mw_status st = branch_args(L, vis, row_elems, dtype);
    if (st != MW_OK) return st;
    if (L->n_tiles == 0) return MW_OK;
    if (!dXp || !dX) return MW_EINVAL;
    const int vec = row_elems * (dtype == MW_F32 ? 4 : 2) / 16;
    count_launches(1);
    if (dtype == MW_F32)
        k_branch_unpack_add<float><<<(unsigned)L->n_tiles, 256, 0, (cudaStream_t)stream>>>(
            make_view(L, vis), vec, (const uint4*)dXp, (uint4*)dX);
    else
        k_branch_unpack_add<__nv_bfloat16><<<(unsigned)L->n_tiles, 256, 0, (cudaStream_t)stream>>>(
            make_view(L, vis), vec, (const uint4*)dXp, (uint4*)dX);
    return launch_status();
}
