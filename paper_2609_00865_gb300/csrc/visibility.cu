// Visibility builder: record -> lifetimes, segments, tile classes, tile lists.
//
// Lifetimes follow the 4D mask of §4.2: key j is visible to row i iff
// j <= i < omega(j), omega(j) = min{J_k : j in E_k}. Segments are the branch
// layers of App. B.1 (rows [J_k, J_{k+1})). Everything here is O(T + tiles):
// a tile's class follows from the min / max lifetime of its keys, because on an
// off-diagonal tile (keys all before the rows) visibility depends on the row
// only through i < omega(j).

#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <mutex>
#include <vector>

#include "common.cuh"

namespace mw {

// tiles per block of the list-pointer scan
constexpr int SCAN_BLOCK = 1024;

static thread_local int g_last_cuda_error = 0;

mw_status cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return MW_OK;
    g_last_cuda_error = (int)e;
    return MW_ECUDA;
}
mw_status launch_status() { return cuda_status(cudaGetLastError()); }

static std::atomic<unsigned long long> g_launches{0};
void count_launches(int n) { g_launches.fetch_add((unsigned long long)n, std::memory_order_relaxed); }

}  // namespace mw

using namespace mw;

extern "C" const char* mw_status_str(int s) {
    switch (s) {
        case MW_OK: return "ok";
        case MW_EINVAL: return "invalid argument";
        case MW_EEDITS: return "record breaks the junction/span conventions";
        case MW_ESHAPE: return "unsupported or inconsistent shape";
        case MW_EDTYPE: return "unsupported dtype";
        case MW_ECUDA: return "CUDA runtime error";
        case MW_ETIMEOUT: return "bounded device wait timed out";
        case MW_EDEVICE: return "device-side check failed";
        case MW_ENOSPACE: return "request exceeds a fixed capacity";
        default: return "unknown status";
    }
}

extern "C" int mw_last_cuda_error(void) { return g_last_cuda_error; }
extern "C" int mw_abi_version(void) { return 7; }
extern "C" int mw_build_flags(void) {
#ifdef MW_DEBUG
    return MW_BUILD_DEBUG;
#else
    return 0;
#endif
}
extern "C" uint64_t mw_kernel_launches(void) { return (uint64_t)g_launches.load(std::memory_order_relaxed); }

static mw_status check_shape(int n_traj, const int32_t* cu, int n_junc, const int32_t* jt,
                             int n_spans) {
    if (n_traj < 0 || n_junc < 0 || n_spans < 0) return MW_EINVAL;
    if (n_traj > 0 && !cu) return MW_EINVAL;
    if (n_junc > 0 && !jt) return MW_EINVAL;
    if (n_traj > 0 && cu[0] != 0) return MW_EEDITS;
    for (int b = 0; b < n_traj; ++b)
        if (cu[b + 1] < cu[b]) return MW_EEDITS;
    for (int k = 0; k < n_junc; ++k) {
        if (jt[k] < 0 || jt[k] >= n_traj) return MW_EEDITS;
        if (k > 0 && jt[k] < jt[k - 1]) return MW_EEDITS;
    }
    return MW_OK;
}

extern "C" mw_status mw_visibility_layout(int n_traj, const int32_t* cu, int n_junc,
                                          const int32_t* jt, int n_spans, mw_vis_layout* L) {
    if (!L) return MW_EINVAL;
    mw_status st = check_shape(n_traj, cu, n_junc, jt, n_spans);
    if (st != MW_OK) return st;
    memset(L, 0, sizeof(*L));
    L->n_traj = n_traj;
    L->n_junc = n_junc;
    L->n_spans = n_spans;
    int64_t tiles = 0, tri = 0, km = 0, max_segs = 0;
    int max_tiles = 0;
    int k = 0;
    for (int b = 0; b < n_traj; ++b) {
        int64_t T = cu[b + 1] - cu[b];
        int64_t nt = ceil_div(T, MW_TILE);
        int Kb = 0;
        while (k < n_junc && jt[k] == b) { ++Kb; ++k; }
        tiles += nt;
        tri += nt * (nt + 1) / 2;
        km += (1 + Kb) * nt;
        if (nt > max_tiles) max_tiles = (int)nt;
        if (1 + Kb > max_segs) max_segs = 1 + Kb;
    }
    L->max_tiles = max_tiles;
    L->total_tokens = n_traj > 0 ? cu[n_traj] : 0;
    L->n_tiles = tiles;
    L->n_tri = tri;
    L->n_segs = (int64_t)n_traj + n_junc;
    L->n_keymask = km;
    int64_t o = 0;
    auto take = [&](int64_t bytes) { int64_t r = o; o = align256(o + bytes); return r; };
    L->off_omega = take(4 * L->total_tokens);
    L->off_seg = take(4 * L->total_tokens);
    L->off_traj_tok = take(4 * (n_traj + 1));
    L->off_traj_tile = take(4 * (n_traj + 1));
    L->off_traj_seg = take(4 * (n_traj + 1));
    L->off_traj_tri = take(8 * (n_traj + 1));
    L->off_traj_km = take(8 * (n_traj + 1));
    L->off_seg_start = take(4 * L->n_segs);
    L->off_tile_traj = take(4 * tiles);
    L->off_cls = take(tri);
    L->off_fwd_ptr = take(4 * (tiles + 1));
    L->off_fwd_idx = take(4 * tri);
    L->off_bwd_ptr = take(4 * (tiles + 1));
    L->off_bwd_idx = take(4 * tri);
    L->off_pairs = take(8 * (n_traj + 1));
    L->off_keymask = take(16 * km);
    L->off_status = take(4 * 8);
    L->off_seg_len = take(4 * L->n_segs);
    L->off_cpos = take(4 * MW_TILE * km);
    L->off_csrc = take(4 * MW_TILE * km);
    L->vis_bytes = o;
    o = 0;
    L->ws_off_spans = take(12 * (int64_t)n_spans);
    L->ws_off_tstat = take(16 * tiles);
    // fwd / bwd counts [2][tiles] int32, per-tile pairs [tiles] uint64, the
    // scan's per-block sums and offsets [2][2][scan blocks] int32
    L->ws_off_cnt = take(8 * tiles + 8 * tiles + 16 * ceil_div(tiles, (int64_t)SCAN_BLOCK));
    L->ws_bytes = o;
    L->max_segs = max_segs;
    return MW_OK;
}

extern "C" mw_status mw_events_layout(int n_traj, const int32_t* cu, int n_junc, const int32_t* jt, int n_spans,
                                      mw_vis_layout* L) {
    mw_status st = mw_visibility_layout(n_traj, cu, n_junc, jt, n_spans, L);
    if (st != MW_OK) return st;
    L->kind = MW_VIEWS_EVENTS;
    // build workspace: spans (a, b), the per-event span ranges, one flag per token
    int64_t o = 0;
    auto take = [&](int64_t bytes) { int64_t r = o; o = align256(o + bytes); return r; };
    L->ws_off_spans = take(8 * (int64_t)n_spans);
    L->ws_off_tstat = take(16 * (int64_t)n_junc);
    L->ws_off_cnt = take(4 * L->total_tokens);
    L->ws_bytes = o;
    return MW_OK;
}

// ---------------------------------------------------------------------------
// kernels

namespace {

struct BuildArgs {
    int n_traj;
    int64_t total;
    int64_t n_tiles;
    int n_spans;
    int32_t* omega;
    int32_t* seg;
    const int32_t* traj_tok;
    const int32_t* traj_tile;
    const int32_t* traj_seg;
    const int64_t* traj_tri;
    const int64_t* traj_km;
    const int32_t* seg_start;
    const int32_t* tile_traj;
    uint8_t* cls;
    int32_t* fwd_ptr;
    int32_t* fwd_idx;
    int32_t* bwd_ptr;
    int32_t* bwd_idx;
    unsigned long long* pairs;
    uint32_t* keymask;
    int32_t* seg_len;       // [n_segs]
    int32_t* cpos;          // [n_keymask][128]
    int32_t* csrc;          // [n_keymask][128]
    const int32_t* spans;   // [n_spans][3]
    int32_t* tstat;         // [n_tiles][4] min, max lifetime; max over keys 0..63, 64..127
    int32_t* fwd_cnt;       // [n_tiles]
    int32_t* bwd_cnt;       // [n_tiles]
    unsigned long long* tpairs;   // [n_tiles] visible pairs per k-tile
    int32_t* bsum;          // [2][n_scan_blocks] per-block count sums, then exclusive offsets
    int32_t* status;        // device status words (debug index checks)
    int64_t n_tri, n_keymask;
};

__device__ __forceinline__ int find_traj(const int32_t* off, int n, int64_t t) {
    int lo = 0, hi = n;  // off[lo] <= t < off[hi]
    while (hi - lo > 1) {
        int mid = (lo + hi) >> 1;
        if (off[mid] <= t) lo = mid; else hi = mid;
    }
    return lo;
}

// omega = never; seg = number of junctions <= local row. A thread takes 16
// consecutive tokens: one search for the first token's trajectory and
// segment, then it steps across boundaries, and stores 64-byte runs.
constexpr int INIT_TPT = 16;
__global__ void k_init_tokens(BuildArgs a) {
    const int64_t n_chunks = (a.total + INIT_TPT - 1) / INIT_TPT;
    for (int64_t c = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; c < n_chunks;
         c += (int64_t)gridDim.x * blockDim.x) {
        const int64_t t0 = c * INIT_TPT;
        int b = find_traj(a.traj_tok, a.n_traj, t0);
        int s0 = a.traj_seg[b], s1 = a.traj_seg[b + 1];
        int i0 = (int)(t0 - a.traj_tok[b]);
        int lo = s0, hi = s1;   // seg_start[lo] <= i0 (seg_start[s0] = 0)
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (a.seg_start[mid] <= i0) lo = mid; else hi = mid;
        }
        int32_t segv[INIT_TPT];
#pragma unroll
        for (int k = 0; k < INIT_TPT; ++k) {
            const int64_t t = t0 + k;
            if (t < a.total) {
                while (t >= a.traj_tok[b + 1]) {   // next non-empty trajectory
                    ++b;
                    s0 = a.traj_seg[b];
                    s1 = a.traj_seg[b + 1];
                    lo = s0;
                }
                const int i = (int)(t - a.traj_tok[b]);
                while (lo + 1 < s1 && a.seg_start[lo + 1] <= i) ++lo;
                segv[k] = lo - s0;
            }
        }
        if (t0 + INIT_TPT <= a.total) {
            const int4 never = make_int4(INT32_MAX, INT32_MAX, INT32_MAX, INT32_MAX);
#pragma unroll
            for (int q = 0; q < INIT_TPT / 4; ++q) {
                reinterpret_cast<int4*>(a.omega + t0)[q] = never;
                reinterpret_cast<int4*>(a.seg + t0)[q] = make_int4(segv[4 * q], segv[4 * q + 1], segv[4 * q + 2],
                                                                   segv[4 * q + 3]);
            }
        } else {
#pragma unroll
            for (int k = 0; k < INIT_TPT; ++k) {
                if (t0 + k < a.total) {
                    a.omega[t0 + k] = INT32_MAX;
                    a.seg[t0 + k] = segv[k];
                }
            }
        }
    }
}

// One block per evicted span: omega(j) = min over the junctions evicting j.
__global__ void k_scatter_spans(BuildArgs a) {
    for (int s = blockIdx.x; s < a.n_spans; s += gridDim.x) {
        int ga = a.spans[3 * s], gb = a.spans[3 * s + 1], J = a.spans[3 * s + 2];
        for (int t = ga + threadIdx.x; t < gb; t += blockDim.x)
            if (MW_DBG_IN(t, a.total, a.status, 101)) atomicMin(&a.omega[t], J);
    }
}

// One warp per global k-tile (a lane takes keys lane, lane + 32, lane + 64,
// lane + 96): min / max lifetime over its keys, visible pairs sum_j
// (min(omega_j, T) - j) (per tile; the scan sums them per trajectory), and the
// per-segment view bits, one 16-byte store per segment. No block-level
// synchronisation: the warps of a block are independent.
__global__ void __launch_bounds__(256) k_tile_stats(BuildArgs a) {
    const int64_t g = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (g >= a.n_tiles) return;   // uniform over the warp
    const int b = a.tile_traj[g];
    const int kt = (int)(g - a.traj_tile[b]);
    const int T = a.traj_tok[b + 1] - a.traj_tok[b];
    const int64_t tok0 = a.traj_tok[b];
    int om[4];
    int vmin[4], vmax[4];
    unsigned long long pr = 0ull;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int j = kt * MW_TILE + 32 * q + lane;
        const bool in = j < T;
        om[q] = in ? a.omega[tok0 + j] : 0;
        vmin[q] = in ? om[q] : INT32_MAX;
        vmax[q] = in ? om[q] : INT32_MIN;
        if (in) pr += (unsigned long long)(min(om[q], T) - j);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            vmin[q] = min(vmin[q], __shfl_xor_sync(0xffffffffu, vmin[q], o));
            vmax[q] = max(vmax[q], __shfl_xor_sync(0xffffffffu, vmax[q], o));
        }
        pr += __shfl_xor_sync(0xffffffffu, pr, o);
    }
    // view bits: key j is in segment s's view iff omega(j) > J_s and j < J_{s+1};
    // lane s holds J_s of the first 32 segments (later ones come from L2)
    const int s0 = a.traj_seg[b], nseg = a.traj_seg[b + 1] - s0;
    const int nt = a.traj_tile[b + 1] - a.traj_tile[b];
    const int my_start = lane < nseg ? a.seg_start[s0 + lane] : T;
    uint4* km = reinterpret_cast<uint4*>(a.keymask) + a.traj_km[b] + kt;
    for (int s = 0; s < nseg; ++s) {
        const int Js = s < 32 ? __shfl_sync(0xffffffffu, my_start, s) : a.seg_start[s0 + s];
        const int Jn = s + 1 < 32 ? __shfl_sync(0xffffffffu, my_start, s + 1)
                                  : (s + 1 < nseg ? a.seg_start[s0 + s + 1] : T);
        uint32_t wd[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int j = kt * MW_TILE + 32 * q + lane;
            wd[q] = __ballot_sync(0xffffffffu, j < T && om[q] > Js && j < Jn);
        }
        if (lane == 0 && MW_DBG_IN(a.traj_km[b] + kt + (int64_t)s * nt, a.n_keymask, a.status, 105))
            km[(int64_t)s * nt] = make_uint4(wd[0], wd[1], wd[2], wd[3]);
    }
    if (lane == 0) {
        *reinterpret_cast<int4*>(a.tstat + 4 * g) =
            make_int4(min(min(vmin[0], vmin[1]), min(vmin[2], vmin[3])),
                      max(max(vmax[0], vmax[1]), max(vmax[2], vmax[3])),
                      max(vmax[0], vmax[1]),    // keys 0..63 (INT32_MIN when none in range)
                      max(vmax[2], vmax[3]));   // keys 64..127
        a.tpairs[g] = pr;
    }
}

// Class of tile (qt, kt) from its k-tile's lifetime statistics st = (min, max,
// max over keys 0..63, max over keys 64..127). Off the diagonal every key
// precedes every row, so row i sees key j iff i < omega(j): a key half is seen
// by some row iff its largest lifetime exceeds the q-tile's first row.
__device__ __forceinline__ int tile_class(int qt, int kt, int T, int4 st) {
    int q0 = qt * MW_TILE, q1 = min(q0 + MW_TILE, T);
    if (kt == qt) return (q1 - q0 == 1) ? MW_TILE_FULL : MW_TILE_PARTIAL;
    if (st.x >= q1) return MW_TILE_FULL;
    if (st.y <= q0) return MW_TILE_EMPTY;
    return MW_TILE_PARTIAL | (st.z <= q0 ? MW_TILE_DEAD_LO : 0) | (st.w <= q0 ? MW_TILE_DEAD_HI : 0);
}
// statistics of global k-tile g (16-byte aligned: the workspace region is)
__device__ __forceinline__ int4 tile_stat(const int32_t* tstat, int64_t g) {
    return *reinterpret_cast<const int4*>(tstat + 4 * g);
}

// One warp per q-tile, 32 consecutive q-tiles of one trajectory per block:
// classes of (qt, 0..qt) and the fwd list length. The trajectory's k-tile
// statistics pass through shared memory in chunks, so each is read from L2
// once per block instead of once per q-tile.
constexpr int CLS_CHUNK = 2048;
__global__ void __launch_bounds__(1024) k_classify(BuildArgs a) {
    __shared__ int4 sst[CLS_CHUNK];
    const int b = blockIdx.x;
    const int tb = a.traj_tile[b], nt = a.traj_tile[b + 1] - tb;
    const int q_first = blockIdx.y * 32;
    if (q_first >= nt) return;   // uniform over the block
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int qt = q_first + warp;
    const bool live = qt < nt;
    const int T = a.traj_tok[b + 1] - a.traj_tok[b];
    const int q_last = min(nt, q_first + 32) - 1;
    uint8_t* row = a.cls + a.traj_tri[b] + (live ? (int64_t)qt * (qt + 1) / 2 : 0);
    int cnt = 0;
    for (int kc = 0; kc <= q_last; kc += CLS_CHUNK) {
        const int kn = min(CLS_CHUNK, q_last + 1 - kc);
        __syncthreads();   // the previous chunk is consumed
        for (int k = threadIdx.x; k < kn; k += blockDim.x) sst[k] = tile_stat(a.tstat, tb + kc + k);
        __syncthreads();
        if (live) {
            const int kend = min(qt + 1, kc + kn);
            for (int kt = kc + lane; kt < kend; kt += 32) {
                const int c = tile_class(qt, kt, T, sst[kt - kc]);
                row[kt] = (uint8_t)c;
                cnt += c != MW_TILE_EMPTY;
            }
        }
    }
    cnt = warp_sum_i(cnt);
    if (live && lane == 0) a.fwd_cnt[tb + qt] = cnt;
}

// One thread per global k-tile: bwd list length, the non-EMPTY tiles of its
// column of the class triangle. The diagonal tile is never EMPTY; below it
// (qt > kt) a tile is EMPTY exactly when the k-tile's largest lifetime is at
// most the q-tile's first row (tile_class), so the column's non-EMPTY tiles
// are the q-tiles kt .. ceil(min(max lifetime, T) / 128) - 1.
__global__ void k_bwd_count(BuildArgs a) {
    const int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (g >= a.n_tiles) return;
    const int b = a.tile_traj[g];
    const int tb = a.traj_tile[b], nt = a.traj_tile[b + 1] - tb;
    const int kt = (int)(g - tb);
    const int T = a.traj_tok[b + 1] - a.traj_tok[b];
    const int lim = min(a.tstat[4 * g + 1], T);
    a.bwd_cnt[g] = 1 + max(0, min(nt, (lim + MW_TILE - 1) / MW_TILE) - kt - 1);
}

// List pointers: exclusive scans of both count arrays, in three launches of
// SCAN_BLOCK-tile blocks (a single block's serial passes were the builder's
// slowest step at batch sizes).
// Phase 1, one block per SCAN_BLOCK tiles: the block's count sums, and the
// visible pairs added into each tile's trajectory (one atomic per warp whose
// 32 tiles share a trajectory, else one per tile).
__global__ void __launch_bounds__(SCAN_BLOCK) k_scan_sums(BuildArgs a) {
    __shared__ int ws[2][SCAN_BLOCK / 32];
    const int64_t i = (int64_t)blockIdx.x * SCAN_BLOCK + threadIdx.x;
    const bool in = i < a.n_tiles;
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int f = warp_sum_i(in ? a.fwd_cnt[i] : 0);
    const int k = warp_sum_i(in ? a.bwd_cnt[i] : 0);
    if (lane == 0) { ws[0][w] = f; ws[1][w] = k; }
    const int bt = in ? a.tile_traj[i] : -1;
    const unsigned long long pr = in ? a.tpairs[i] : 0ull;
    const int b0 = __shfl_sync(0xffffffffu, bt, 0);
    if (__all_sync(0xffffffffu, bt == b0)) {
        const unsigned long long sum = warp_sum_u64(pr);
        if (lane == 0 && b0 >= 0) atomicAdd(&a.pairs[b0], sum);
    } else if (in) {
        atomicAdd(&a.pairs[bt], pr);
    }
    __syncthreads();
    if (threadIdx.x < 2) {
        int t = 0;
        for (int q = 0; q < SCAN_BLOCK / 32; ++q) t += ws[threadIdx.x][q];
        a.bsum[threadIdx.x * gridDim.x + blockIdx.x] = t;
    }
}

// Phase 2, one block: exclusive offsets of the block sums (in place), both
// lists' totals, and the job total of the visible pairs (phase 1 completed
// every trajectory's sum).
__global__ void __launch_bounds__(1024) k_scan_offsets(BuildArgs a, int nb) {
    __shared__ int wsum[2][32];
    __shared__ int carry[2];
    __shared__ unsigned long long psum[32];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
    if (threadIdx.x < 2) carry[threadIdx.x] = 0;
    __syncthreads();
    for (int c0 = 0; c0 < nb; c0 += blockDim.x) {
        const int i = c0 + threadIdx.x;
        int v[2], inc[2];
        for (int q = 0; q < 2; ++q) {
            v[q] = i < nb ? a.bsum[q * nb + i] : 0;
            int x = v[q];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, x, o);
                if (lane >= o) x += y;
            }
            inc[q] = x;
            if (lane == 31) wsum[q][w] = x;
        }
        __syncthreads();
        if (w == 0) {
            for (int q = 0; q < 2; ++q) {
                int x = lane < nw ? wsum[q][lane] : 0;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int y = __shfl_up_sync(0xffffffffu, x, o);
                    if (lane >= o) x += y;
                }
                if (lane < nw) wsum[q][lane] = x;   // inclusive over warps
            }
        }
        __syncthreads();
        for (int q = 0; q < 2; ++q)
            if (i < nb) a.bsum[q * nb + i] = carry[q] + (w > 0 ? wsum[q][w - 1] : 0) + inc[q] - v[q];
        __syncthreads();
        if (threadIdx.x == 0) {
            carry[0] += wsum[0][nw - 1];
            carry[1] += wsum[1][nw - 1];
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        a.fwd_ptr[a.n_tiles] = carry[0];
        a.bwd_ptr[a.n_tiles] = carry[1];
    }
    unsigned long long tp = 0;
    for (int b = threadIdx.x; b < a.n_traj; b += blockDim.x) tp += a.pairs[b];
    tp = warp_sum_u64(tp);
    if (lane == 0) psum[w] = tp;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned long long t = 0;
        for (int q = 0; q < nw; ++q) t += psum[q];
        a.pairs[a.n_traj] = t;
    }
}

// Phase 3, one block per SCAN_BLOCK tiles: the block's exclusive scan plus its
// offset.
__global__ void __launch_bounds__(SCAN_BLOCK) k_scan_ptrs(BuildArgs a) {
    __shared__ int wsum[2][SCAN_BLOCK / 32];
    const int64_t i = (int64_t)blockIdx.x * SCAN_BLOCK + threadIdx.x;
    const bool in = i < a.n_tiles;
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    int v[2], inc[2];
    v[0] = in ? a.fwd_cnt[i] : 0;
    v[1] = in ? a.bwd_cnt[i] : 0;
    for (int q = 0; q < 2; ++q) {
        int x = v[q];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        inc[q] = x;
        if (lane == 31) wsum[q][w] = x;
    }
    __syncthreads();
    if (w == 0) {
        for (int q = 0; q < 2; ++q) {
            int x = wsum[q][lane];   // SCAN_BLOCK / 32 = 32 warps
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, x, o);
                if (lane >= o) x += y;
            }
            wsum[q][lane] = x;
        }
    }
    __syncthreads();
    if (in) {
        a.fwd_ptr[i] = a.bsum[blockIdx.x] + (w > 0 ? wsum[0][w - 1] : 0) + inc[0] - v[0];
        a.bwd_ptr[i] = a.bsum[gridDim.x + blockIdx.x] + (w > 0 ? wsum[1][w - 1] : 0) + inc[1] - v[1];
    }
}

// One warp per global q-tile (fwd) or k-tile (bwd): ordered compaction. The
// fwd list reads its row of the class triangle; the bwd list recomputes its
// column's classes from the k-tile's statistics (the values k_classify
// stored), which avoids reading the triangle by columns.
__global__ void k_fill(BuildArgs a) {
    int64_t g = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    int lane = threadIdx.x & 31;
    if (g >= a.n_tiles) return;
    int b = a.tile_traj[g];
    int tb = a.traj_tile[b], nt = a.traj_tile[b + 1] - tb;
    int t = (int)(g - tb);
    const int T = a.traj_tok[b + 1] - a.traj_tok[b];
    const uint8_t* tri = a.cls + a.traj_tri[b];
    uint32_t lt = (1u << lane) - 1u;
    int base = a.fwd_ptr[g];
#pragma unroll 4
    for (int k0 = 0; k0 <= t; k0 += 32) {
        int kt = k0 + lane;
        int c = kt <= t ? tri[(int64_t)t * (t + 1) / 2 + kt] : MW_TILE_EMPTY;
        uint32_t m = __ballot_sync(0xffffffffu, c != MW_TILE_EMPTY);
        if (c != MW_TILE_EMPTY && MW_DBG_IN(base + __popc(m & lt), a.n_tri, a.status, 102))
            a.fwd_idx[base + __popc(m & lt)] = (kt << 4) | c;
        base += __popc(m);
    }
    // the column's non-EMPTY tiles are exactly the q-tiles t .. qend - 1
    // (k_bwd_count), so the bwd list is written without compaction
    base = a.bwd_ptr[g];
    const int4 st = tile_stat(a.tstat, g);
    const int qend = max(t + 1, min(nt, (min(st.y, T) + MW_TILE - 1) / MW_TILE));
    for (int qt = t + lane; qt < qend; qt += 32)
        if (MW_DBG_IN(base + qt - t, a.n_tri, a.status, 103)) a.bwd_idx[base + qt - t] = (qt << 4) | tile_class(qt, t, T, st);
}

// Compact views. An exclusive prefix popcount of the segment's view bits,
// tile by tile, gives every member key its rank in view_s (cpos; -1 for
// non-members) and the inverse map (csrc: the key at each rank); the total is
// |view_s|, and csrc is -1 from there to the end of the last 128-entry tile.
// For a monotone record view_s is in physical order, so the rank is the key's
// index in the segment's compact sequence (§4.1). One block per (global
// segment, chunk of 256 k-tiles): the chunk's first rank is the popcount of the
// segment's earlier tiles; the block holding the segment's last tile writes
// |view_s| and the tail.
constexpr int CMAP_TILES = 256;
__global__ void __launch_bounds__(256) k_compact_map(BuildArgs a) {
    __shared__ int tp[256];
    __shared__ int wsum[8];
    const int sg = blockIdx.x;
    int lo = 0, hi = a.n_traj;   // largest b with traj_seg[b] <= sg
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (a.traj_seg[mid] <= sg) lo = mid; else hi = mid;
    }
    const int b = lo;
    const int s = sg - a.traj_seg[b];
    const int nt = a.traj_tile[b + 1] - a.traj_tile[b];
    const int c0 = blockIdx.y * CMAP_TILES;
    if (c0 >= nt) {   // uniform over the block; an empty trajectory's segment has an empty view
        if (blockIdx.y == 0 && threadIdx.x == 0) a.seg_len[sg] = 0;
        return;
    }
    const int64_t ent0 = a.traj_km[b] + (int64_t)s * nt;   // keymask entry of (s, kt = 0)
    const uint32_t* km = a.keymask + ent0 * 4;
    int32_t* pos = a.cpos + ent0 * MW_TILE;
    int32_t* src = a.csrc + ent0 * MW_TILE;
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    auto tile_cnt = [&](int kt) -> int {
        return __popc(km[4 * kt]) + __popc(km[4 * kt + 1]) + __popc(km[4 * kt + 2]) + __popc(km[4 * kt + 3]);
    };
    // first rank of the chunk: members of the segment's tiles 0 .. c0 - 1
    int before_chunk = 0;
    for (int kt = t; kt < c0; kt += 256) before_chunk += tile_cnt(kt);
    before_chunk = warp_sum_i(before_chunk);
    if (lane == 0) wsum[w] = before_chunk;
    __syncthreads();
    int base = 0;
#pragma unroll
    for (int q = 0; q < 8; ++q) base += wsum[q];
    __syncthreads();
    const int kt = c0 + t;
    // this thread's tile: its four view-bit words and their exclusive prefix
    // counts, kept in shared memory for the element loop below
    __shared__ uint4 words[CMAP_TILES];
    __shared__ uint4 wpre[CMAP_TILES];
    const uint4 wv = kt < nt ? *reinterpret_cast<const uint4*>(km + 4 * kt) : make_uint4(0u, 0u, 0u, 0u);
    const int c0w = __popc(wv.x), c1w = __popc(wv.y), c2w = __popc(wv.z), c3w = __popc(wv.w);
    words[t] = wv;
    wpre[t] = make_uint4(0u, (uint32_t)c0w, (uint32_t)(c0w + c1w), (uint32_t)(c0w + c1w + c2w));
    const int cnt = c0w + c1w + c2w + c3w;
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) wsum[w] = incl;
    __syncthreads();
    int before = base;
    for (int q = 0; q < w; ++q) before += wsum[q];
    tp[t] = before + incl - cnt;
    __syncthreads();
    const int ntc = min(CMAP_TILES, nt - c0);
    for (int k = t; k < ntc * MW_TILE; k += 256) {
        const int tl = k >> 7, jj = k & 127, wd = jj >> 5, bit = jj & 31;
        const uint4 w4 = words[tl], p4 = wpre[tl];
        const uint32_t word = wd == 0 ? w4.x : wd == 1 ? w4.y : wd == 2 ? w4.z : w4.w;
        const uint32_t pre = wd == 0 ? p4.x : wd == 1 ? p4.y : wd == 2 ? p4.z : p4.w;
        int32_t r = -1;
        if ((word >> bit) & 1u) {
            r = tp[tl] + (int)pre + __popc(word & ((1u << bit) - 1u));
            if (MW_DBG_IN(r, (int64_t)nt * MW_TILE, a.status, 104)) src[r] = (c0 + tl) * MW_TILE + jj;
        }
        pos[(int64_t)(c0 + tl) * MW_TILE + jj] = r;
    }
    if (c0 + CMAP_TILES >= nt) {   // the block holding the segment's last tile
        int total = 0;
#pragma unroll
        for (int q = 0; q < 8; ++q) total += wsum[q];
        const int len = base + total;
        if (t == 0) a.seg_len[sg] = len;
        const int end = (len + MW_TILE - 1) / MW_TILE * MW_TILE;
        for (int r = len + t; r < end; r += 256) src[r] = -1;
    }
}

// Dense visibility of one trajectory, bit-packed (the 4D mask of Eq. 7 for
// small T, for comparing with a dense-mask implementation): row i sees key j
// iff j is in the view of i's segment at or before i's own place in it. For an
// edits record the view is in physical order, so that is the segment's
// view-bit word cut at j <= i; for offload / retrieve views it is 0 <=
// cpos_s(j) <= cpos_s(i), from the 32 keys' ranks (eight 16-byte loads).
// DM_ROWS rows per block (their segment ids loaded up front, independently),
// a thread per 32-key word.
constexpr int DM_ROWS = 8;
__global__ void __launch_bounds__(256) k_dense_mask(VisView v, int b, int T, int words, int by_rank,
                                                    uint32_t* __restrict__ mask) {
    const int i0 = blockIdx.x * DM_ROWS;
    const int64_t tok0 = v.traj_tok[b];
    const int nt = v.traj_tile[b + 1] - v.traj_tile[b];
    const int64_t km0 = v.traj_km[b];
    int sr[DM_ROWS];
#pragma unroll
    for (int r = 0; r < DM_ROWS; ++r) sr[r] = i0 + r < T ? v.seg[tok0 + i0 + r] : 0;
#pragma unroll
    for (int r = 0; r < DM_ROWS; ++r) {
        const int i = i0 + r;
        if (i >= T) break;   // uniform over the block
        const int64_t ent0 = km0 + (int64_t)sr[r] * nt;        // (segment, k-tile 0) entry
        const int32_t* cp = v.cpos + ent0 * MW_TILE;           // key j's rank at cp[j]
        const uint32_t* km = v.keymask + ent0 * 4;             // key j's view bit: word j / 32
        const int ci = by_rank ? cp[i] : 0;
        for (int w = threadIdx.x; w < words; w += blockDim.x) {
            const int j0 = 32 * w;
            uint32_t bits = 0u;
            if (!by_rank) {
                if (j0 <= i) {
                    const int hi = i - j0;   // keys j0 .. j0 + hi are at or before i
                    bits = km[w] & (hi >= 31 ? 0xffffffffu : ((2u << hi) - 1u));
                }
            } else if (j0 + 32 <= T) {
                const int4* c4 = reinterpret_cast<const int4*>(cp + j0);
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const int4 c = c4[q];
                    bits |= (uint32_t)(c.x >= 0 && c.x <= ci) << (4 * q) | (uint32_t)(c.y >= 0 && c.y <= ci) << (4 * q + 1) |
                            (uint32_t)(c.z >= 0 && c.z <= ci) << (4 * q + 2) |
                            (uint32_t)(c.w >= 0 && c.w <= ci) << (4 * q + 3);
                }
            } else {
                for (int k = 0; j0 + k < T; ++k) {
                    const int c = cp[j0 + k];
                    bits |= (uint32_t)(c >= 0 && c <= ci) << k;
                }
            }
            mask[(int64_t)i * words + w] = bits;
        }
    }
}

// EVENTS records: one block per trajectory replays its events segment by
// segment into the compact views. view_s = (view_{s-1} without the event's
// out-spans, order kept) + the in-spans in the given order + the segment's
// rows. A key is dropped when its flag holds the current segment (set from
// the out-spans just before); flags never need clearing. Also the per-row
// compact index sum gives the visible pairs: a row at index c sees c + 1 keys.
struct EventArgs {
    int n_traj;
    const int32_t* traj_tok;
    const int32_t* traj_tile;
    const int32_t* traj_seg;
    const int64_t* traj_km;
    const int32_t* seg_start;
    const int32_t* spans;    // [n_spans][2] global positions
    const int32_t* jtab;     // [n_junc][4] out begin, out end, in begin, in end (into spans)
    int32_t* flag;           // [total] segment that last evicted the key, -1 never
    int32_t* seg_len;
    int32_t* cpos;
    int32_t* csrc;
    unsigned long long* pairs;
    int32_t* status;         // device status words (debug index checks)
};

__global__ void __launch_bounds__(1024) k_event_views(EventArgs a) {
    __shared__ int wsum[32];
    const int b = blockIdx.x;
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    const int64_t tok0 = a.traj_tok[b];
    const int T = a.traj_tok[b + 1] - (int)tok0;
    const int nt = a.traj_tile[b + 1] - a.traj_tile[b];
    const int g0 = a.traj_seg[b], S = a.traj_seg[b + 1] - g0;
    if (T == 0) {   // an empty trajectory has one empty segment
        if (t == 0) {
            for (int s = 0; s < S; ++s) a.seg_len[g0 + s] = 0;
            a.pairs[b] = 0;
        }
        return;
    }
    int32_t* flag = a.flag + tok0;
    unsigned long long pairs = 0;
    for (int s = 0; s < S; ++s) {
        const int64_t base = (a.traj_km[b] + (int64_t)s * nt) * MW_TILE;
        const int64_t prev = base - (int64_t)nt * MW_TILE;
        const int lo = a.seg_start[g0 + s], hi = s + 1 < S ? a.seg_start[g0 + s + 1] : T;
        for (int x = t; x < nt * MW_TILE; x += blockDim.x) a.cpos[base + x] = -1;
        int n = 0;
        if (s >= 1) {
            const int32_t* jt = a.jtab + 4 * (int64_t)(g0 - b + s - 1);   // this trajectory's event s - 1
            for (int q = jt[0]; q < jt[1]; ++q)
                for (int j = a.spans[2 * q] + t; j < a.spans[2 * q + 1]; j += blockDim.x)
                    if (MW_DBG_IN(j - tok0, T, a.status, 111)) flag[j - tok0] = s;
            __syncthreads();
            // ordered compaction of view_{s-1} without the keys flagged s
            const int Lp = a.seg_len[g0 + s - 1];
            for (int c0 = 0; c0 < Lp; c0 += blockDim.x) {
                const int c = c0 + t;
                const int key = c < Lp ? a.csrc[prev + c] : -1;
                const int keep = c < Lp && MW_DBG_IN(key, T, a.status, 112) && flag[key] != s;
                const unsigned bal = __ballot_sync(0xffffffffu, keep);
                if (lane == 0) wsum[w] = __popc(bal);
                __syncthreads();
                int before = 0, total = 0;
                for (int q = 0; q < 32; ++q) {
                    before += q < w ? wsum[q] : 0;
                    total += wsum[q];
                }
                if (keep && MW_DBG_IN(n + before + __popc(bal & ((1u << lane) - 1u)), (int64_t)nt * MW_TILE,
                                      a.status, 113))
                    a.csrc[base + n + before + __popc(bal & ((1u << lane) - 1u))] = key;
                n += total;
                __syncthreads();
            }
            for (int q = jt[2]; q < jt[3]; ++q) {
                const int ga = a.spans[2 * q], gb = a.spans[2 * q + 1];
                for (int j = ga + t; j < gb; j += blockDim.x)
                    if (MW_DBG_IN(n + (j - ga), (int64_t)nt * MW_TILE, a.status, 114))
                        a.csrc[base + n + (j - ga)] = (int)(j - tok0);
                n += gb - ga;
            }
        }
        for (int r = lo + t; r < hi; r += blockDim.x)
            if (MW_DBG_IN(n + (r - lo), (int64_t)nt * MW_TILE, a.status, 115)) a.csrc[base + n + (r - lo)] = r;
        const int R = hi - lo;
        pairs += (unsigned long long)R * (unsigned long long)n + (unsigned long long)R * (R + 1) / 2;
        n += R;
        const int end = (n + MW_TILE - 1) / MW_TILE * MW_TILE;
        for (int c = n + t; c < end; c += blockDim.x) a.csrc[base + c] = -1;
        if (t == 0) a.seg_len[g0 + s] = n;
        __syncthreads();
        for (int c = t; c < n; c += blockDim.x)
            if (MW_DBG_IN(a.csrc[base + c], T, a.status, 116)) a.cpos[base + a.csrc[base + c]] = c;
        __syncthreads();
    }
    if (t == 0) {
        a.pairs[b] = pairs;
        atomicAdd(&a.pairs[a.n_traj], pairs);
    }
}

// View bits from the compact ranks: one warp per (segment, k-tile) entry.
__global__ void k_event_keymask(int64_t n_keymask, const int32_t* __restrict__ cpos, uint32_t* __restrict__ km) {
    const int64_t e = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (e >= n_keymask) return;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        const unsigned bal = __ballot_sync(0xffffffffu, cpos[e * MW_TILE + 32 * w + lane] >= 0);
        if (lane == 0) km[e * 4 + w] = bal;
    }
}

// Copy of up to four staged host arrays into device memory: part blockIdx.y,
// 16-byte vectors (both ends are 16-byte aligned), the ragged tail by bytes.
struct UploadArgs {
    const char* src[4];
    char* dst[4];
    long long bytes[4];
};
__global__ void __launch_bounds__(256) k_upload(UploadArgs u) {
    const int p = blockIdx.y;
    const char* src = u.src[p];
    char* dst = u.dst[p];
    const long long n = u.bytes[p], n16 = n >> 4;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n16; i += (long long)gridDim.x * blockDim.x)
        reinterpret_cast<uint4*>(dst)[i] = reinterpret_cast<const uint4*>(src)[i];
    if (blockIdx.x == 0 && threadIdx.x < (n & 15)) dst[16 * n16 + threadIdx.x] = src[16 * n16 + threadIdx.x];
}

}  // namespace

// ---------------------------------------------------------------------------
// Upload of the host-packed build inputs (the metadata image, the span table,
// the events table). A copy from pageable memory goes through the runtime's
// staging memory and a copy engine, where it shares the engines with the
// caller's own uploads (a training loop prefetching its next batch on another
// stream). The builders instead pack into page-locked, device-mapped host
// buffers, and k_upload on the build's stream reads them over the host link
// into place: no copy engine, and the call returns without a host-side
// staging copy. Two buffers per device alternate; before a buffer is
// rewritten, the event recorded after its last upload is waited on, so the
// host runs at most two builds ahead of the GPU. The buffers live as long as
// the process. A build that may not allocate (mw_build_visibility_noalloc),
// or a failed page-locked allocation, copies from pageable memory instead.
struct UploadPart {
    const void* src;
    void* dst;
    size_t bytes;
};

namespace {
struct StageSlot {
    char* host = nullptr;
    size_t cap = 0;
    cudaEvent_t done = nullptr;
    bool pending = false;
};
struct DevStage {
    std::mutex mu;
    StageSlot slot[2];
    int next = 0;
};
constexpr int kStageDevices = 64;
DevStage g_stage[kStageDevices];

mw_status upload_pageable(const UploadPart* parts, int n, cudaStream_t s) {
    for (int i = 0; i < n; ++i)
        if (parts[i].bytes) {
            mw_status st = cuda_status(
                cudaMemcpyAsync(parts[i].dst, parts[i].src, parts[i].bytes, cudaMemcpyHostToDevice, s));
            if (st != MW_OK) return st;
        }
    return MW_OK;
}
}  // namespace

static mw_status upload_parts(const UploadPart* parts, int n, cudaStream_t s, bool staged) {
    size_t total = 0;
    for (int i = 0; i < n; ++i) total += (parts[i].bytes + 15) & ~size_t(15);
    int dev = 0;
    if (!staged || total == 0 || n > 4 || cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kStageDevices)
        return upload_pageable(parts, n, s);
    DevStage& d = g_stage[dev];
    std::lock_guard<std::mutex> lock(d.mu);
    StageSlot& slot = d.slot[d.next];
    d.next ^= 1;
    mw_status st = MW_OK;
    if (slot.pending && (st = cuda_status(cudaEventSynchronize(slot.done))) != MW_OK) return st;
    slot.pending = false;
    if (slot.cap < total) {
        if (slot.host) cudaFreeHost(slot.host);
        slot.host = nullptr;
        slot.cap = 0;
        const size_t cap = std::max<size_t>(total + total / 4, 1 << 16);
        void* h = nullptr;
        if (cudaHostAlloc(&h, cap, cudaHostAllocMapped | cudaHostAllocPortable) != cudaSuccess) {
            cudaGetLastError();   // clear the failed allocation; copy from pageable memory instead
            return upload_pageable(parts, n, s);
        }
        slot.host = (char*)h;
        slot.cap = cap;
    }
    if (!slot.done && (st = cuda_status(cudaEventCreateWithFlags(&slot.done, cudaEventDisableTiming))) != MW_OK)
        return st;
    void* dbase = nullptr;
    if ((st = cuda_status(cudaHostGetDevicePointer(&dbase, slot.host, 0))) != MW_OK) return st;
    UploadArgs u = {};
    long long most = 0;
    size_t off = 0;
    for (int i = 0; i < n; ++i) {
        if (parts[i].bytes) memcpy(slot.host + off, parts[i].src, parts[i].bytes);
        u.src[i] = (const char*)dbase + off;
        u.dst[i] = (char*)parts[i].dst;
        u.bytes[i] = (long long)parts[i].bytes;
        most = std::max(most, u.bytes[i]);
        off += (parts[i].bytes + 15) & ~size_t(15);
    }
    const unsigned gx = (unsigned)std::min<long long>(std::max<long long>(1, ceil_div(most >> 4, 256)), 152);
    count_launches(1);
    k_upload<<<dim3(gx, (unsigned)n), 256, 0, s>>>(u);
    if ((st = launch_status()) != MW_OK) return st;
    if ((st = cuda_status(cudaEventRecord(slot.done, s))) != MW_OK) return st;
    slot.pending = true;
    return MW_OK;
}

// Host image of the per-trajectory tables (token, tile, segment, triangle and
// keymask offsets, segment starts, tile owners): the bytes of the metadata
// region [off_traj_tok, off_cls) of `vis`, uploaded as one part.
static void pack_meta(const mw_vis_layout* L, const int32_t* cu, int n_junc, const int32_t* J, const int32_t* jt,
                      std::vector<char>& img) {
    const int n_traj = L->n_traj;
    // host-side packing of the small per-trajectory tables
    const int64_t n_tiles = L->n_tiles;
    std::vector<int32_t> traj_tile(n_traj + 1), traj_seg(n_traj + 1), seg_start(L->n_segs),
        tile_traj(n_tiles);
    std::vector<int64_t> traj_tri(n_traj + 1), traj_km(n_traj + 1);
    {
        int k = 0;
        int64_t tiles = 0, tri = 0, km = 0;
        int segs = 0;
        for (int b = 0; b < n_traj; ++b) {
            int64_t nt = ceil_div(cu[b + 1] - cu[b], MW_TILE);
            traj_tile[b] = (int32_t)tiles;
            traj_tri[b] = tri;
            traj_km[b] = km;
            traj_seg[b] = segs;
            seg_start[segs++] = 0;
            int Kb = 0;
            while (k < n_junc && jt[k] == b) { seg_start[segs++] = J[k]; ++k; ++Kb; }
            for (int64_t t = 0; t < nt; ++t) tile_traj[tiles + t] = b;
            tiles += nt;
            tri += nt * (nt + 1) / 2;
            km += (1 + Kb) * nt;
        }
        traj_tile[n_traj] = (int32_t)tiles;
        traj_tri[n_traj] = tri;
        traj_km[n_traj] = km;
        traj_seg[n_traj] = segs;
    }
    // one contiguous host image of the metadata region [off_traj_tok, off_cls)
    const int64_t meta0 = L->off_traj_tok, meta1 = L->off_cls;
    img.assign(meta1 - meta0, 0);
    auto put = [&](int64_t off, const void* src, size_t bytes) {
        if (bytes) memcpy(img.data() + (off - meta0), src, bytes);
    };
    put(L->off_traj_tok, cu, 4 * (size_t)(n_traj + 1));
    put(L->off_traj_tile, traj_tile.data(), 4 * traj_tile.size());
    put(L->off_traj_seg, traj_seg.data(), 4 * traj_seg.size());
    put(L->off_traj_tri, traj_tri.data(), 8 * traj_tri.size());
    put(L->off_traj_km, traj_km.data(), 8 * traj_km.size());
    put(L->off_seg_start, seg_start.data(), 4 * seg_start.size());
    put(L->off_tile_traj, tile_traj.data(), 4 * tile_traj.size());
}

namespace mw {
// mw_build_visibility; `staged` uploads the packed record through the pinned
// staging buffers (false: from pageable memory, no allocation).
mw_status build_visibility(const mw_vis_layout* L, const int32_t* cu, int n_junc, const int32_t* J,
                           const int32_t* jt, const int32_t* span_off, const int32_t* spans, void* ws, void* vis,
                           void* stream_, bool staged) {
    if (!L) return MW_EINVAL;
    if (L->kind != MW_VIEWS_EDITS || n_junc != L->n_junc) return MW_EINVAL;
    mw_status st = check_shape(L->n_traj, cu, n_junc, jt, L->n_spans);
    if (st != MW_OK) return st;
    const int n_traj = L->n_traj;
    if (n_traj > 0 && cu[n_traj] != L->total_tokens) return MW_EINVAL;
    if (n_junc > 0 && (!J || !span_off)) return MW_EINVAL;
    if (L->n_spans > 0 && !spans) return MW_EINVAL;
    if (L->vis_bytes > 0 && !vis) return MW_EINVAL;
    if (L->ws_bytes > 0 && !ws) return MW_EINVAL;
    if (((uintptr_t)vis | (uintptr_t)ws) % 256) return MW_EINVAL;   // arrays sit at 256-byte offsets
    if (n_junc > 0 && (span_off[0] != 0 || span_off[n_junc] != L->n_spans)) return MW_EEDITS;
    // validate junctions and spans (App. B Def. "trajectory tree")
    for (int k = 0; k < n_junc; ++k) {
        int b = jt[k];
        int T = cu[b + 1] - cu[b];
        if (J[k] < 1 || J[k] > T - 1) return MW_EEDITS;
        if (k > 0 && jt[k - 1] == b && J[k] <= J[k - 1]) return MW_EEDITS;
        if (span_off[k + 1] < span_off[k]) return MW_EEDITS;
        for (int s = span_off[k]; s < span_off[k + 1]; ++s) {
            int a0 = spans[2 * s], b0 = spans[2 * s + 1];
            if (!(0 <= a0 && a0 < b0 && b0 <= J[k])) return MW_EEDITS;
        }
    }
    cudaStream_t stream = (cudaStream_t)stream_;
    if (L->vis_bytes == 0) return MW_OK;

    const int64_t n_tiles = L->n_tiles;
    std::vector<char> img;
    pack_meta(L, cu, n_junc, J, jt, img);
    std::vector<int32_t> span3(3 * (size_t)L->n_spans);
    for (int k = 0; k < n_junc; ++k)
        for (int s = span_off[k]; s < span_off[k + 1]; ++s) {
            span3[3 * s] = cu[jt[k]] + spans[2 * s];
            span3[3 * s + 1] = cu[jt[k]] + spans[2 * s + 1];
            span3[3 * s + 2] = J[k];
        }
    const UploadPart parts[2] = {{img.data(), at<char>(vis, L->off_traj_tok), img.size()},
                                 {span3.data(), at<char>(ws, L->ws_off_spans), span3.size() * 4}};
    if ((st = upload_parts(parts, 2, stream, staged)) != MW_OK) return st;
    if ((st = cuda_status(cudaMemsetAsync(at<char>(vis, L->off_pairs), 0, 8 * (n_traj + 1), stream))) != MW_OK)
        return st;
    if ((st = cuda_status(cudaMemsetAsync(at<char>(vis, L->off_status), 0, 32, stream))) != MW_OK)
        return st;

    BuildArgs a;
    a.n_traj = n_traj;
    a.total = L->total_tokens;
    a.n_tiles = n_tiles;
    a.n_spans = L->n_spans;
    a.omega = at<int32_t>(vis, L->off_omega);
    a.seg = at<int32_t>(vis, L->off_seg);
    a.traj_tok = at<int32_t>(vis, L->off_traj_tok);
    a.traj_tile = at<int32_t>(vis, L->off_traj_tile);
    a.traj_seg = at<int32_t>(vis, L->off_traj_seg);
    a.traj_tri = at<int64_t>(vis, L->off_traj_tri);
    a.traj_km = at<int64_t>(vis, L->off_traj_km);
    a.seg_start = at<int32_t>(vis, L->off_seg_start);
    a.tile_traj = at<int32_t>(vis, L->off_tile_traj);
    a.cls = at<uint8_t>(vis, L->off_cls);
    a.fwd_ptr = at<int32_t>(vis, L->off_fwd_ptr);
    a.fwd_idx = at<int32_t>(vis, L->off_fwd_idx);
    a.bwd_ptr = at<int32_t>(vis, L->off_bwd_ptr);
    a.bwd_idx = at<int32_t>(vis, L->off_bwd_idx);
    a.pairs = at<unsigned long long>(vis, L->off_pairs);
    a.keymask = at<uint32_t>(vis, L->off_keymask);
    a.seg_len = at<int32_t>(vis, L->off_seg_len);
    a.cpos = at<int32_t>(vis, L->off_cpos);
    a.csrc = at<int32_t>(vis, L->off_csrc);
    a.spans = at<int32_t>(ws, L->ws_off_spans);
    a.tstat = at<int32_t>(ws, L->ws_off_tstat);
    a.fwd_cnt = at<int32_t>(ws, L->ws_off_cnt);
    a.bwd_cnt = at<int32_t>(ws, L->ws_off_cnt) + n_tiles;
    a.tpairs = reinterpret_cast<unsigned long long*>(at<int32_t>(ws, L->ws_off_cnt) + 2 * n_tiles);
    a.bsum = at<int32_t>(ws, L->ws_off_cnt) + 4 * n_tiles;
    a.status = at<int32_t>(vis, L->off_status);
    a.n_tri = L->n_tri;
    a.n_keymask = L->n_keymask;

    count_launches((a.total > 0 ? 1 + (L->n_spans > 0) : 0) + (n_tiles > 0 ? 3 : 0) + 1 + 4 * (n_tiles > 0));
    if (a.total > 0) {
        int grid = (int)std::min<int64_t>(ceil_div(ceil_div(a.total, INIT_TPT), 256), 152 * 16);
        k_init_tokens<<<grid, 256, 0, stream>>>(a);
        if (L->n_spans > 0) k_scatter_spans<<<(int)std::min<int64_t>(L->n_spans, 152 * 8), 256, 0, stream>>>(a);
    }
    if (n_tiles > 0) {
        k_tile_stats<<<(unsigned)ceil_div(n_tiles * 32, 256), 256, 0, stream>>>(a);
        k_classify<<<dim3((unsigned)L->n_traj, (unsigned)ceil_div(L->max_tiles, 32)), 1024, 0, stream>>>(a);
        k_bwd_count<<<(unsigned)ceil_div(n_tiles, 256), 256, 0, stream>>>(a);
    }
    {
        const unsigned nb = (unsigned)ceil_div(n_tiles, (int64_t)SCAN_BLOCK);
        if (nb > 0) k_scan_sums<<<nb, SCAN_BLOCK, 0, stream>>>(a);
        k_scan_offsets<<<1, 1024, 0, stream>>>(a, (int)nb);
        if (nb > 0) k_scan_ptrs<<<nb, SCAN_BLOCK, 0, stream>>>(a);
    }
    if (n_tiles > 0) {
        k_fill<<<(unsigned)ceil_div(n_tiles * 32, 256), 256, 0, stream>>>(a);
        k_compact_map<<<dim3((unsigned)L->n_segs, (unsigned)ceil_div(L->max_tiles, CMAP_TILES)), 256, 0, stream>>>(a);
    }
    return launch_status();
}
}  // namespace mw

extern "C" mw_status mw_build_visibility(const mw_vis_layout* L, const int32_t* cu, int n_junc, const int32_t* J,
                                         const int32_t* jt, const int32_t* span_off, const int32_t* spans, void* ws,
                                         void* vis, void* stream) {
    return build_visibility(L, cu, n_junc, J, jt, span_off, spans, ws, vis, stream, true);
}

extern "C" mw_status mw_build_views_events(const mw_vis_layout* L, const int32_t* cu, int n_junc, const int32_t* J,
                                           const int32_t* jt, const int32_t* out_off, const int32_t* in_off,
                                           const int32_t* spans, void* ws, void* vis, void* stream_) {
    if (!L) return MW_EINVAL;
    if (L->kind != MW_VIEWS_EVENTS || n_junc != L->n_junc) return MW_EINVAL;
    mw_status st = check_shape(L->n_traj, cu, n_junc, jt, L->n_spans);
    if (st != MW_OK) return st;
    const int n_traj = L->n_traj;
    const int n_spans = L->n_spans;
    if (n_traj > 0 && cu[n_traj] != L->total_tokens) return MW_EINVAL;
    if (n_junc > 0 && (!J || !out_off || !in_off)) return MW_EINVAL;
    if (n_spans > 0 && !spans) return MW_EINVAL;
    if (L->vis_bytes > 0 && !vis) return MW_EINVAL;
    if (L->ws_bytes > 0 && !ws) return MW_EINVAL;
    if (((uintptr_t)vis | (uintptr_t)ws) % 256) return MW_EINVAL;   // arrays sit at 256-byte offsets
    // validate: junctions ascending inside [1, T-1], spans inside [0, J), and
    // every retrieved position out of the view when its event fires (replayed
    // per trajectory on the host, one state byte per position)
    std::vector<int32_t> jtab(4 * (size_t)n_junc), sp2(2 * (size_t)n_spans);
    {
        std::vector<uint8_t> out;
        int cur = -1;
        for (int k = 0; k < n_junc; ++k) {
            const int b = jt[k];
            const int T = cu[b + 1] - cu[b];
            if (b != cur) {
                out.assign((size_t)T, 0);
                cur = b;
            } else if (J[k] <= J[k - 1]) {
                return MW_EEDITS;
            }
            if (J[k] < 1 || J[k] > T - 1) return MW_EEDITS;
            const int r[4] = {out_off[k], out_off[k + 1], in_off[k], in_off[k + 1]};
            if (r[0] < 0 || r[0] > r[1] || r[1] > n_spans || r[2] < 0 || r[2] > r[3] || r[3] > n_spans)
                return MW_EEDITS;
            for (int part = 0; part < 2; ++part)
                for (int q = r[2 * part]; q < r[2 * part + 1]; ++q) {
                    const int a0 = spans[2 * q], b0 = spans[2 * q + 1];
                    if (!(0 <= a0 && a0 < b0 && b0 <= J[k])) return MW_EEDITS;
                }
            for (int q = r[0]; q < r[1]; ++q)
                for (int j = spans[2 * q]; j < spans[2 * q + 1]; ++j) out[j] = 1;
            for (int q = r[2]; q < r[3]; ++q)
                for (int j = spans[2 * q]; j < spans[2 * q + 1]; ++j) {
                    if (!out[j]) return MW_EEDITS;
                    out[j] = 0;
                }
            for (int x = 0; x < 4; ++x) jtab[4 * k + x] = r[x];
        }
        for (int k = 0; k < n_junc; ++k)
            for (int part = 0; part < 2; ++part)
                for (int q = jtab[4 * k + 2 * part]; q < jtab[4 * k + 2 * part + 1]; ++q) {
                    sp2[2 * q] = cu[jt[k]] + spans[2 * q];
                    sp2[2 * q + 1] = cu[jt[k]] + spans[2 * q + 1];
                }
    }
    cudaStream_t stream = (cudaStream_t)stream_;
    if (L->vis_bytes == 0) return MW_OK;
    const int64_t n_tiles = L->n_tiles;
    std::vector<char> img;
    pack_meta(L, cu, n_junc, J, jt, img);
    const UploadPart parts[3] = {{img.data(), at<char>(vis, L->off_traj_tok), img.size()},
                                 {sp2.data(), at<char>(ws, L->ws_off_spans), sp2.size() * 4},
                                 {jtab.data(), at<char>(ws, L->ws_off_tstat), jtab.size() * 4}};
    if ((st = upload_parts(parts, 3, stream, true)) != MW_OK) return st;
    // no tile classes or lists for these views: empty lists, zero classes
    if ((st = cuda_status(cudaMemsetAsync(at<char>(vis, L->off_cls), 0, (size_t)L->n_tri, stream))) != MW_OK ||
        (st = cuda_status(cudaMemsetAsync(at<char>(vis, L->off_fwd_ptr), 0, 4 * (size_t)(n_tiles + 1), stream))) !=
            MW_OK ||
        (st = cuda_status(cudaMemsetAsync(at<char>(vis, L->off_bwd_ptr), 0, 4 * (size_t)(n_tiles + 1), stream))) !=
            MW_OK ||
        (st = cuda_status(cudaMemsetAsync(at<char>(vis, L->off_pairs), 0, 8 * (size_t)(n_traj + 1), stream))) !=
            MW_OK ||
        (st = cuda_status(cudaMemsetAsync(at<char>(vis, L->off_status), 0, 32, stream))) != MW_OK ||
        (st = cuda_status(cudaMemsetAsync(at<char>(ws, L->ws_off_cnt), 0xff, 4 * (size_t)L->total_tokens, stream))) !=
            MW_OK)
        return st;
    BuildArgs a = {};
    a.n_traj = n_traj;
    a.total = L->total_tokens;
    a.omega = at<int32_t>(vis, L->off_omega);
    a.seg = at<int32_t>(vis, L->off_seg);
    a.traj_tok = at<int32_t>(vis, L->off_traj_tok);
    a.traj_seg = at<int32_t>(vis, L->off_traj_seg);
    a.seg_start = at<int32_t>(vis, L->off_seg_start);
    a.status = at<int32_t>(vis, L->off_status);
    EventArgs e;
    e.n_traj = n_traj;
    e.status = a.status;
    e.traj_tok = at<int32_t>(vis, L->off_traj_tok);
    e.traj_tile = at<int32_t>(vis, L->off_traj_tile);
    e.traj_seg = at<int32_t>(vis, L->off_traj_seg);
    e.traj_km = at<int64_t>(vis, L->off_traj_km);
    e.seg_start = at<int32_t>(vis, L->off_seg_start);
    e.spans = at<int32_t>(ws, L->ws_off_spans);
    e.jtab = at<int32_t>(ws, L->ws_off_tstat);
    e.flag = at<int32_t>(ws, L->ws_off_cnt);
    e.seg_len = at<int32_t>(vis, L->off_seg_len);
    e.cpos = at<int32_t>(vis, L->off_cpos);
    e.csrc = at<int32_t>(vis, L->off_csrc);
    e.pairs = at<unsigned long long>(vis, L->off_pairs);
    if (a.total > 0) {
        count_launches(1);
        k_init_tokens<<<(int)std::min<int64_t>(ceil_div(ceil_div(a.total, INIT_TPT), 256), 152 * 16), 256, 0,
                        stream>>>(a);
    }
    if (n_traj > 0) {
        count_launches(1);
        k_event_views<<<(unsigned)n_traj, 1024, 0, stream>>>(e);
    }
    if (L->n_keymask > 0) {
        count_launches(1);
        k_event_keymask<<<(unsigned)ceil_div(L->n_keymask * 32, 256), 256, 0, stream>>>(
            L->n_keymask, e.cpos, at<uint32_t>(vis, L->off_keymask));
    }
    return launch_status();
}

extern "C" mw_status mw_check_status(const mw_vis_layout* L, const void* vis, void* stream) {
    if (!L || !vis) return MW_EINVAL;
    int32_t h[8];
    mw_status st = cuda_status(cudaMemcpyAsync(h, at<char>(vis, L->off_status), sizeof(h),
                                               cudaMemcpyDeviceToHost, (cudaStream_t)stream));
    if (st != MW_OK) return st;
    if ((st = cuda_status(cudaStreamSynchronize((cudaStream_t)stream))) != MW_OK) return st;
    if (h[ST_TIMEOUT]) return MW_ETIMEOUT;
    if (h[ST_BOUNDS]) return MW_EDEVICE;
    return MW_OK;
}

extern "C" mw_status mw_export_dense_mask(const mw_vis_layout* L, const void* vis, const int32_t* cu_seqlens,
                                          int traj, uint32_t* mask, void* stream) {
    if (!L || !cu_seqlens) return MW_EINVAL;
    if (traj < 0 || traj >= L->n_traj || cu_seqlens[L->n_traj] != L->total_tokens) return MW_EINVAL;
    const int64_t T = (int64_t)cu_seqlens[traj + 1] - cu_seqlens[traj];
    if (T < 0) return MW_EINVAL;
    if (T == 0) return MW_OK;
    if (T > MW_DENSE_MASK_MAX_T) return MW_ESHAPE;
    if (!vis || !mask) return MW_EINVAL;
    count_launches(1);
    k_dense_mask<<<(unsigned)ceil_div(T, DM_ROWS), 256, 0, (cudaStream_t)stream>>>(
        make_view(L, vis), traj, (int)T, (int)((T + 31) / 32), L->kind != MW_VIEWS_EDITS, mask);
    return launch_status();
}
