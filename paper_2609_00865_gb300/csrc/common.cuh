// Shared device/host helpers for libmw (no method arithmetic here).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "mw.h"

namespace mw {

// Record the CUDA error (if any) in the thread-local slot and map to status.
mw_status cuda_status(cudaError_t e);
mw_status launch_status();
// Count `n` kernel launches issued by the library (see mw_kernel_launches).
void count_launches(int n);

inline int64_t align256(int64_t x) { return (x + 255) & ~int64_t(255); }
inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

template <typename T>
__host__ __device__ inline T* at(void* base, int64_t off) {
    return reinterpret_cast<T*>(reinterpret_cast<char*>(base) + off);
}
template <typename T>
__host__ __device__ inline const T* at(const void* base, int64_t off) {
    return reinterpret_cast<const T*>(reinterpret_cast<const char*>(base) + off);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ int warp_sum_i(int v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Element loads that widen to float (the inputs are float32 or bfloat16).
__device__ __forceinline__ float ld_f(const float* p) { return *p; }
__device__ __forceinline__ float ld_f(const __nv_bfloat16* p) { return __bfloat162float(*p); }
__device__ __forceinline__ void st_f(float* p, float v) { *p = v; }
__device__ __forceinline__ void st_f(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

// Visibility context for one launch: base pointers into the `vis` buffer.
struct VisView {
    const int32_t* omega;
    const int32_t* seg;
    const int32_t* traj_tok;
    const int32_t* traj_tile;
    const int32_t* traj_seg;
    const int64_t* traj_tri;
    const int64_t* traj_km;
    const int32_t* seg_start;
    const int32_t* tile_traj;
    const uint8_t* cls;
    const int32_t* fwd_ptr;
    const int32_t* fwd_idx;
    const int32_t* bwd_ptr;
    const int32_t* bwd_idx;
    const uint32_t* keymask;
    const int32_t* seg_len;   // [n_segs] |view_s|
    const int32_t* cpos;      // [n_keymask][128] rank of key j in view_s, -1 if absent
    const int32_t* csrc;      // [n_keymask][128] key (traj-local) at each rank of view_s
    int32_t* status;
    int64_t total, n_keymask; // sizes for the debug library's index checks
};

inline VisView make_view(const mw_vis_layout* L, const void* vis) {
    VisView v;
    v.omega = at<int32_t>(vis, L->off_omega);
    v.seg = at<int32_t>(vis, L->off_seg);
    v.traj_tok = at<int32_t>(vis, L->off_traj_tok);
    v.traj_tile = at<int32_t>(vis, L->off_traj_tile);
    v.traj_seg = at<int32_t>(vis, L->off_traj_seg);
    v.traj_tri = at<int64_t>(vis, L->off_traj_tri);
    v.traj_km = at<int64_t>(vis, L->off_traj_km);
    v.seg_start = at<int32_t>(vis, L->off_seg_start);
    v.tile_traj = at<int32_t>(vis, L->off_tile_traj);
    v.cls = at<uint8_t>(vis, L->off_cls);
    v.fwd_ptr = at<int32_t>(vis, L->off_fwd_ptr);
    v.fwd_idx = at<int32_t>(vis, L->off_fwd_idx);
    v.bwd_ptr = at<int32_t>(vis, L->off_bwd_ptr);
    v.bwd_idx = at<int32_t>(vis, L->off_bwd_idx);
    v.keymask = at<uint32_t>(vis, L->off_keymask);
    v.seg_len = at<int32_t>(vis, L->off_seg_len);
    v.cpos = at<int32_t>(vis, L->off_cpos);
    v.csrc = at<int32_t>(vis, L->off_csrc);
    v.status = const_cast<int32_t*>(at<int32_t>(vis, L->off_status));
    v.total = L->total_tokens;
    v.n_keymask = L->n_keymask;
    return v;
}

// Status-word slots written by device code.
enum { ST_BOUNDS = 0, ST_TIMEOUT = 1, ST_WHERE = 2 };

// Loss rows and their targets are device arrays filled by the caller, so no
// host check sees them. A kernel takes such an index through checked_index:
// inside [0, n) it is returned, otherwise -1 and the row is not read or
// written; the kernel then raises the bounds flag of its status word (the
// status check reports MW_EDEVICE).
__device__ __forceinline__ int checked_index(int i, int n) { return (unsigned)i < (unsigned)n ? i : -1; }
__device__ __forceinline__ void flag_bounds(int32_t* status) {
    if (status) atomicExch(status + ST_BOUNDS, 1);
}

// Index checks of the debug library (compiled with -DMW_DEBUG into
// libmw_debug.so). At the accesses whose index is read from memory (a
// record's spans, the compact maps, segment tables) or derived from one,
// MW_DBG_IN(i, n, status, where) is false for i outside [0, n), after
// raising the bounds flag and recording the site `where` (the first one
// wins); the caller then skips the access. The status check reports
// MW_EDEVICE. In the release library it is the constant true and the
// check compiles away.
#ifdef MW_DEBUG
__device__ __forceinline__ bool dbg_in(long long i, long long n, int32_t* status, int where) {
    if (i >= 0 && i < n) return true;
    if (status) {
        atomicExch(status + ST_BOUNDS, 1);
        atomicCAS(status + ST_WHERE, 0, where);
    }
    return false;
}
#define MW_DBG_IN(i, n, status, where) (::mw::dbg_in((long long)(i), (long long)(n), (status), (where)))
#else
#define MW_DBG_IN(i, n, status, where) (true)
#endif

}  // namespace mw
