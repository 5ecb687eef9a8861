// mw_build_visibility_noalloc: the visibility builder for callers that are
// handed their input and output buffers and may not allocate device memory
// themselves -- for example a plugin inside a host framework that owns all
// device memory through its own pool, where a cudaMalloc would synchronise the
// device or bypass the pool's accounting. The build workspace (span table,
// per-k-tile lifetime bounds, tile-list lengths) lives in a fixed file-scope
// device array instead of a caller-provided buffer.
//
// The array is kStaticWsBytes long and is resident on every GPU that loads
// this library until the process exits. Every call on a device shares it and
// it keeps the previous call's contents; nothing in it has to start at zero,
// because each call overwrites every byte it later reads (the span table is
// copied in, the tile statistics and list lengths are written by kernels
// before they are read). Calls whose GPU work overlaps (different streams or
// threads on one device) race on the array and must be serialised by the
// caller.
//
// With lazy module loading (CUDA's default) the first cudaGetSymbolAddress on
// a device loads this library's device code there, which places the array
// and may synchronise the device; callers make a warm-up call at set-up time.
// The looked-up address is cached per device ordinal for the life of the
// process and is stale after a cudaDeviceReset of that device.

#include <mutex>

#include "common.cuh"

namespace mw {
mw_status build_visibility(const mw_vis_layout*, const int32_t*, int, const int32_t*, const int32_t*, const int32_t*,
                           const int32_t*, void*, void*, void*, bool);
}

namespace {

constexpr long long kStaticWsBytes = 1ll << 20;  // 1 MiB
static __device__ __align__(256) unsigned char g_vis_ws[kStaticWsBytes];

constexpr int kMaxDevices = 64;
static void* g_ws_addr[kMaxDevices];  // device address of g_vis_ws, per device
static std::mutex g_ws_mu;

}  // namespace

extern "C" mw_status mw_build_visibility_noalloc(const mw_vis_layout* L, const int32_t* cu_seqlens, int n_junc,
                                                 const int32_t* junctions, const int32_t* junc_traj,
                                                 const int32_t* junc_span_off, const int32_t* spans, void* vis,
                                                 void* stream) {
    if (!L) return MW_EINVAL;
    if (L->ws_bytes > kStaticWsBytes) return MW_ENOSPACE;
    int dev = 0;
    mw_status st = mw::cuda_status(cudaGetDevice(&dev));
    if (st != MW_OK) return st;
    if (dev < 0 || dev >= kMaxDevices) return MW_ENOSPACE;
    void* ws = nullptr;
    {
        // First call on a device: look up the array's device address with
        // that device current (host code cannot use the symbol itself).
        std::lock_guard<std::mutex> lock(g_ws_mu);
        if (!g_ws_addr[dev]) {
            void* p = nullptr;
            st = mw::cuda_status(cudaGetSymbolAddress(&p, g_vis_ws));
            if (st != MW_OK) return st;
            g_ws_addr[dev] = p;
        }
        ws = g_ws_addr[dev];
    }
    // the record goes up from pageable memory: no page-locked staging buffer
    return mw::build_visibility(L, cu_seqlens, n_junc, junctions, junc_traj, junc_span_off, spans, ws, vis, stream,
                                false);
}
