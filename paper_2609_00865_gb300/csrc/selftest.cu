// Self-test of the bounded-wait failure path: a kernel waits on an mbarrier
// that nothing arrives on, gives up after a caller-chosen limit, records the
// timeout in a status word and returns, leaving the context usable. No GPU
// fault, trap or unbounded loop is involved.

#include "common.cuh"
#include "tc.cuh"

namespace mw {
namespace {

__global__ void k_wait_timeout(uint64_t limit_ns, int32_t* status) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x != 0) return;
    tc::mbar_init(&bar, 1);
    tc::fence_mbar_init();
    const uint32_t a = tc::smem_u32(&bar);
    const uint64_t t0 = tc::globaltimer_ns();
    for (uint32_t i = 0;; ++i) {
        if (tc::mbar_try_wait(a, 0)) return;   // never: no thread arrives
        if ((i & 255u) == 0 && tc::globaltimer_ns() - t0 > limit_ns) break;
    }
    atomicExch(&status[1], 1);
    atomicCAS(&status[2], 0, 999);
}

}  // namespace
}  // namespace mw

using namespace mw;

extern "C" mw_status mw_selftest_wait_timeout(int64_t limit_ns, int32_t* status, void* stream) {
    if (!status || limit_ns <= 0 || limit_ns > 1000000000ll) return MW_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    mw_status st = cuda_status(cudaMemsetAsync(status, 0, 8 * sizeof(int32_t), s));
    if (st != MW_OK) return st;
    count_launches(1);
    k_wait_timeout<<<1, 32, 0, s>>>((uint64_t)limit_ns, status);
    if ((st = launch_status()) != MW_OK) return st;
    int32_t h[8];
    if ((st = cuda_status(cudaMemcpyAsync(h, status, sizeof(h), cudaMemcpyDeviceToHost, s))) != MW_OK) return st;
    if ((st = cuda_status(cudaStreamSynchronize(s))) != MW_OK) return st;
    return h[1] ? MW_ETIMEOUT : MW_OK;
}
