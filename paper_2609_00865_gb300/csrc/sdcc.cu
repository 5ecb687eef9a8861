// SDCC support (§5, self-distillation for conditioning consistency): the
// diverging rows.
//
// A row diverges when its live prefix differs from its prefix on the final
// compressed walk (App. B Def. "trajectory tree"): some key it saw is evicted
// by a later edit, i.e. there is j <= r with r < omega(j) < never. With
// F(r) = max{omega(j) : j <= r, omega(j) finite} (or -1), row r diverges iff
// F(r) > r: one prefix-max scan of the lifetimes per trajectory. These are
// the rows where SDCC places its KL term.

#include "common.cuh"

namespace mw {
namespace {

constexpr int DIV_NT = 1024;

// One block per trajectory: chunks of 1024 rows, warp max-scans, carry.
__global__ void __launch_bounds__(DIV_NT) k_diverging_rows(VisView v, uint8_t* __restrict__ out) {
    __shared__ int wmax[DIV_NT / 32];
    __shared__ int carry_s;
    const int b = blockIdx.x;
    const int64_t tok0 = v.traj_tok[b];
    const int T = v.traj_tok[b + 1] - (int)tok0;
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    if (t == 0) carry_s = -1;
    __syncthreads();
    for (int c0 = 0; c0 < T; c0 += DIV_NT) {
        const int r = c0 + t;
        int x = -1;
        if (r < T) {
            const int om = v.omega[tok0 + r];
            x = om < INT32_MAX ? om : -1;
        }
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x = max(x, y);
        }
        if (lane == 31) wmax[w] = x;
        __syncthreads();
        int f = carry_s;
        for (int q = 0; q < w; ++q) f = max(f, wmax[q]);
        f = max(f, x);
        if (r < T) out[tok0 + r] = f > r ? 1 : 0;
        __syncthreads();
        if (t == DIV_NT - 1) carry_s = f;
        __syncthreads();
    }
}

}  // namespace
}  // namespace mw

using namespace mw;

extern "C" mw_status mw_diverging_rows(const mw_vis_layout* L, const void* vis, uint8_t* out, void* stream) {
    if (!L) return MW_EINVAL;
    if (L->total_tokens == 0) return MW_OK;
    if (!vis || !out) return MW_EINVAL;
    count_launches(1);
    k_diverging_rows<<<(unsigned)L->n_traj, DIV_NT, 0, (cudaStream_t)stream>>>(make_view(L, vis), out);
    return launch_status();
}
