// Tensor-core LM-head backward without materialising logits.
//
//   dz_{m,v} = dloss g_m (1[v = tgt_m] - exp(z_{m,v} - lse_m)),  z = Hg W^T
//   dH_{rows[m]} = sum_v dz_{m,v} W_v        (pass 0: loss rows stationary)
//   dW_v         = sum_m dz_{m,v} Hg_m       (pass 1: vocab rows stationary)
//
// The accumulator of one 128-row tile over the whole hidden size d (128 x d
// fp32) is larger than one SM's tensor memory, so a thread-block cluster of C
// CTAs splits d: CTA c owns columns [c ds, (c+1) ds), ds = d / C, keeps its
// slice X_c of the stationary 128-row operand resident in shared memory and
// streams NY-row tiles Y_t of the other operand (TMA, YS-stage ring). Per step t:
//   1. Zp = X_c Y_t,c^T            partial logits over the CTA's d-slice (TMEM,
//                                  ZB buffers so the next steps run ahead)
//   2. reduce-scatter through distributed shared memory: sender warps push
//      row i of the partial to owner CTA i / (128 / C) with st.async (the
//      stores complete the owner's mbarrier); owner warps sum the C partials,
//      form dz (bf16) for their rows and st.async them into every CTA's dz
//      buffer
//   3. Acc_c += dz Y_t,c           (Y_t read again as an MN-major operand)
// Cross-CTA hand-offs use mbarriers only (transaction bytes, remote
// release-arrives for buffer-free signals, MMA completion multicast to every
// CTA); every wait is bounded in time. Before exiting each CTA waits for every
// remote arrival aimed at it.

#include <math.h>

#include "common.cuh"
#include "tc.cuh"
#include "tmap.cuh"

namespace mw {

namespace {

using namespace tc;

constexpr int NT = 320;   // TMA, MMA, 4 sender warps, 4 owner warps
constexpr float LOG2E_B = 1.4426950408889634f;

struct LmBwdParams {
    int mode;            // 0: dH pass, 1: dW pass
    int C, ds, NY, XB;   // cluster size, d-slice, streamed rows per step, exchange buffers
    int YS, ZB;          // streamed-tile stages (<= 3), partial-logit TMEM buffers (<= 3)
    int NS;              // steps
    int M, M_pad, d, V;
    float dloss;
    const int32_t* rows;   // [M]
    const int32_t* tg;     // [M_pad] targets of the loss rows
    const float* g;        // [M]
    const float* lse;      // [M]
    __nv_bfloat16* dH;     // [N, d]
    float* dW;             // [V, d]
    int32_t* status;
    // shared-memory map (bytes from the 1024-aligned base)
    uint32_t sm_x, sm_y, sm_dz, sm_xb, y_stage_b, dz_b;
};

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ uint32_t mapa(uint32_t addr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}
// Asynchronous store into a peer CTA's shared memory that completes 16 bytes
// of the transaction count of the peer's mbarrier when it lands (no fence).
__device__ __forceinline__ void st_async_v4(uint32_t addr, uint4 v, uint32_t remote_bar) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.b32 [%0], {%1,%2,%3,%4}, [%5];" ::"r"(addr),
                 "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "r"(remote_bar)
                 : "memory");
}
__device__ __forceinline__ void arrive_remote(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
// Non-suspending poll: the arrivals on these barriers come from other CTAs,
// and a suspended try_wait is not woken promptly by them.
__device__ __forceinline__ bool try_wait_cluster(uint32_t addr, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(addr), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded acquire-at-cluster-scope wait (for barriers that other CTAs arrive on).
__device__ __forceinline__ bool wait_cluster(uint64_t* bar, uint32_t parity, int32_t* status, int where) {
    const uint32_t a = smem_u32(bar);
    if (try_wait_cluster(a, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t i = 1;; ++i) {
        if (try_wait_cluster(a, parity)) return true;
        if ((i & 255u) == 0 &&
            ((status && *(volatile int32_t*)&status[1]) || globaltimer_ns() - t0 > kWaitLimitNs))
            break;
    }
    if (status) {
        atomicExch(&status[1], 1);
        atomicCAS(&status[2], 0, where);
    }
    return false;
}
__device__ __forceinline__ void commit_multicast(uint64_t* bar, uint16_t mask) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::
                     "r"(smem_u32(bar)),
                 "h"(mask)
                 : "memory");
}

__global__ void __launch_bounds__(NT, 1)
    k_lm_bwd_tc(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmY, LmBwdParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t x_full, y_full[3], y_empty[3], z_full[3], z_free[3], p_full[2], p_free[2],
        dz_full[2], dz_free[2], acc_done, sent[2], done[2];
    __shared__ uint32_t tmem_base;
    __shared__ float4 colpar[2][128];   // dW pass: (g dloss, lse log2 e, target, valid) per streamed row

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int C = p.C, ds = p.ds, NY = p.NY, XB = p.XB, NS = p.NS, YS = p.YS, ZB = p.ZB;
    const int rank = (int)cluster_rank();
    const int tile = blockIdx.x / C;           // stationary 128-row tile
    const int RPO = 128 / C;                   // rows owned by each CTA in the exchange
    const int col0 = rank * ds;                // this CTA's d-slice
    const uint32_t TM_ACC = 0, TM_Z = (uint32_t)ds;
    int32_t* status = p.status;

    if (threadIdx.x == 0) {
        mbar_init(&x_full, 1);
        for (int s = 0; s < 3; ++s) {
            mbar_init(&y_full[s], 1);
            mbar_init(&y_empty[s], 1);
            mbar_init(&z_full[s], 1);
            mbar_init(&z_free[s], 128);
        }
        for (int s = 0; s < 2; ++s) {
            // data barriers: armed once per phase by their own CTA with the
            // byte count; the peers' st.async stores complete the bytes
            mbar_init(&p_full[s], 1);
            mbar_init(&dz_full[s], 1);
            // buffer-free signals: one arrive from each CTA of the cluster
            mbar_init(&p_free[s], C);
            mbar_init(&dz_free[s], C);
            mbar_init(&sent[s], 128);
            mbar_init(&done[s], 128);
        }
        mbar_init(&acc_done, 1);
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&tmem_base, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    // every CTA's barriers are initialised before any remote arrive
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
    tc_fence_after();
    const uint32_t tmem = tmem_base;
    const uint32_t base = smem_u32(sm);

    if (warp == 0) {
        if (lane == 0) {
            prefetch_tmap(&tmX);
            prefetch_tmap(&tmY);
            const int nbox = ds / 64;
            mbar_expect_tx(&x_full, (uint32_t)(128 * ds * 2));
            for (int j = 0; j < nbox; ++j)
                tma_load_2d(sm + p.sm_x + j * 16384, &tmX, &x_full, col0 + j * 64, tile * 128);
            for (int t = 0; t < NS; ++t) {
                const int s = t % YS;
                if (t >= YS && !mbar_wait(&y_empty[s], ((t - YS) / YS) & 1, status, 501)) break;
                mbar_expect_tx(&y_full[s], (uint32_t)(NY * ds * 2));
                uint8_t* dst = sm + p.sm_y + s * p.y_stage_b;
                for (int j = 0; j < nbox; ++j) tma_load_2d(dst + j * NY * 128, &tmY, &y_full[s], col0 + j * 64, t * NY);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t iZ = idesc_bf16(128, NY, 0, 0);
            const uint32_t xb = base + p.sm_x;
            const uint16_t mask = (uint16_t)((1u << C) - 1u);
            bool ok = mbar_wait(&x_full, 0, status, 511);
            auto issue_z = [&](int t) -> bool {
                const int ys = t % YS, zs = t % ZB;
                if (!mbar_wait(&y_full[ys], (t / YS) & 1, status, 512)) return false;
                if (t >= ZB && !mbar_wait(&z_free[zs], ((t - ZB) / ZB) & 1, status, 513)) return false;
                tc_fence_after();
                const uint32_t yb = base + p.sm_y + ys * p.y_stage_b;
                for (int ks = 0; ks < ds / 16; ++ks)
                    mma_ss(tmem + TM_Z + zs * NY, sdesc_sw128(xb + (ks >> 2) * 16384 + (ks & 3) * 32, 16, 1024),
                           sdesc_sw128(yb + (ks >> 2) * (NY * 128) + (ks & 3) * 32, 16, 1024), iZ, ks > 0);
                mma_commit(&z_full[zs]);
                return true;
            };
            auto issue_acc = [&](int t) -> bool {
                const int s = t & 1;
                // arm: this step's dz tile is 128 rows x NY bf16 from the owners
                mbar_expect_tx(&dz_full[s], (uint32_t)(128 * NY * 2));
                if (!wait_cluster(&dz_full[s], (t >> 1) & 1, status, 514)) return false;
                // dz was written by other CTAs' threads; order it before this
                // thread's tensor-core (async proxy) reads
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                tc_fence_after();
                const int ys = t % YS;
                const uint32_t yb = base + p.sm_y + ys * p.y_stage_b;
                const uint32_t db = base + p.sm_dz + (NY <= 32 ? s * 64 : s * p.dz_b);
                for (int n0 = 0; n0 < ds; n0 += 256) {
                    const int nn = min(256, ds - n0);
                    const uint32_t iA = idesc_bf16(128, nn, 0, 1);
                    for (int ks = 0; ks < NY / 16; ++ks)
                        mma_ss(tmem + TM_ACC + n0, sdesc_sw128(db + (ks >> 2) * 16384 + (ks & 3) * 32, 16, 1024),
                               sdesc_sw128(yb + (n0 / 64) * (NY * 128) + ks * 2048, NY * 128, 1024), iA,
                               (t > 0 || ks > 0));
                }
                mma_commit(&y_empty[ys]);
                commit_multicast(&dz_free[s], mask);
                return true;
            };
            // the partial logits of the next ZB-1 steps are issued before the
            // accumulation of step t, which waits for the exchange
            for (int t = 0; ok && t < ZB - 1 && t < NS; ++t) ok = issue_z(t);
            for (int t = 0; ok && t < NS; ++t) {
                if (t + ZB - 1 < NS && !issue_z(t + ZB - 1)) { ok = false; break; }
                if (!issue_acc(t)) { ok = false; break; }
            }
            if (ok) mma_commit(&acc_done);
        }
    } else if (warp < 6) {
        // ------------------------------------------------------------ senders
        // warps 2..5: partial logits of step t -> the row's owner CTA; the
        // st.async stores complete the owner's barrier themselves
        const int qw = warp & 3;
        const int rl = qw * 32 + lane;                      // stationary row = TMEM lane
        const uint32_t lane_base = tmem + ((uint32_t)(qw * 32) << 16);
        const uint32_t xbuf_bytes = (uint32_t)(128 * NY * 4);
        const int cpr = NY / 4, cmask = (cpr < 8 ? cpr : 8) - 1;   // 16-byte chunks per row, swizzle mask
        const int owner = rl / RPO;
        bool ok = true;
        for (int t = 0; t < NS; ++t) {
            const int xs = t % XB, zb = t % ZB;
            if (!mbar_wait(&z_full[zb], (t / ZB) & 1, status, 521)) { ok = false; break; }
            if (t >= XB && !wait_cluster(&p_free[xs], ((t - XB) / XB) & 1, status, 522)) { ok = false; break; }
            tc_fence_after();
            // row rl of the partial goes to row (rank RPO + rl % RPO) of the
            // owner's exchange buffer, 16-byte chunks XOR-swizzled by the row
            const uint32_t dst = mapa(base + p.sm_xb + xs * xbuf_bytes + (uint32_t)((rank * RPO + rl % RPO) * NY * 4),
                                      (uint32_t)owner);
            const uint32_t obar = mapa(smem_u32(&p_full[xs]), (uint32_t)owner);
            for (int q = 0; q < NY / 16; ++q) {
                uint32_t z[16];
                tmem_ld16(lane_base + TM_Z + zb * NY + q * 16, z);
                tmem_wait_ld();
#pragma unroll
                for (int x = 0; x < 4; ++x) {
                    const int c = q * 4 + x;
                    st_async_v4(dst + 16 * (c ^ (rl & cmask)), make_uint4(z[4 * x], z[4 * x + 1], z[4 * x + 2], z[4 * x + 3]),
                                obar);
                }
            }
            tc_fence_before();
            mbar_arrive(&z_free[zb]);
        }
        // the owners' last buffer-free signals are still aimed at this CTA
        for (int t = max(0, NS - XB); ok && t < NS; ++t)
            if (!wait_cluster(&p_free[t % XB], (t / XB) & 1, status, 526)) ok = false;
    } else {
        // ------------------------------------------------------------ owners
        // warps 6..9: sum the C partials of this CTA's RPO rows, form dz and
        // write it (bf16) into every CTA's dz buffer; then the output
        const int qw = warp & 3;
        const int rl = qw * 32 + lane;
        const int tid = threadIdx.x - 192;                  // 0..127
        const uint32_t lane_base = tmem + ((uint32_t)(qw * 32) << 16);
        const uint32_t xbuf_bytes = (uint32_t)(128 * NY * 4);
        const int groups = RPO * NY / 8;
        const int cpr = NY / 4, cmask = (cpr < 8 ? cpr : 8) - 1;   // the senders' chunk swizzle
        const bool packed = NY <= 32;   // both dz buffers share one swizzled tile
        bool ok = true;
        for (int t = 0; t < NS; ++t) {
            const int s = t & 1, xs = t % XB;
            if (p.mode == 1 && tid < NY) {
                const int m = t * NY + tid;
                colpar[s][tid] = m < p.M ? make_float4(p.g[m] * p.dloss, p.lse[m] * LOG2E_B, __int_as_float(p.tg[m]), 1.f)
                                         : make_float4(0.f, 0.f, __int_as_float(-1), 0.f);
            }
            // arm this CTA's owner barrier: RPO rows x C senders x NY fp32
            if (tid == 0) mbar_expect_tx(&p_full[xs], (uint32_t)(128 * NY * 4));
            mbar_arrive(&sent[s]);   // makes colpar visible to all owner threads
            if (!mbar_wait(&sent[s], (t >> 1) & 1, status, 528)) { ok = false; break; }
            if (!wait_cluster(&p_full[xs], (t / XB) & 1, status, 523)) { ok = false; break; }
            if (t >= 2 && !wait_cluster(&dz_free[s], ((t - 2) >> 1) & 1, status, 524)) { ok = false; break; }
            const float* xb = reinterpret_cast<const float*>(sm + p.sm_xb + xs * xbuf_bytes);
            for (int gi = tid; gi < groups; gi += 128) {
                const int ro = gi / (NY / 8), cg = gi % (NY / 8);
                float zs[8];
#pragma unroll
                for (int x = 0; x < 8; ++x) zs[x] = 0.f;
                for (int snd = 0; snd < C; ++snd) {
                    const float* rowp = xb + (snd * RPO + ro) * NY;
                    const float4 a = *reinterpret_cast<const float4*>(rowp + 4 * ((2 * cg) ^ (ro & cmask)));
                    const float4 b = *reinterpret_cast<const float4*>(rowp + 4 * ((2 * cg + 1) ^ (ro & cmask)));
                    zs[0] += a.x; zs[1] += a.y; zs[2] += a.z; zs[3] += a.w;
                    zs[4] += b.x; zs[5] += b.y; zs[6] += b.z; zs[7] += b.w;
                }
                const int row = rank * RPO + ro;   // stationary row inside the tile
                float dz[8];
                if (p.mode == 0) {
                    const int m = tile * 128 + row;
                    const bool okm = m < p.M;
                    const float gm = okm ? p.g[m] * p.dloss : 0.f;
                    const float l2 = okm ? p.lse[m] * LOG2E_B : 0.f;
                    const int tgm = okm ? p.tg[m] : -1;
#pragma unroll
                    for (int x = 0; x < 8; ++x) {
                        const int v = t * NY + cg * 8 + x;
                        const float pr = ex2f_approx(fmaf(zs[x], LOG2E_B, -l2));
                        dz[x] = (okm && v < p.V) ? gm * ((v == tgm ? 1.f : 0.f) - pr) : 0.f;
                    }
                } else {
                    const int v = tile * 128 + row;
#pragma unroll
                    for (int x = 0; x < 8; ++x) {
                        const float4 cp = colpar[s][cg * 8 + x];
                        const float pr = ex2f_approx(fmaf(zs[x], LOG2E_B, -cp.y));
                        dz[x] = (cp.w != 0.f && v < p.V)
                                    ? cp.x * ((v == __float_as_int(cp.z) ? 1.f : 0.f) - pr)
                                    : 0.f;
                    }
                }
                uint4 pk;
                pk.x = pack_bf16(dz[0], dz[1]);
                pk.y = pack_bf16(dz[2], dz[3]);
                pk.z = pack_bf16(dz[4], dz[5]);
                pk.w = pack_bf16(dz[6], dz[7]);
                // every CTA's dz buffer s, in the 128-byte-swizzled K-major layout
                // of the accumulation MMA's A operand (two buffers share one
                // tile, one 64-byte half of each row each, when NY <= 32)
                const uint32_t off = (uint32_t)((packed ? 0 : s * p.dz_b) + (cg >> 3) * 16384) +
                                     sw128_off((uint32_t)row, (uint32_t)((cg & 7) + (packed ? s * 4 : 0)));
                const uint32_t dzbar = smem_u32(&dz_full[s]);
                for (int dcta = 0; dcta < C; ++dcta)
                    st_async_v4(mapa(base + p.sm_dz + off, (uint32_t)dcta), pk, mapa(dzbar, (uint32_t)dcta));
            }
            // every read of this CTA's exchange buffer is done: free it
            mbar_arrive(&done[s]);
            if (!mbar_wait(&done[s], (t >> 1) & 1, status, 529)) { ok = false; break; }
            if (tid < C) arrive_remote(mapa(smem_u32(&p_free[xs]), (uint32_t)tid));
        }
        // output: this CTA's d-slice of the accumulator
        if (ok && NS > 0 && mbar_wait(&acc_done, 0, status, 525)) {
            tc_fence_after();
            const int srow = tile * 128 + rl;
            bool valid;
            int64_t orow;
            if (p.mode == 0) {
                valid = srow < p.M;
                orow = valid ? (int64_t)p.rows[srow] : 0;
            } else {
                valid = srow < p.V;
                orow = srow;
            }
            for (int c0 = 0; c0 < ds; c0 += 32) {
                uint32_t o[32];
                tmem_ld32(lane_base + TM_ACC + c0, o);
                tmem_wait_ld();
                if (!valid) continue;
                if (p.mode == 0) {
                    __nv_bfloat16* dst = p.dH + orow * p.d + col0 + c0;
#pragma unroll
                    for (int x = 0; x < 4; ++x) {
                        uint4 pk;
                        pk.x = pack_bf16(__uint_as_float(o[8 * x + 0]), __uint_as_float(o[8 * x + 1]));
                        pk.y = pack_bf16(__uint_as_float(o[8 * x + 2]), __uint_as_float(o[8 * x + 3]));
                        pk.z = pack_bf16(__uint_as_float(o[8 * x + 4]), __uint_as_float(o[8 * x + 5]));
                        pk.w = pack_bf16(__uint_as_float(o[8 * x + 6]), __uint_as_float(o[8 * x + 7]));
                        reinterpret_cast<uint4*>(dst)[x] = pk;
                    }
                } else {
                    float* dst = p.dW + orow * p.d + col0 + c0;
#pragma unroll
                    for (int x = 0; x < 8; ++x)
                        reinterpret_cast<uint4*>(dst)[x] = make_uint4(o[4 * x], o[4 * x + 1], o[4 * x + 2], o[4 * x + 3]);
                }
            }
        }
        // the last dz-free signals (MMA completions of every CTA) aim here
        for (int t = max(0, NS - 2); ok && t < NS; ++t)
            if (!wait_cluster(&dz_free[t & 1], (t >> 1) & 1, status, 527)) ok = false;
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

struct BwdCfg {
    int C, ds, NY, XB, YS, ZB;
    uint32_t smem;
};

// dz buffers: two [128][NY] bf16 tiles, or one shared 128-byte-swizzled tile
// (each buffer in one 64-byte half of every row) when NY <= 32.
// dz buffers: two [128][NY] bf16 128-byte-swizzled tiles, or one shared tile
// (each buffer in one 64-byte half of every row) when NY <= 32.
uint32_t dz_region(int NY) { return NY <= 32 ? 16384u : (NY <= 64 ? 2 * 16384u : 2 * 32768u); }

uint32_t bwd_smem(int ds, int NY, int XB, int YS, int C) {
    return (uint32_t)(128 * ds * 2          // X slice
                      + YS * NY * ds * 2    // Y ring
                      + dz_region(NY)       // dz buffers
                      + XB * 128 * NY * 4   // exchange buffers
                      + 1024);
}

// Smallest cluster that fits TMEM (ds + ZB NY <= 512) and shared memory; then
// the widest streamed tile; then double exchange buffers (they decouple the
// senders from the owners); then the deepest pipeline. ZB <= YS: each extra
// partial-logit tile in flight needs its own streamed-tile stage.
bool choose_cfg(int d, BwdCfg& c) {
    const uint32_t limit = 220 * 1024;
    for (int C : {1, 2, 4, 8}) {
        if (d % C) continue;
        const int ds = d / C;
        if (ds % 64 || ds > 448) continue;
        for (int NY : {128, 64, 32, 16})
            for (int XB : {2, 1})
                for (int ZB : {3, 2}) {
                    if (ds + ZB * NY > 512) continue;
                    for (int YS : {3, 2}) {
                        if (ZB > YS) continue;
                        const uint32_t sm = bwd_smem(ds, NY, XB, YS, C);
                        if (sm <= limit) {
                            c = {C, ds, NY, XB, YS, ZB, sm};
                            return true;
                        }
                    }
                }
    }
    return false;
}

}  // namespace

bool lm_bwd_tc_supported(int d) {
    BwdCfg c;
    return choose_cfg(d, c);
}

mw_status lm_bwd_tc(const void* W, int M, int N, int d, int V, const int32_t* rows, const void* Hg, const int32_t* tg,
                    const float* lse, const float* g, float dloss, void* dH, float* dW, int32_t* status,
                    cudaStream_t s) {
    BwdCfg c;
    if (!choose_cfg(d, c)) return MW_ESHAPE;
    mw_status st = cuda_status(cudaMemsetAsync(dH, 0, (size_t)N * d * 2, s));
    if (st != MW_OK) return st;
    if (M == 0) return cuda_status(cudaMemsetAsync(dW, 0, (size_t)V * d * 4, s));
    const int M_pad = (int)ceil_div(M, 128) * 128;
    CUtensorMap hx, hy, wx, wy;
    if (!tmap_bf16_2d(&hx, Hg, M_pad, d, d, 128, 64) || !tmap_bf16_2d(&hy, Hg, M_pad, d, d, c.NY, 64) ||
        !tmap_bf16_2d(&wx, W, V, d, d, 128, 64) || !tmap_bf16_2d(&wy, W, V, d, d, c.NY, 64))
        return MW_ECUDA;
    if ((st = cuda_status(cudaFuncSetAttribute(k_lm_bwd_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)c.smem))) != MW_OK)
        return st;
    LmBwdParams p;
    p.C = c.C;
    p.ds = c.ds;
    p.NY = c.NY;
    p.XB = c.XB;
    p.YS = c.YS;
    p.ZB = c.ZB;
    p.M = M;
    p.M_pad = M_pad;
    p.d = d;
    p.V = V;
    p.dloss = dloss;
    p.rows = rows;
    p.tg = tg;
    p.g = g;
    p.lse = lse;
    p.dH = (__nv_bfloat16*)dH;
    p.dW = dW;
    p.status = status;
    p.sm_x = 0;
    p.sm_y = (uint32_t)(128 * c.ds * 2);
    p.y_stage_b = (uint32_t)(c.NY * c.ds * 2);
    p.sm_dz = p.sm_y + c.YS * p.y_stage_b;
    p.dz_b = c.NY <= 64 ? 16384u : 32768u;
    p.sm_xb = p.sm_dz + dz_region(c.NY);
    for (int mode = 0; mode < 2; ++mode) {
        p.mode = mode;
        const int tiles = mode == 0 ? M_pad / 128 : (int)ceil_div(V, 128);
        p.NS = mode == 0 ? (int)ceil_div(V, c.NY) : M_pad / c.NY;
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = c.C;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3((unsigned)(tiles * c.C));
        cfg.blockDim = dim3(NT);
        cfg.dynamicSmemBytes = c.smem;
        cfg.stream = s;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        count_launches(1);
        if ((st = cuda_status(cudaLaunchKernelEx(&cfg, k_lm_bwd_tc, mode == 0 ? hx : wx, mode == 0 ? wy : hy, p))) !=
            MW_OK)
            return st;
    }
    return launch_status();
}

}  // namespace mw
