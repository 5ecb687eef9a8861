// Tensor-core LM-head backward without materialising logits.
//
//   dz_{m,v} = dloss g_m (1[v = tgt_m] - exp(z_{m,v} - lse_m)),  z = Hg W^T
//   dH_{rows[m]} = sum_v dz_{m,v} W_v        (pass 0: loss rows stationary)
//   dW_v         = sum_m dz_{m,v} Hg_m       (pass 1: vocab rows stationary)
//
// A pass holds a 128-row tile X of the stationary operand and streams the
// other operand Y. The tile's accumulator over the whole hidden size (128 x d
// fp32) is larger than one SM's tensor memory, so a cluster of C CTAs shares
// the tile: CTA r accumulates hidden columns [r ds, (r+1) ds), ds = d / C.
// Step t of the cluster covers C NY streamed rows; CTA r
//   1. computes the logits of its own NY streamed rows over the full hidden
//      size, Z_r = X Y_{t,r}^T (TMEM; X and Y k-slices streamed by TMA),
//   2. forms dz_r (bf16, 128 x NY) in the epilogue, writes it into its slot
//      of a per-cluster ring in global memory (R = L + 1 steps deep, a few
//      MB in all, so it stays in L2) and signals every CTA of the cluster,
//   3. accumulates Acc_r += sum_q dz_q Y_{t,q}[:, slice r] over the C dz
//      tiles of the step (dz tiles and Y slices loaded by TMA).
// Only bf16 dz tiles cross CTAs, once per step. The accumulation of step t
// is issued after the logits of step t + L, so the exchange has L steps of
// tensor work to complete in. Clusters are persistent (as many as fit on the
// GPU at once), so each owns a fixed ring region. One operand ring in shared
// memory carries the stages in the order the MMA thread consumes them: the
// k-slices of Z(t), then the Y slices of Acc(t - L). Every wait is bounded in
// time.

#include <math.h>

#include "common.cuh"
#include "tc.cuh"
#include "tmap.cuh"

namespace mw {

namespace {

using namespace tc;

constexpr int NT = 224;              // warp 0 TMA, warp 1 MMA, warp 2 signals, warps 3..6 epilogue
constexpr int MAX_S = 8, MAX_DS = 2, MAX_R = 4;
constexpr uint32_t SLOT = 32768;     // bytes per operand stage
constexpr int RING_CTAS = 160;       // ring capacity, in CTAs
constexpr float LOG2E_B = 1.4426950408889634f;

struct LmBwdParams {
    int mode;            // 0: dH pass, 1: dW pass
    int C, ds;           // cluster size, d-slice
    int S, DS;           // operand stages, dz-tile stages
    int L, R;            // accumulation lag in steps, ring depth R = L + 1
    int KD;              // 64-wide k-slices of d
    int NS;              // steps per tile
    int tiles, nclus;    // stationary tiles, clusters in the grid
    int M, M_pad, V;
    const int32_t* rows;   // [M]
    const float4* par;     // [M_pad] per loss row: (dloss g, lse log2 e, target bits, valid)
    __nv_bfloat16* dH;     // [N, d]
    float* dW;             // [V, d]
    __nv_bfloat16* ring;   // [nclus][R][C][128][NY] dz exchange ring
    int32_t* status;
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
__device__ __forceinline__ void arrive_remote(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
// Orders this thread's generic global accesses with the async proxy (TMA).
__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}
// Non-suspending poll: the arrivals on these barriers come from other CTAs.
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

template <int NY>
__global__ void __launch_bounds__(NT, 1)
    k_lm_bwd_tc(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmYz,
                const __grid_constant__ CUtensorMap tmYa, const __grid_constant__ CUtensorMap tmD, LmBwdParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t op_full[MAX_S], op_empty[MAX_S], dz_full[MAX_DS], dz_empty[MAX_DS], zt_full,
        zt_free, acc_full, acc_free, epi_done[MAX_R], dz_ready[MAX_R], dz_free[MAX_R];
    __shared__ uint32_t tmem_base;

    constexpr int KA = NY / 64;                 // 64-row k-chunks of a dz tile
    constexpr uint32_t dzb = NY * 256;          // bytes of one dz tile
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int C = p.C, ds = p.ds, S = p.S, DS = p.DS, KD = p.KD, NS = p.NS, L = p.L, R = p.R;
    const int rank = (int)cluster_rank();
    const int cid = blockIdx.x / C;
    const int col0 = rank * ds;                 // this CTA's hidden-column slice
    const int NB = ds / 64;                     // 64-column boxes of the slice
    const int NG = (NB + 3) / 4;                // accumulation MMAs (N <= 256) per k-chunk
    const int my_tiles = cid < p.tiles ? (p.tiles - 1 - cid) / p.nclus + 1 : 0;
    const int G = my_tiles * NS;                // steps of this cluster
    const uint32_t TM_ACC = 0, TM_Z = (uint32_t)ds;
    int32_t* status = p.status;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&op_full[s], 1);
            mbar_init(&op_empty[s], 1);
        }
        for (int s = 0; s < DS; ++s) {
            mbar_init(&dz_full[s], 1);
            mbar_init(&dz_empty[s], 2);   // the MMA's completion and the signaller
        }
        mbar_init(&zt_full, 1);
        mbar_init(&zt_free, 128);
        mbar_init(&acc_full, 1);
        mbar_init(&acc_free, 128);
        for (int s = 0; s < R; ++s) {
            mbar_init(&epi_done[s], 128);
            mbar_init(&dz_ready[s], C);   // one arrive per writer CTA and step
            mbar_init(&dz_free[s], C);    // one arrive per reader CTA and step
        }
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
    const uint32_t dz_base = base + (uint32_t)S * SLOT;   // dz stages follow the operand stages

    // first ring row of writer q's tile in ring slot `slot`
    auto ring_row = [&](int slot, int q) { return ((cid * R + slot) * C + q) * 128; };

    // The single-thread roles keep every ring position in running counters:
    // integer division by a runtime value on these threads costs more than
    // the tensor work it feeds.
    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            prefetch_tmap(&tmX);
            prefetch_tmap(&tmYz);
            prefetch_tmap(&tmYa);
            prefetch_tmap(&tmD);
            int s = 0, dsl = 0;
            uint32_t ph = 0, dph = 0;
            bool filled = false, dfilled = false;
            int zt = 0, ztile = cid;               // Z stream: step in tile, tile
            int at = 0, aslot = 0;                 // accumulation stream: step in tile, ring slot
            uint32_t aph = 0;
            bool ok = true;
            auto acquire = [&](uint32_t bytes) -> int {
                const int slot = s;
                if (filled && !mbar_wait(&op_empty[slot], ph ^ 1u, status, 601)) return -1;
                mbar_expect_tx(&op_full[slot], bytes);
                if (++s == S) {
                    s = 0;
                    ph ^= 1u;
                    filled = true;
                }
                return slot;
            };
            for (int gt = 0; ok && gt < G + L; ++gt) {
                if (gt < G) {
                    // Z(gt): X k-slice (128 x 64) and this CTA's Y k-slice (NY x 64)
                    const int xr = ztile * 128;
                    const int yr = zt * C * NY + rank * NY;
                    for (int kk = 0; kk < KD; ++kk) {
                        const int slot = acquire(16384u + NY * 128u);
                        if (slot < 0) {
                            ok = false;
                            break;
                        }
                        uint8_t* dst = sm + slot * SLOT;
                        tma_load_2d(dst, &tmX, &op_full[slot], kk * 64, xr);
                        tma_load_2d(dst + 16384, &tmYz, &op_full[slot], kk * 64, yr);
                    }
                    if (!ok) break;
                    if (++zt == NS) {
                        zt = 0;
                        ztile += p.nclus;
                    }
                }
                if (gt >= L) {
                    // Acc(gt - L): the C dz tiles of the step and, for each, the
                    // matching Y rows restricted to this CTA's column slice
                    if (!wait_cluster(&dz_ready[aslot], aph, status, 602)) {
                        ok = false;
                        break;
                    }
                    fence_proxy_async_global();
                    const int yb = at * C * NY;
                    for (int q = 0; ok && q < C; ++q) {
                        if (dfilled && !mbar_wait(&dz_empty[dsl], dph ^ 1u, status, 603)) {
                            ok = false;
                            break;
                        }
                        mbar_expect_tx(&dz_full[dsl], dzb);
                        const int rr = ring_row(aslot, q);
                        for (int kc = 0; kc < KA; ++kc)
                            tma_load_2d(sm + S * SLOT + dsl * dzb + kc * 16384, &tmD, &dz_full[dsl], kc * 64, rr);
                        if (++dsl == DS) {
                            dsl = 0;
                            dph ^= 1u;
                            dfilled = true;
                        }
                        for (int kc = 0; ok && kc < KA; ++kc)
                            for (int g = 0; g < NG; ++g) {
                                const int nb = min(4, NB - 4 * g);
                                const int slot = acquire((uint32_t)nb * 8192u);
                                if (slot < 0) {
                                    ok = false;
                                    break;
                                }
                                for (int j = 0; j < nb; ++j)
                                    tma_load_2d(sm + slot * SLOT + j * 8192, &tmYa, &op_full[slot],
                                                col0 + (4 * g + j) * 64, yb + q * NY + kc * 64);
                            }
                    }
                    if (++at == NS) at = 0;
                    if (++aslot == R) {
                        aslot = 0;
                        aph ^= 1u;
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t iZ = idesc_bf16(128, NY, 0, 0);
            const uint32_t iA0 = idesc_bf16(128, min(4, NB) * 64, 0, 1);
            const uint32_t iA1 = idesc_bf16(128, NB > 4 ? (NB - 4) * 64 : 64, 0, 1);
            // descriptors of byte 0 of the operand ring (K-major / MN-major with
            // 64-row boxes) and of the dz stages; a byte offset b adds b >> 4
            const uint64_t dK0 = sdesc_sw128(base, 16, 1024);
            const uint64_t dM0 = sdesc_sw128(base, 8192, 1024);
            const uint64_t dD0 = sdesc_sw128(dz_base, 16, 1024);
            int s = 0, dsl = 0;
            uint32_t ph = 0, dph = 0;
            int at = 0, an = 0;                    // accumulation stream: step in tile, tiles done
            bool ok = true;
            for (int gt = 0; ok && gt < G + L; ++gt) {
                if (gt < G) {
                    // the epilogue has read Z(gt-1) out of TMEM
                    if (gt >= 1 && !mbar_wait(&zt_free, (uint32_t)(gt - 1) & 1u, status, 611)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    for (int kk = 0; kk < KD; ++kk) {
                        if (!mbar_wait(&op_full[s], ph, status, 612)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint64_t da = dK0 + (uint64_t)((s * SLOT) >> 4), db = da + (16384 >> 4);
#pragma unroll
                        for (int ks = 0; ks < 4; ++ks)
                            mma_ss(tmem + TM_Z, da + 2 * ks, db + 2 * ks, iZ, (kk | ks) != 0);
                        mma_commit(&op_empty[s]);
                        if (++s == S) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
                    if (!ok) break;
                    mma_commit(&zt_full);
                }
                if (gt >= L) {
                    // a new tile overwrites the accumulator: the epilogue has drained it
                    if (at == 0 && an > 0 && !mbar_wait(&acc_free, (uint32_t)(an - 1) & 1u, status, 613)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    for (int q = 0; ok && q < C; ++q) {
                        if (!mbar_wait(&dz_full[dsl], dph, status, 614)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint64_t dzd = dD0 + (uint64_t)((dsl * dzb) >> 4);
                        for (int kc = 0; ok && kc < KA; ++kc)
                            for (int g = 0; g < NG; ++g) {
                                if (!mbar_wait(&op_full[s], ph, status, 615)) {
                                    ok = false;
                                    break;
                                }
                                tc_fence_after();
                                // B: 64 streamed rows (K) x nb 64-column boxes (N), MN-major
                                const uint64_t da = dzd + (uint64_t)(kc * (16384 >> 4));
                                const uint64_t db = dM0 + (uint64_t)((s * SLOT) >> 4);
                                const uint32_t iA = g ? iA1 : iA0;
#pragma unroll
                                for (int ks = 0; ks < 4; ++ks)
                                    mma_ss(tmem + TM_ACC + g * 256, da + 2 * ks, db + 128 * ks, iA,
                                           (at | q | kc | ks) != 0);
                                mma_commit(&op_empty[s]);
                                if (++s == S) {
                                    s = 0;
                                    ph ^= 1u;
                                }
                            }
                        mma_commit(&dz_empty[dsl]);
                        if (++dsl == DS) {
                            dsl = 0;
                            dph ^= 1u;
                        }
                    }
                    if (ok && at == NS - 1) mma_commit(&acc_full);
                    if (++at == NS) {
                        at = 0;
                        ++an;
                    }
                }
            }
        }
    } else if (warp == 2) {
        // ------------------------------------------------------------ signaller
        // remote arrivals, kept off the MMA thread: dz tile of step gt
        // published (to every CTA), dz tiles of step gt - L read (to their writers)
        if (lane == 0) {
            int slot = 0, aslot = 0, dsl = 0;
            uint32_t sph = 0, dph = 0;
            bool ok = true;
            for (int gt = 0; ok && gt < G + L; ++gt) {
                if (gt < G) {
                    if (!mbar_wait(&epi_done[slot], sph, status, 631)) {
                        ok = false;
                        break;
                    }
                    const uint32_t a = smem_u32(&dz_ready[slot]);
                    for (int q = 0; q < C; ++q) arrive_remote(mapa(a, (uint32_t)q));
                    if (++slot == R) {
                        slot = 0;
                        sph ^= 1u;
                    }
                }
                if (gt >= L) {
                    const uint32_t a = smem_u32(&dz_free[aslot]);
                    for (int q = 0; q < C; ++q) {
                        // writer q's tile is in shared memory: q may reuse its ring slot
                        if (!mbar_wait(&dz_full[dsl], dph, status, 632)) {
                            ok = false;
                            break;
                        }
                        arrive_remote(mapa(a, (uint32_t)q));
                        mbar_arrive(&dz_empty[dsl]);
                        if (++dsl == DS) {
                            dsl = 0;
                            dph ^= 1u;
                        }
                    }
                    if (++aslot == R) aslot = 0;
                }
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        // warps 3..6: thread = stationary row rl = TMEM lane
        const int qw = warp & 3;
        const int rl = qw * 32 + lane;
        const int et = threadIdx.x - 96;
        const uint32_t lane_base = tmem + ((uint32_t)(qw * 32) << 16);
        bool ok = true;
        // drain the accumulator of tile `tile` (its `n`-th) into dH / dW
        auto output = [&](int tile, int n) -> bool {
            if (!mbar_wait(&acc_full, (uint32_t)n & 1u, status, 621)) return false;
            tc_fence_after();
            const int srow = tile * 128 + rl;
            const bool valid = p.mode == 0 ? srow < p.M : srow < p.V;
            const int64_t orow = valid ? (p.mode == 0 ? (int64_t)p.rows[srow] : (int64_t)srow) : 0;
            const int64_t d = (int64_t)C * ds;
            for (int c0 = 0; c0 < ds; c0 += 32) {
                uint32_t o[32];
                tmem_ld32(lane_base + TM_ACC + c0, o);
                tmem_wait_ld();
                if (!valid) continue;
                if (p.mode == 0) {
                    __nv_bfloat16* dst = p.dH + orow * d + col0 + c0;
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
                    float* dst = p.dW + orow * d + col0 + c0;
#pragma unroll
                    for (int x = 0; x < 8; ++x)
                        reinterpret_cast<uint4*>(dst)[x] = make_uint4(o[4 * x], o[4 * x + 1], o[4 * x + 2], o[4 * x + 3]);
                }
            }
            tc_fence_before();
            mbar_arrive(&acc_free);
            return true;
        };
        // dz = x ((c == tgt) - 2^(z log2 e - y)) with (x, y, tgt) = (dloss g, lse
        // log2 e, target) of the loss row: per thread in pass 0, per column in
        // pass 1. Padded loss rows carry x = 0; streamed rows past the end are
        // zero-filled by TMA, so their dz contributes nothing.
        float4 rp = make_float4(0.f, 0.f, __int_as_float(-1), 0.f);
        int t = 0, tile = cid, slot = 0, drained = 0;
        int next_drain = NS + L - 1;            // step after which tile `drained` is complete
        for (int gt = 0; ok && gt < G; ++gt) {
            if (p.mode == 0 && t == 0) rp = p.par[tile * 128 + rl];
            const int cb = t * C * NY + rank * NY;   // first streamed row of this CTA's tile
            float4 cpar[NY / 32];                    // pass 1: parameters of columns cb + 32 j + lane
            if (p.mode == 1) {
#pragma unroll
                for (int j = 0; j < NY / 32; ++j) {
                    const int c = cb + 32 * j + lane;
                    cpar[j] = c < p.M_pad ? __ldg(&p.par[c]) : make_float4(0.f, 0.f, __int_as_float(-1), 0.f);
                }
            }
            // every CTA has loaded this ring slot's previous tile (step gt - R)
            if (gt >= R) {
                bool w = true;
                if (lane == 0) w = wait_cluster(&dz_free[slot], (uint32_t)((gt - R) / R) & 1u, status, 622);
                w = __shfl_sync(0xffffffffu, w, 0);
                if (!w) {
                    ok = false;
                    break;
                }
            }
            if (!mbar_wait(&zt_full, (uint32_t)gt & 1u, status, 623)) {
                ok = false;
                break;
            }
            tc_fence_after();
            uint32_t z[NY];
#pragma unroll
            for (int j = 0; j < NY / 32; ++j)
                tmem_ld32(lane_base + TM_Z + 32 * j, *reinterpret_cast<uint32_t(*)[32]>(z + 32 * j));
            tmem_wait_ld();
            tc_fence_before();
            mbar_arrive(&zt_free);   // the MMA may overwrite Z now
            __nv_bfloat16* dst = p.ring + (int64_t)(ring_row(slot, rank) + rl) * NY;
            const int vrow = tile * 128 + rl;        // pass 1: this row's vocabulary entry
            const int tj = __float_as_int(rp.z) - cb;   // pass 0: target column inside the tile
#pragma unroll
            for (int j = 0; j < NY / 32; ++j) {
                uint32_t pk[16];
#pragma unroll
                for (int x = 0; x < 32; x += 2) {
                    float dz[2];
#pragma unroll
                    for (int y = 0; y < 2; ++y) {
                        const int c = 32 * j + x + y;
                        const float zv = __uint_as_float(z[c]);
                        if (p.mode == 0) {
                            const float pr = ex2f_approx(fmaf(zv, LOG2E_B, -rp.y));
                            dz[y] = rp.x * ((c == tj ? 1.f : 0.f) - pr);
                        } else {
                            const float cx = __shfl_sync(0xffffffffu, cpar[j].x, x + y);
                            const float cy = __shfl_sync(0xffffffffu, cpar[j].y, x + y);
                            const int ct = __shfl_sync(0xffffffffu, __float_as_int(cpar[j].z), x + y);
                            const float pr = ex2f_approx(fmaf(zv, LOG2E_B, -cy));
                            dz[y] = cx * ((vrow == ct ? 1.f : 0.f) - pr);
                        }
                    }
                    pk[x / 2] = pack_bf16(dz[0], dz[1]);
                }
                uint4* d4 = reinterpret_cast<uint4*>(dst + 32 * j);
#pragma unroll
                for (int x = 0; x < 4; ++x) d4[x] = make_uint4(pk[4 * x], pk[4 * x + 1], pk[4 * x + 2], pk[4 * x + 3]);
            }
            // publish: the tile is in global memory before any CTA's TMA reads it
            fence_proxy_async_global();
            mbar_arrive(&epi_done[slot]);
            if (++slot == R) slot = 0;
            if (++t == NS) {
                t = 0;
                tile += p.nclus;
            }
            // the last accumulation of a tile is issued after the logits of
            // step (first step of the next tile) + L - 1: drain the tile now
            if (gt == next_drain) {
                if (!output(cid + drained * p.nclus, drained)) {
                    ok = false;
                    break;
                }
                ++drained;
                next_drain += NS;
            }
        }
        for (; ok && drained < my_tiles; ++drained) ok = output(cid + drained * p.nclus, drained);
        // the last R steps' slot-free signals from the readers aim here
        if (et == 0)
            for (int gt = max(0, G - R); ok && gt < G; ++gt)
                if (!wait_cluster(&dz_free[gt % R], (uint32_t)(gt / R) & 1u, status, 625)) ok = false;
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

__global__ void k_lm_bwd_par(int M, int M_pad, const float* __restrict__ g, const float* __restrict__ lse,
                             const int32_t* __restrict__ tg, float dloss, float4* __restrict__ par) {
    const int m = blockIdx.x * blockDim.x + threadIdx.x;
    if (m >= M_pad) return;
    par[m] = m < M ? make_float4(g[m] * dloss, lse[m] * LOG2E_B, __int_as_float(tg[m]), 1.f)
                   : make_float4(0.f, 0.f, __int_as_float(-1), 0.f);
}

struct BwdCfg {
    int C, ds, NY, S, DS, L;
    uint32_t smem;
};

// Smallest cluster whose d-slice leaves TMEM room for a logit tile of at
// least 64 columns (ds + NY <= 512 columns); 128 columns when they fit. The
// operand ring takes what two dz stages leave of the shared memory.
bool choose_cfg(int d, BwdCfg& c) {
    const uint32_t limit = 224 * 1024;
    for (int C : {1, 2, 4, 8}) {
        if (d % C) continue;
        const int ds = d / C;
        if (ds % 64 || ds > 448) continue;
        const int NY = ds + 128 <= 512 ? 128 : 64;
        const int DS = 2;
        const uint32_t dzb = (uint32_t)NY * 256u;
        const int S = std::min<int>(MAX_S, (int)((limit - DS * dzb) / SLOT));
        if (S < 3) continue;
        c = {C, ds, NY, S, DS, 2, (uint32_t)S * SLOT + DS * dzb + 1024};
        return true;
    }
    return false;
}

}  // namespace

bool lm_bwd_tc_supported(int d) {
    BwdCfg c;
    return choose_cfg(d, c);
}

// Scratch of the backward inside the log-prob workspace: the per-row
// parameters and the dz exchange ring.
int64_t lm_bwd_tc_scratch(int M, int d) {
    BwdCfg c;
    if (!choose_cfg(d, c)) return 0;
    const int64_t M_pad = ceil_div(M, 128) * 128;
    return align256(16 * M_pad) + (int64_t)RING_CTAS * MAX_R * 128 * c.NY * 2;
}

mw_status lm_bwd_tc(const void* W, int M, int N, int d, int V, const int32_t* rows, const void* Hg, const int32_t* tg,
                    const float* lse, const float* g, float dloss, void* dH, float* dW, int32_t* status, void* scratch,
                    cudaStream_t s) {
    BwdCfg c;
    if (!choose_cfg(d, c)) return MW_ESHAPE;
    mw_status st = cuda_status(cudaMemsetAsync(dH, 0, (size_t)N * d * 2, s));
    if (st != MW_OK) return st;
    if (M == 0) return cuda_status(cudaMemsetAsync(dW, 0, (size_t)V * d * 4, s));
    const int M_pad = (int)ceil_div(M, 128) * 128;
    float4* par = (float4*)scratch;
    __nv_bfloat16* ring = at<__nv_bfloat16>(scratch, align256(16 * (int64_t)M_pad));
    count_launches(1);
    k_lm_bwd_par<<<(unsigned)ceil_div(M_pad, 256), 256, 0, s>>>(M, M_pad, g, lse, tg, dloss, par);
    if ((st = launch_status()) != MW_OK) return st;

    const int ring_rows = RING_CTAS * MAX_R * 128;
    CUtensorMap hx, hyz, hya, wx, wyz, wya, dm;
    if (!tmap_bf16_2d(&hx, Hg, M_pad, d, d, 128, 64) || !tmap_bf16_2d(&hyz, Hg, M_pad, d, d, c.NY, 64) ||
        !tmap_bf16_2d(&hya, Hg, M_pad, d, d, 64, 64) || !tmap_bf16_2d(&wx, W, V, d, d, 128, 64) ||
        !tmap_bf16_2d(&wyz, W, V, d, d, c.NY, 64) || !tmap_bf16_2d(&wya, W, V, d, d, 64, 64) ||
        !tmap_bf16_2d(&dm, ring, ring_rows, c.NY, c.NY, 128, 64))
        return MW_ECUDA;
    auto kern = c.NY == 128 ? k_lm_bwd_tc<128> : k_lm_bwd_tc<64>;
    if ((st = cuda_status(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)c.smem))) != MW_OK)
        return st;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = c.C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.blockDim = dim3(NT);
    cfg.dynamicSmemBytes = c.smem;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.gridDim = dim3((unsigned)c.C);
    int max_clusters = 0;
    if ((st = cuda_status(cudaOccupancyMaxActiveClusters(&max_clusters, kern, &cfg))) != MW_OK) return st;
    if (max_clusters < 1) return MW_EDEVICE;
    max_clusters = std::min(max_clusters, RING_CTAS / c.C);

    LmBwdParams p;
    p.C = c.C;
    p.ds = c.ds;
    p.S = c.S;
    p.DS = c.DS;
    p.L = c.L;
    p.R = c.L + 1;
    p.KD = d / 64;
    p.M = M;
    p.M_pad = M_pad;
    p.V = V;
    p.rows = rows;
    p.par = par;
    p.dH = (__nv_bfloat16*)dH;
    p.dW = dW;
    p.ring = ring;
    p.status = status;
    for (int mode = 0; mode < 2; ++mode) {
        p.mode = mode;
        p.tiles = mode == 0 ? M_pad / 128 : (int)ceil_div(V, 128);
        p.NS = (int)ceil_div(mode == 0 ? V : M_pad, (int64_t)c.C * c.NY);
        p.nclus = std::min(p.tiles, max_clusters);
        cfg.gridDim = dim3((unsigned)(p.nclus * c.C));
        count_launches(1);
        if ((st = cuda_status(cudaLaunchKernelEx(&cfg, kern, mode == 0 ? hx : wx, mode == 0 ? wyz : hyz,
                                                 mode == 0 ? wya : hya, dm, p))) != MW_OK)
            return st;
    }
    return launch_status();
}

}  // namespace mw
