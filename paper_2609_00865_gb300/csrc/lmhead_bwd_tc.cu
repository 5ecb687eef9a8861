// Tensor-core LM-head passes over the whole vocabulary without materialising
// logits, z = Hg W^T (Hg: the gathered loss rows):
//
//   fused forward (mode 2, loss rows stationary): with a fixed per-row
//     reference r_m (log2 units, the row's largest logit over the first
//     vocabulary entries), p~_{m,v} = 2^(z_{m,v} log2 e - r_m) and
//       l_m = sum_v p~_{m,v},  E_m = sum_v p~_{m,v} W_v,  z_{m,tgt_m},
//     so that lse_m = ln 2 (r_m + log2 l_m) and the softmax-weighted mean
//     of the W rows, E_m / l_m, is ready for the backward;
//   dW pass (mode 1, vocab rows stationary):
//     dz_{m,v} = dloss g_m (1[v = tgt_m] - exp(z_{m,v} - lse_m)),
//     dW_v = sum_m dz_{m,v} Hg_m;
//   dH (elementwise, k_lm_dh_from_e): dH_{rows[m]} = sum_v dz_{m,v} W_v
//     = dloss g_m (W_{tgt_m} - E_m / l_m).
// A logit more than kGuard (log2 units) above its row's reference is
// clamped and flags the row; k_lm_repair then recomputes that row's r, l, E
// and target logit exactly on CUDA cores, so the result never depends on
// how well the reference was chosen, only the speed does.
//
// A pass holds a 128-row tile X of the stationary operand and streams the
// other operand Y. The tile's accumulator over the whole hidden size (128 x d
// fp32) is larger than one SM's tensor memory, so a group of C CTAs shares
// the tile: CTA r accumulates hidden columns [r ds, (r+1) ds), ds = d / C <=
// 256. Step t of the group covers C NY streamed rows (NY = 256); CTA r
//   1. computes the logits of its own NY streamed rows over the full hidden
//      size, Z_r = X Y_{t,r}^T (TMEM; X and Y k-slices streamed by TMA),
//   2. forms dz_r (bf16, 128 x NY) in the epilogue, writes it into its slot
//      of a per-group ring in global memory (R = L + 2 steps deep, tens of
//      MB in all, so it stays in L2) and counts it on the slot's "ready"
//      counter,
//   3. accumulates Acc_r += sum_q dz_q Y_{t,q}[:, slice r] over the C dz
//      tiles of the step (dz k-chunks and Y slices loaded by TMA) and then
//      counts the slot on its "freed" counter.
// Only bf16 dz tiles cross CTAs, once per step. The accumulation of step t
// is issued after the logits of step t + L, so the exchange has L steps of
// tensor work to complete in. The two counters per ring slot live in global
// memory and only grow (release adds, acquire polls): a group is not a
// hardware cluster, so any C co-resident CTAs can form one. The launch is
// cooperative (every CTA resident at once, as the counters' waits require)
// and the groups are persistent, each owning a fixed ring region. Hardware
// clusters of 14 or 16 CTAs fit only 7 at a time (98 or 112 SMs); software
// groups of 14 fill 140 SMs. One ring of 48 KB stages in
// shared memory carries the operands in the order the MMA thread consumes
// them: the k-slices of Z(t) (X 16 KB + Y 32 KB), then the stages of
// Acc(t - L) (a 64-column chunk of one dz tile + the matching 64 Y rows).
//
// Every stage feeds at least 384 cycles of tensor work (N >= 192, K = 64):
// one thread issues about one tcgen05.mma per 60 cycles and pays a few
// hundred cycles per wait/commit, so narrower stages leave the tensor pipe
// idle. Every wait is bounded in time.

#include <math.h>

#include "common.cuh"
#include "tc.cuh"
#include "tmap.cuh"

namespace mw {

namespace {

using namespace tc;

// warp 0 TMA, warp 1 MMA, warp 2 counts published dz tiles, warps 3..6
// epilogue, warp 7 counts consumed ring slots
constexpr int NT = 256;
constexpr int FREE_WARP = 7;
constexpr int NY = 256;              // streamed rows per CTA and step
constexpr int S = 4;                 // operand stages
constexpr uint32_t SLOT = 49152;     // bytes per operand stage
constexpr uint32_t SMEM = S * SLOT + 1024;
constexpr int MAX_R = 4;             // ring depth
constexpr int RING_CTAS = 160;       // ring capacity, in CTAs
constexpr float LOG2E_B = 1.4426950408889634f;
// Largest exponent (log2 units above the row's reference) the fused forward
// accepts: p~ <= 2^96 keeps bf16 p~, the fp32 row sums (<= 2^96 V) and E
// finite with room to spare; a larger one flags the row for k_lm_repair.
constexpr float kGuard = 96.f;

struct LmBwdParams {
    int mode;            // 1: dW pass, 2: fused forward (E, row sums, target logit)
    int add;             // mode 1: add the pass's dW to the array instead of overwriting it
    int C, ds;           // cluster size, d-slice (<= 256)
    int L, R;            // accumulation lag in steps, ring depth R = L + 2
    int KD;              // 64-wide k-slices of d
    int NS;              // steps per tile
    int tiles, nclus;    // stationary tiles, clusters in the grid
    int M, M_pad, V;
    const float4* par;     // [M_pad] per loss row: mode 1 (dloss g, lse log2 e, target bits, -);
                           // mode 2 (-, r, target bits, -)
    float* dW;             // [V, d]
    float* E;              // mode 2: [M_pad, d] sum_v p~ W_v
    float* lpart;          // mode 2: [C][M_pad] row sums of p~ over each group rank's columns
    float* zt;             // mode 2: [M] target logits
    int32_t* flag;         // mode 2: [M_pad] set where a logit exceeded the reference by kGuard
    __nv_bfloat16* ring;   // [nclus][R][C][128][NY] dz exchange ring
    uint32_t* ready;       // [nclus][R] dz tiles published into the slot, all uses
    uint32_t* freed;       // [nclus][R] CTAs done reading the slot, all uses
    int32_t* status;
};

// Counters of the ring slots, in global memory. A group's CTAs are not a
// hardware cluster: they synchronise through gpu-scope release / acquire.
__device__ __forceinline__ void count_release_gpu(uint32_t* ctr) {
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(ctr) : "memory");
}
__device__ __forceinline__ uint32_t load_acquire_gpu(const uint32_t* ctr) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
    return v;
}
// Orders this thread's generic global accesses with the async proxy (TMA).
__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}
// Bounded wait until *ctr >= target; the counters only grow during a launch.
__device__ __forceinline__ bool wait_count(const uint32_t* ctr, uint32_t target, int32_t* status, int where) {
    if (load_acquire_gpu(ctr) >= target) return true;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t i = 1;; ++i) {
        __nanosleep(32);
        if (load_acquire_gpu(ctr) >= target) return true;
        if ((i & 63u) == 0 &&
            ((status && *(volatile int32_t*)&status[1]) || globaltimer_ns() - t0 > kWaitLimitNs))
            break;
    }
    if (status) {
        atomicExch(&status[1], 1);
        atomicCAS(&status[2], 0, where);
    }
    return false;
}

__global__ void __launch_bounds__(NT, 1)
    k_lm_bwd_tc(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmYz,
                const __grid_constant__ CUtensorMap tmYa, const __grid_constant__ CUtensorMap tmD, LmBwdParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t op_full[S], op_empty[S], zt_full, zt_free, acc_full, acc_free, epi_done[MAX_R],
        acc_done[MAX_R];
    __shared__ uint32_t tmem_base;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int C = p.C, ds = p.ds, KD = p.KD, NS = p.NS, L = p.L, R = p.R;
    const int rank = (int)(blockIdx.x % C);
    const int cid = blockIdx.x / C;
    const int col0 = rank * ds;                 // this CTA's hidden-column slice
    const int NB = (ds + 63) / 64;              // 64-column Y boxes covering the slice
    const int my_tiles = cid < p.tiles ? (p.tiles - 1 - cid) / p.nclus + 1 : 0;
    const int G = my_tiles * NS;                // steps of this cluster
    const uint32_t TM_ACC = 0, TM_Z = (uint32_t)ds;
    int32_t* status = p.status;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&op_full[s], 1);
            mbar_init(&op_empty[s], 1);
        }
        mbar_init(&zt_full, 1);
        mbar_init(&zt_free, 128);
        mbar_init(&acc_full, 1);
        mbar_init(&acc_free, 128);
        for (int s = 0; s < R; ++s) {
            mbar_init(&epi_done[s], 128);
            mbar_init(&acc_done[s], 1);   // this CTA's accumulation of the slot's step completed
        }
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&tmem_base, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base;
    const uint32_t base = smem_u32(sm);

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
            int s = 0;
            uint32_t ph = 0;
            bool filled = false;
            int zt = 0, ztile = cid;               // Z stream: step in tile, tile
            int at = 0, aslot = 0;                 // accumulation stream: step in tile, ring slot
            uint32_t ause = 0;                     // earlier uses of ring slot `aslot`
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
                    // Acc(gt - L): for each writer q and 64-row k-chunk, the dz
                    // chunk (128 x 64) and Y rows restricted to this CTA's slice
                    if (!wait_count(&p.ready[cid * R + aslot], (uint32_t)C * (ause + 1u), status, 602)) {
                        ok = false;
                        break;
                    }
                    fence_proxy_async_global();
                    const int yb = at * C * NY;
                    for (int q = 0; ok && q < C; ++q) {
                        const int rr = ring_row(aslot, q);
                        for (int kc = 0; kc < NY / 64; ++kc) {
                            const int slot = acquire(16384u + (uint32_t)NB * 8192u);
                            if (slot < 0) {
                                ok = false;
                                break;
                            }
                            uint8_t* dst = sm + slot * SLOT;
                            tma_load_2d(dst, &tmD, &op_full[slot], kc * 64, rr);
                            for (int j = 0; j < NB; ++j)
                                tma_load_2d(dst + 16384 + j * 8192, &tmYa, &op_full[slot], col0 + j * 64,
                                            yb + q * NY + kc * 64);
                        }
                    }
                    if (++at == NS) at = 0;
                    if (++aslot == R) {
                        aslot = 0;
                        ++ause;
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t iZ = idesc_bf16(128, NY, 0, 0);
            const uint32_t iA = idesc_bf16(128, ds, 0, 1);
            // descriptors of byte 0 of the ring (K-major) and of byte 16384 of
            // the ring (MN-major, 64-row boxes); a byte offset b adds b >> 4
            const uint64_t dK0 = sdesc_sw128(base, 16, 1024);
            const uint64_t dM0 = sdesc_sw128(base + 16384, 8192, 1024);
            int s = 0;
            uint32_t ph = 0;
            int at = 0, an = 0, aslot = 0;         // accumulation stream: step in tile, tiles done, ring slot
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
                        for (int kc = 0; kc < NY / 64; ++kc) {
                            if (!mbar_wait(&op_full[s], ph, status, 615)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                            const uint64_t da = dK0 + (uint64_t)((s * SLOT) >> 4);
                            const uint64_t db = dM0 + (uint64_t)((s * SLOT) >> 4);
#pragma unroll
                            for (int ks = 0; ks < 4; ++ks)
                                mma_ss(tmem + TM_ACC, da + 2 * ks, db + 128 * ks, iA, (at | q | kc | ks) != 0);
                            mma_commit(&op_empty[s]);
                            if (++s == S) {
                                s = 0;
                                ph ^= 1u;
                            }
                        }
                    }
                    // the writers may reuse the slot once these MMAs (and so
                    // the loads of its tiles) have completed
                    if (ok) mma_commit(&acc_done[aslot]);
                    if (ok && at == NS - 1) mma_commit(&acc_full);
                    if (++at == NS) {
                        at = 0;
                        ++an;
                    }
                    if (++aslot == R) aslot = 0;
                }
            }
        }
    } else if (warp == 2 || warp == FREE_WARP) {
        // ------------------------------------------------------------ counters
        // warp 2: this CTA's dz tile of step gt is in the ring (epilogue done);
        // warp FREE_WARP: this CTA's accumulation of step gt has completed
        if (lane == 0) {
            int slot = 0;
            uint32_t sph = 0;
            uint64_t* bars = warp == 2 ? epi_done : acc_done;
            uint32_t* ctr = (warp == 2 ? p.ready : p.freed) + cid * R;
            for (int gt = 0; gt < G; ++gt) {
                if (!mbar_wait(&bars[slot], sph, status, warp == 2 ? 631 : 632)) break;
                __threadfence();
                count_release_gpu(&ctr[slot]);
                if (++slot == R) {
                    slot = 0;
                    sph ^= 1u;
                }
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        // warps 3..6: thread = stationary row rl = TMEM lane
        const int qw = warp & 3;
        const int rl = qw * 32 + lane;
        const uint32_t lane_base = tmem + ((uint32_t)(qw * 32) << 16);
        bool ok = true;
        // drain the accumulator of tile `tile` (its `n`-th) into dW (mode 1) or E (mode 2)
        auto output = [&](int tile, int n) -> bool {
            if (!mbar_wait(&acc_full, (uint32_t)n & 1u, status, 621)) return false;
            tc_fence_after();
            const int srow = tile * 128 + rl;
            const bool valid = p.mode == 1 ? srow < p.V : srow < p.M;
            const int64_t orow = valid ? (int64_t)srow : 0;
            const int64_t d = (int64_t)C * ds;
            for (int c0 = 0; c0 < ds; c0 += 32) {
                uint32_t o[32];
                tmem_ld32(lane_base + TM_ACC + c0, o);
                tmem_wait_ld();
                if (!valid) continue;
                float* dst = (p.mode == 1 ? p.dW : p.E) + orow * d + col0 + c0;
                if (p.add) {
#pragma unroll
                    for (int x = 0; x < 8; ++x) {
                        float4 q = reinterpret_cast<float4*>(dst)[x];
                        q.x += __uint_as_float(o[4 * x]);
                        q.y += __uint_as_float(o[4 * x + 1]);
                        q.z += __uint_as_float(o[4 * x + 2]);
                        q.w += __uint_as_float(o[4 * x + 3]);
                        reinterpret_cast<float4*>(dst)[x] = q;
                    }
                } else {
#pragma unroll
                    for (int x = 0; x < 8; ++x)
                        reinterpret_cast<uint4*>(dst)[x] =
                            make_uint4(o[4 * x], o[4 * x + 1], o[4 * x + 2], o[4 * x + 3]);
                }
            }
            tc_fence_before();
            mbar_arrive(&acc_free);
            return true;
        };
        // mode 1: dz = x ((c == tgt) - 2^(z log2 e - y)) with (x, y, tgt) =
        // (dloss g, lse log2 e, target) of the loss row of each column; padded
        // loss rows carry x = 0. Mode 2: dz = p~ = 2^(z log2 e - r) of this
        // thread's row, 0 past the vocabulary. Streamed rows past the end are
        // zero-filled by TMA, so their dz contributes nothing.
        float4 rp = make_float4(0.f, 0.f, __int_as_float(-1), 0.f);
        float lsum = 0.f, zt_v = 0.f, xmax = -INFINITY;   // mode 2: this row over this CTA's columns
        bool zt_found = false;
        int t = 0, tile = cid, slot = 0, drained = 0;
        uint32_t uses = 0;                      // earlier uses of ring slot `slot`
        int next_drain = NS + L - 1;            // step after which tile `drained` is complete
        for (int gt = 0; ok && gt < G; ++gt) {
            if (p.mode != 1 && t == 0) {
                rp = p.par[tile * 128 + rl];
                lsum = 0.f;
                xmax = -INFINITY;
                zt_found = false;
            }
            const int cb = t * C * NY + rank * NY;   // first streamed row of this CTA's tile
            float4 cpar[NY / 32];                    // pass 1: parameters of columns cb + 32 j + lane
            if (p.mode == 1) {
#pragma unroll
                for (int j = 0; j < NY / 32; ++j) {
                    const int c = cb + 32 * j + lane;
                    cpar[j] = c < p.M_pad ? __ldg(&p.par[c]) : make_float4(0.f, 0.f, __int_as_float(-1), 0.f);
                }
            }
            if (!mbar_wait(&zt_full, (uint32_t)gt & 1u, status, 623)) {
                ok = false;
                break;
            }
            tc_fence_after();
            // every CTA of the group has consumed this ring slot's previous
            // tiles (step gt - R)
            if (gt >= R) {
                bool w = true;
                if (lane == 0) w = wait_count(&p.freed[cid * R + slot], (uint32_t)C * uses, status, 622);
                w = __shfl_sync(0xffffffffu, w, 0);
                if (!w) {
                    ok = false;
                    break;
                }
            }
            __nv_bfloat16* dst = p.ring + (int64_t)(ring_row(slot, rank) + rl) * NY;
            const int vrow = tile * 128 + rl;        // pass 1: this row's vocabulary entry
            const int tj = __float_as_int(rp.z) - cb;   // passes 0, 2: target column inside the tile
            const int nvalid = p.V - cb;                // mode 2: columns inside the vocabulary
#pragma unroll
            for (int j = 0; j < NY / 32; ++j) {
                uint32_t z[32];
                tmem_ld32(lane_base + TM_Z + 32 * j, z);
                tmem_wait_ld();
                if (j == NY / 32 - 1) {
                    tc_fence_before();
                    mbar_arrive(&zt_free);   // the MMA may overwrite Z now
                }
                uint32_t pk[16];
#pragma unroll
                for (int x = 0; x < 32; x += 2) {
                    float dz[2];
#pragma unroll
                    for (int y = 0; y < 2; ++y) {
                        const int c = 32 * j + x + y;
                        const float zv = __uint_as_float(z[x + y]);
                        if (p.mode == 2) {
                            // columns past the vocabulary (zero-filled W rows) get p~ = 0
                            float pr = 0.f;
                            if (c < nvalid) {
                                const float xe = fmaf(zv, LOG2E_B, -rp.y);
                                xmax = fmaxf(xmax, xe);
                                pr = ex2f_approx(fminf(xe, kGuard));
                                lsum += pr;
                            }
                            if (c == tj) {
                                zt_v = zv;
                                zt_found = true;
                            }
                            dz[y] = pr;
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
            if (++slot == R) {
                slot = 0;
                ++uses;
            }
            if (p.mode == 2 && t == NS - 1) {
                // the row has met all of this CTA's columns
                const int m = tile * 128 + rl;
                p.lpart[(int64_t)rank * p.M_pad + m] = lsum;
                if (zt_found && m < p.M) p.zt[m] = zt_v;
                if (xmax > kGuard && m < p.M) p.flag[m] = 1;
            }
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

// Exact recomputation of a flagged row of the fused forward (some logit more
// than kGuard above the row's reference), on CUDA cores: r = the row's largest
// logit over the whole vocabulary (log2 units), l = sum_v 2^(z_v log2 e - r),
// E = sum_v 2^(z_v log2 e - r) W_v, the target logit. A block takes 256
// consecutive rows at a time, reads their flags in one load and then works
// the flagged ones one after another (with none flagged, the usual case, it
// is done after that load); warp w takes vocabulary entries w, w + 8, ...; a
// logit is a warp dot product over d in float32. Both passes form z_v the
// same way, so the weights of pass 2 are consistent with r and l of pass 1.
// A row's results depend on that row alone, so the order of the flagged rows
// within a chunk does not change them.
constexpr int RP_WARPS = 8;
__global__ void __launch_bounds__(RP_WARPS * 32)
    k_lm_repair(int M, int M_pad, int d, int V, int C, const __nv_bfloat16* __restrict__ Hg,
                const __nv_bfloat16* __restrict__ W, const int32_t* __restrict__ tg, const int32_t* __restrict__ flag,
                float4* __restrict__ par, float* __restrict__ lpart, float* __restrict__ zt, float* __restrict__ E) {
    extern __shared__ float rp_smem[];
    float* h = rp_smem;               // [d]
    float* acc = rp_smem + d;         // [RP_WARPS][d]
    __shared__ float wm[RP_WARPS], wl[RP_WARPS];
    __shared__ int flagged[RP_WARPS * 32];
    __shared__ int n_flagged;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nvec = d / 8;           // 16-byte vectors of a row
    for (int c0 = blockIdx.x * blockDim.x; c0 < M; c0 += gridDim.x * blockDim.x) {
        if (threadIdx.x == 0) n_flagged = 0;
        __syncthreads();
        if (c0 + (int)threadIdx.x < M && flag[c0 + threadIdx.x]) flagged[atomicAdd(&n_flagged, 1)] = c0 + threadIdx.x;
        __syncthreads();
        const int nf = n_flagged;
        for (int fi = 0; fi < nf; ++fi) {
            const int m = flagged[fi];    // uniform over the block
            for (int k = threadIdx.x; k < d; k += blockDim.x) h[k] = __bfloat162float(Hg[(int64_t)m * d + k]);
            for (int k = threadIdx.x; k < RP_WARPS * d; k += blockDim.x) acc[k] = 0.f;
            __syncthreads();
            auto logit = [&](int v) -> float {
                const uint4* wr = reinterpret_cast<const uint4*>(W + (int64_t)v * d);
                float a = 0.f;
                for (int k = lane; k < nvec; k += 32) {
                    const uint4 u = __ldg(&wr[k]);
                    const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
    #pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        a = fmaf(__uint_as_float(w4[e] << 16), h[8 * k + 2 * e], a);
                        a = fmaf(__uint_as_float(w4[e] & 0xffff0000u), h[8 * k + 2 * e + 1], a);
                    }
                }
                return warp_sum(a);
            };
            const int t = tg[m];
            // pass 1: online (max, sum) per warp, log2 units
            float mx = -INFINITY, l = 0.f;
            for (int v = warp; v < V; v += RP_WARPS) {
                const float z = logit(v);
                if (v == t && lane == 0) zt[m] = z;
                const float x = z * LOG2E_B;
                if (x > mx) {
                    l = l * exp2f(mx - x) + 1.f;
                    mx = x;
                } else {
                    l += exp2f(x - mx);
                }
            }
            if (lane == 0) {
                wm[warp] = mx;
                wl[warp] = l;
            }
            __syncthreads();
            float r = -INFINITY;
            for (int w = 0; w < RP_WARPS; ++w) r = fmaxf(r, wm[w]);
            float lt = 0.f;
            for (int w = 0; w < RP_WARPS; ++w) lt += wl[w] > 0.f ? wl[w] * exp2f(wm[w] - r) : 0.f;
            // pass 2: E = sum_v 2^(z_v log2 e - r) W_v, per warp into its own row of acc
            float* aw = acc + warp * d;
            for (int v = warp; v < V; v += RP_WARPS) {
                const float pv = exp2f(logit(v) * LOG2E_B - r);
                const uint4* wr = reinterpret_cast<const uint4*>(W + (int64_t)v * d);
                for (int k = lane; k < nvec; k += 32) {
                    const uint4 u = __ldg(&wr[k]);
                    const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
    #pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        aw[8 * k + 2 * e] = fmaf(pv, __uint_as_float(w4[e] << 16), aw[8 * k + 2 * e]);
                        aw[8 * k + 2 * e + 1] = fmaf(pv, __uint_as_float(w4[e] & 0xffff0000u), aw[8 * k + 2 * e + 1]);
                    }
                }
            }
            __syncthreads();
            for (int k = threadIdx.x; k < d; k += blockDim.x) {
                float e = 0.f;
                for (int w = 0; w < RP_WARPS; ++w) e += acc[w * d + k];
                E[(int64_t)m * d + k] = e;
            }
            if (threadIdx.x == 0) {
                float4 q = par[m];
                q.y = r;
                par[m] = q;
                lpart[m] = lt;
                for (int c = 1; c < C; ++c) lpart[(int64_t)c * M_pad + m] = 0.f;
            }
            __syncthreads();
        }
        __syncthreads();   // every thread has read n_flagged before the next chunk resets it
    }
}

// lse = ln 2 (r + log2 sum_c lpart_c), lp = z_target - lse, 1 / l for the dH.
__global__ void k_lm_grp_combine(int M, int M_pad, int C, const float4* __restrict__ par,
                                 const float* __restrict__ lpart, const float* __restrict__ zt,
                                 float* __restrict__ lse, float* __restrict__ lp, float* __restrict__ linv) {
    const int m = blockIdx.x * blockDim.x + threadIdx.x;
    if (m >= M) return;
    float l = 0.f;
    for (int c = 0; c < C; ++c) l += lpart[(int64_t)c * M_pad + m];
    const float v = (par[m].y + log2f(l)) * 0.6931471805599453f;
    lse[m] = v;
    lp[m] = zt[m] - v;
    linv[m] = 1.f / l;
}

// dH_{rows[m]} = dloss g_m (W_{tgt_m} - E_m / l_m), bf16; one block per loss
// row (grid-stride), 16-byte vectors along d. Rows outside the loss stay 0,
// and so does a row outside [0, N) or without a valid target (the forward's
// gather gave it target -1; bounds flag).
__global__ void k_lm_dh_from_e(int M, int d, int N, const __nv_bfloat16* __restrict__ W,
                               const int32_t* __restrict__ tg, const float* __restrict__ E,
                               const float* __restrict__ linv, const float* __restrict__ g, float dloss,
                               const int32_t* __restrict__ rows, __nv_bfloat16* __restrict__ dH,
                               int32_t* __restrict__ status) {
    const int nvec = d / 8;
    for (int m = blockIdx.x; m < M; m += gridDim.x) {
        const int r = checked_index(rows[m], N), t = tg[m];
        if (r < 0 || t < 0) {   // uniform over the block
            if (threadIdx.x == 0) flag_bounds(status);
            continue;
        }
        const float a = dloss * g[m], il = linv[m];
        const uint4* wr = reinterpret_cast<const uint4*>(W + (int64_t)t * d);
        const float4* er = reinterpret_cast<const float4*>(E + (int64_t)m * d);
        uint4* out = reinterpret_cast<uint4*>(dH + (int64_t)r * d);
        for (int k = threadIdx.x; k < nvec; k += blockDim.x) {
            const uint4 u = __ldg(&wr[k]);
            const float4 e0 = er[2 * k], e1 = er[2 * k + 1];
            const float ev[8] = {e0.x, e0.y, e0.z, e0.w, e1.x, e1.y, e1.z, e1.w};
            const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
            uint32_t o[4];
#pragma unroll
            for (int x = 0; x < 4; ++x) {
                const float lo = a * (__uint_as_float(w4[x] << 16) - ev[2 * x] * il);
                const float hi = a * (__uint_as_float(w4[x] & 0xffff0000u) - ev[2 * x + 1] * il);
                o[x] = pack_bf16(lo, hi);
            }
            out[k] = make_uint4(o[0], o[1], o[2], o[3]);
        }
    }
}

// SDCC's forward KL from the fused passes of the teacher and the student
// rows of each pair (E_T, E_S: sum_v p~ W_v; linv: 1 / l). With z = h W^T,
// E_{p_T}[z_T - z_S] = (h_T - h_S) . Ebar_T, Ebar_T = E_T / l_T, so
//   KL(p_T || p_S) = (h_T - h_S) . Ebar_T - lse_T + lse_S.
// One warp per pair, float32 over d.
__global__ void k_kl_from_e(int M, int d, const __nv_bfloat16* __restrict__ hgT, const __nv_bfloat16* __restrict__ hgS,
                            const float* __restrict__ ET, const float* __restrict__ linvT,
                            const float* __restrict__ lseT, const float* __restrict__ lseS, float* __restrict__ kl) {
    const int m = (int)((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    if (m >= M) return;
    const uint4* t8 = reinterpret_cast<const uint4*>(hgT + (int64_t)m * d);
    const uint4* s8 = reinterpret_cast<const uint4*>(hgS + (int64_t)m * d);
    const float4* e4 = reinterpret_cast<const float4*>(ET + (int64_t)m * d);
    float a = 0.f;
    for (int k = lane; k < d / 8; k += 32) {
        const uint4 ut = t8[k], us = s8[k];
        const float4 e0 = e4[2 * k], e1 = e4[2 * k + 1];
        const uint32_t tw[4] = {ut.x, ut.y, ut.z, ut.w}, sw[4] = {us.x, us.y, us.z, us.w};
        const float ev[8] = {e0.x, e0.y, e0.z, e0.w, e1.x, e1.y, e1.z, e1.w};
#pragma unroll
        for (int x = 0; x < 4; ++x) {
            a = fmaf(__uint_as_float(tw[x] << 16) - __uint_as_float(sw[x] << 16), ev[2 * x], a);
            a = fmaf(__uint_as_float(tw[x] & 0xffff0000u) - __uint_as_float(sw[x] & 0xffff0000u), ev[2 * x + 1], a);
        }
    }
    a = warp_sum(a);
    if (lane == 0) kl[m] = a * linvT[m] - lseT[m] + lseS[m];
}

// dH_S of the KL: c (Ebar_S - Ebar_T) at the student row of each pair (bf16).
// Both products are rounded before the difference (no fused multiply-add), so
// a student equal to its teacher gets exactly 0.
__global__ void k_kl_dh_from_e(int M, int d, int N_S, const float* __restrict__ ES, const float* __restrict__ linvS,
                               const float* __restrict__ ET, const float* __restrict__ linvT, float c,
                               const int32_t* __restrict__ rowsS, int accumulate, __nv_bfloat16* __restrict__ dHS,
                               int32_t* __restrict__ status) {
    for (int m = blockIdx.x; m < M; m += gridDim.x) {
        const int r = checked_index(rowsS[m], N_S);
        if (r < 0) {   // uniform over the block
            if (threadIdx.x == 0) flag_bounds(status);
            continue;
        }
        const float as = c * linvS[m], at_ = c * linvT[m];
        const float4* s4 = reinterpret_cast<const float4*>(ES + (int64_t)m * d);
        const float4* t4 = reinterpret_cast<const float4*>(ET + (int64_t)m * d);
        uint2* out = reinterpret_cast<uint2*>(dHS + (int64_t)r * d);
        for (int k = threadIdx.x; k < d / 4; k += blockDim.x) {
            const float4 x = s4[k], y = t4[k];
            float g[4] = {__fmul_rn(as, x.x) - __fmul_rn(at_, y.x), __fmul_rn(as, x.y) - __fmul_rn(at_, y.y),
                          __fmul_rn(as, x.z) - __fmul_rn(at_, y.z), __fmul_rn(as, x.w) - __fmul_rn(at_, y.w)};
            if (accumulate) {
                const uint2 o = out[k];
                g[0] += __uint_as_float(o.x << 16);
                g[1] += __uint_as_float(o.x & 0xffff0000u);
                g[2] += __uint_as_float(o.y << 16);
                g[3] += __uint_as_float(o.y & 0xffff0000u);
            }
            out[k] = make_uint2(pack_bf16(g[0], g[1]), pack_bf16(g[2], g[3]));
        }
    }
}

// Per-pair parameters of a softmax-only dW pass: dz_v = -x p_v (no target).
__global__ void k_kl_par(int M, int M_pad, float x, const float* __restrict__ lse, float4* __restrict__ par) {
    const int m = blockIdx.x * blockDim.x + threadIdx.x;
    if (m >= M_pad) return;
    par[m] = m < M ? make_float4(x, lse[m] * LOG2E_B, __int_as_float(-1), 1.f)
                   : make_float4(0.f, 0.f, __int_as_float(-1), 0.f);
}

// Group sizes whose d-slice fits beside a 256-column logit tile in TMEM
// (ds <= 256) and keeps 32-column output chunks (ds % 32 == 0).
bool slice_ok(int d, int C) { return d % C == 0 && d / C <= 256 && (d / C) % 32 == 0; }
constexpr int kGroupSizes[] = {1, 2, 3, 4, 5, 6, 7, 8, 10, 12, 14, 16};
constexpr int kMaxGroup = 16;
constexpr int64_t kCounterBytes = 2 * RING_CTAS * MAX_R * 4;   // ready, freed

// The fewest CTAs per group (the widest slice): a CTA's tensor work per
// step is 2 * 128 * NY * d FLOP for any C, but its dz chunk loads, stages
// and waits per step grow with C (d = 3584 measured: C = 14, 140 CTAs,
// 114 ms; C = 16, 144 CTAs, 127 ms; d = 1536: C = 6 beats C = 8 and 12).
int group_size(int d) {
    for (int c : kGroupSizes)
        if (slice_ok(d, c)) return c;
    return 0;
}

// One launch of k_lm_bwd_tc in `mode` over M loss rows; the scratch holds the
// per-row parameters (filled by the caller), the ring and its counters. Mode
// 1 forms the logits from the rows Hg and takes the dW product with the rows
// HgA (the same rows unless the caller passes others).
mw_status launch_group(LmBwdParams p, const void* W, int d, const void* Hg, void* scratch, cudaStream_t s,
                       const void* HgA = nullptr) {
    if (!HgA) HgA = Hg;
    const int M = p.M, V = p.V;
    const int M_pad = (int)ceil_div(M, 128) * 128;
    __nv_bfloat16* ring = at<__nv_bfloat16>(scratch, align256(16 * (int64_t)M_pad));
    uint32_t* counters = at<uint32_t>(ring, (int64_t)RING_CTAS * MAX_R * 128 * NY * 2);
    mw_status st = cuda_status(cudaMemsetAsync(counters, 0, kCounterBytes, s));
    if (st != MW_OK) return st;
    if ((st = cuda_status(cudaFuncSetAttribute(k_lm_bwd_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)SMEM))) != MW_OK)
        return st;
    // The CTAs of a group wait on one another's counters, so every CTA must be
    // resident at once: the launch is cooperative (it fails rather than run
    // CTAs in waves) and the grid never exceeds what fits.
    int dev = 0, sms = 0, per_sm = 0;
    if ((st = cuda_status(cudaGetDevice(&dev))) != MW_OK ||
        (st = cuda_status(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev))) != MW_OK ||
        (st = cuda_status(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_lm_bwd_tc, NT, SMEM))) != MW_OK)
        return st;
    const int resident = std::min(per_sm * sms, RING_CTAS);
    const int C = group_size(d);
    const int max_groups = C > 0 ? resident / C : 0;
    if (max_groups == 0) return MW_EDEVICE;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.blockDim = dim3(NT);
    cfg.dynamicSmemBytes = SMEM;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;

    const int ring_rows = RING_CTAS * MAX_R * 128;
    const bool rows_x = p.mode != 1;   // loss rows stationary
    CUtensorMap tx, tyz, tya, dm;
    const bool ok = rows_x ? (tmap_bf16_2d(&tx, Hg, M_pad, d, d, 128, 64) && tmap_bf16_2d(&tyz, W, V, d, d, NY, 64) &&
                              tmap_bf16_2d(&tya, W, V, d, d, 64, 64))
                           : (tmap_bf16_2d(&tx, W, V, d, d, 128, 64) && tmap_bf16_2d(&tyz, Hg, M_pad, d, d, NY, 64) &&
                              tmap_bf16_2d(&tya, HgA, M_pad, d, d, 64, 64));
    if (!ok || !tmap_bf16_2d(&dm, ring, ring_rows, NY, NY, 128, 64)) return MW_ECUDA;

    p.C = C;
    p.ds = d / C;
    p.L = 2;
    p.R = p.L + 2;
    p.KD = d / 64;
    p.M_pad = M_pad;
    p.par = (const float4*)scratch;
    p.ring = ring;
    p.ready = counters;
    p.freed = counters + RING_CTAS * MAX_R;
    p.tiles = rows_x ? M_pad / 128 : (int)ceil_div(V, 128);
    p.NS = (int)ceil_div(rows_x ? V : M_pad, (int64_t)C * NY);
    p.nclus = std::min(p.tiles, max_groups);
    cfg.gridDim = dim3((unsigned)(p.nclus * C));
    count_launches(1);
    if ((st = cuda_status(cudaLaunchKernelEx(&cfg, k_lm_bwd_tc, tx, tyz, tya, dm, p))) != MW_OK) return st;
    return launch_status();
}

}  // namespace

bool lm_bwd_tc_supported(int d) {
    if (d % 64) return false;
    return group_size(d) > 0;
}

// Scratch of the group passes inside the log-prob workspace: the per-row
// parameters, the dz exchange ring and the ring slots' counters.
int64_t lm_bwd_tc_scratch(int M, int d) {
    if (!lm_bwd_tc_supported(d)) return 0;
    const int64_t M_pad = ceil_div(M, 128) * 128;
    return align256(16 * M_pad) + (int64_t)RING_CTAS * MAX_R * 128 * NY * 2 + kCounterBytes;
}

// Fused-forward arrays inside the log-prob workspace, after the scratch:
// E [M_pad, d] fp32, lpart [kMaxGroup][M_pad], linv [M_pad], flag [M_pad].
int64_t lm_fwd_grp_bytes(int M, int d) {
    if (!lm_bwd_tc_supported(d)) return 0;
    const int64_t M_pad = ceil_div(M, 128) * 128;
    return align256(4 * M_pad * d) + align256(4 * kMaxGroup * M_pad) + 2 * align256(4 * M_pad);
}

struct GrpArrays {
    float *E, *lpart, *linv;
    int32_t* flag;
};
static GrpArrays grp_arrays(void* fwd, int M, int d) {
    const int64_t M_pad = ceil_div(M, 128) * 128;
    GrpArrays a;
    a.E = (float*)fwd;
    a.lpart = at<float>(a.E, align256(4 * M_pad * d));
    a.linv = at<float>(a.lpart, align256(4 * kMaxGroup * M_pad));
    a.flag = at<int32_t>(a.linv, align256(4 * M_pad));
    return a;
}

// Fused forward over the whole vocabulary: the gathered rows Hg / tg and the
// references in the scratch's parameter array (k_lm_ref) are in place. Writes
// lse, lp (per loss row), zt, and keeps E and 1 / l for the backward.
mw_status lm_fwd_grp_tc(const void* W, int M, int d, int V, const void* Hg, const int32_t* tg, float* zt, float* lse,
                        float* lp, int32_t* status, void* scratch, void* fwd, cudaStream_t s) {
    if (!lm_bwd_tc_supported(d)) return MW_ESHAPE;
    if (M == 0) return MW_OK;
    const int M_pad = (int)ceil_div(M, 128) * 128;
    GrpArrays a = grp_arrays(fwd, M, d);
    mw_status st = cuda_status(cudaMemsetAsync(a.flag, 0, 4 * (size_t)M_pad, s));
    if (st != MW_OK) return st;
    LmBwdParams p = {};
    p.mode = 2;
    p.M = M;
    p.V = V;
    p.E = a.E;
    p.lpart = a.lpart;
    p.zt = zt;
    p.flag = a.flag;
    p.status = status;
    if ((st = launch_group(p, W, d, Hg, scratch, s)) != MW_OK) return st;
    const size_t rp_smem = (size_t)(RP_WARPS + 1) * d * 4;
    if ((st = cuda_status(cudaFuncSetAttribute(k_lm_repair, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)rp_smem))) != MW_OK)
        return st;
    const int C = group_size(d);
    count_launches(2);
    k_lm_repair<<<(unsigned)std::min<int64_t>(ceil_div(M, RP_WARPS * 32), 4 * 152), RP_WARPS * 32, rp_smem, s>>>(
        M, M_pad, d, V, C, (const __nv_bfloat16*)Hg, (const __nv_bfloat16*)W, tg, a.flag, (float4*)scratch, a.lpart,
        zt, a.E);
    k_lm_grp_combine<<<(unsigned)ceil_div(M, 256), 256, 0, s>>>(M, M_pad, C, (const float4*)scratch, a.lpart, zt,
                                                                lse, lp, a.linv);
    return launch_status();
}

// Backward: dW by the vocabulary-stationary pass, dH from the forward's E.
mw_status lm_bwd_tc(const void* W, int M, int N, int d, int V, const int32_t* rows, const void* Hg, const int32_t* tg,
                    const float* lse, const float* g, float dloss, void* dH, float* dW, int32_t* status, void* scratch,
                    void* fwd, cudaStream_t s) {
    if (!lm_bwd_tc_supported(d)) return MW_ESHAPE;
    mw_status st = cuda_status(cudaMemsetAsync(dH, 0, (size_t)N * d * 2, s));
    if (st != MW_OK) return st;
    if (M == 0) return cuda_status(cudaMemsetAsync(dW, 0, (size_t)V * d * 4, s));
    const int M_pad = (int)ceil_div(M, 128) * 128;
    count_launches(1);
    k_lm_bwd_par<<<(unsigned)ceil_div(M_pad, 256), 256, 0, s>>>(M, M_pad, g, lse, tg, dloss, (float4*)scratch);
    if ((st = launch_status()) != MW_OK) return st;
    LmBwdParams p = {};
    p.mode = 1;
    p.M = M;
    p.V = V;
    p.dW = dW;
    p.status = status;
    if ((st = launch_group(p, W, d, Hg, scratch, s)) != MW_OK) return st;
    GrpArrays a = grp_arrays(fwd, M, d);
    count_launches(1);
    k_lm_dh_from_e<<<(unsigned)std::min(M, 8 * 152), 128, 0, s>>>(
        M, d, N, (const __nv_bfloat16*)W, tg, a.E, a.linv, g, dloss, rows, (__nv_bfloat16*)dH, status);
    return launch_status();
}

// SDCC's forward KL on the tensor cores (§5, Eq. "soft_loss"). Workspace:
// gathered teacher and student rows, the reference prepass's partials,
// dummy targets / target logits / log-probs, lse of both, status words, the
// group passes' scratch and the two fused forwards' arrays (E, 1 / l).
struct KlWs {
    int64_t hgT, hgS, tg, part, zt, lp, lseT, lseS, status, scratch, fwdT, fwdS, bytes;
};
static KlWs kl_ws_layout(int M, int d) {
    KlWs w;
    const int64_t M_pad = ceil_div(M, 128) * 128;
    int64_t o = 0;
    auto take = [&](int64_t b) { int64_t r = o; o = align256(o + b); return r; };
    w.hgT = take(2 * M_pad * d);
    w.hgS = take(2 * M_pad * d);
    w.tg = take(4 * M_pad);
    w.part = take(8 * 64 * M_pad);
    w.zt = take(4 * M_pad);
    w.lp = take(4 * M_pad);
    w.lseT = take(4 * M_pad);
    w.lseS = take(4 * M_pad);
    w.status = take(32);
    w.scratch = take(lm_bwd_tc_scratch(M, d));
    w.fwdT = take(lm_fwd_grp_bytes(M, d));
    w.fwdS = take(lm_fwd_grp_bytes(M, d));
    w.bytes = o;
    return w;
}

int64_t kl_tc_ws(int M, int d) { return lm_bwd_tc_supported(d) ? kl_ws_layout(M, d).bytes : 0; }

mw_status lm_ref_tc(const void*, const void*, const int32_t*, const int32_t*, int, int, int, int, void*, int32_t*,
                    float2*, float*, float4*, int32_t*, cudaStream_t);

// Forward: for the teacher rows and then the student rows, the reference
// prepass and the fused pass (lse, E, 1 / l); then KL per pair.
mw_status kl_fwd_tc(const void* HT, const int32_t* rowsT, const void* HS, const int32_t* rowsS, int M, const void* W,
                    int N_T, int N_S, int d, int V, float* kl, void* ws, cudaStream_t s) {
    if (!lm_bwd_tc_supported(d)) return MW_ESHAPE;
    const KlWs w = kl_ws_layout(M, d);
    mw_status st = cuda_status(cudaMemsetAsync(at<char>(ws, w.status), 0, 32, s));
    if (st == MW_OK) st = cuda_status(cudaMemsetAsync(at<char>(ws, w.zt), 0, 4 * (size_t)M, s));
    for (int side = 0; st == MW_OK && side < 2; ++side) {
        const void* H = side == 0 ? HT : HS;
        const int32_t* rows = side == 0 ? rowsT : rowsS;
        void* hg = at<char>(ws, side == 0 ? w.hgT : w.hgS);
        st = lm_ref_tc(H, W, nullptr, rows, M, side == 0 ? N_T : N_S, d, V, hg, at<int32_t>(ws, w.tg),
                       at<float2>(ws, w.part), at<float>(ws, w.zt), at<float4>(ws, w.scratch),
                       at<int32_t>(ws, w.status), s);
        if (st == MW_OK)
            st = lm_fwd_grp_tc(W, M, d, V, hg, at<int32_t>(ws, w.tg), at<float>(ws, w.zt),
                               at<float>(ws, side == 0 ? w.lseT : w.lseS), at<float>(ws, w.lp),
                               at<int32_t>(ws, w.status), at<char>(ws, w.scratch),
                               at<char>(ws, side == 0 ? w.fwdT : w.fwdS), s);
    }
    if (st != MW_OK) return st;
    const GrpArrays aT = grp_arrays(at<char>(ws, w.fwdT), M, d);
    count_launches(1);
    k_kl_from_e<<<(unsigned)ceil_div((int64_t)M * 32, 256), 256, 0, s>>>(
        M, d, at<__nv_bfloat16>(ws, w.hgT), at<__nv_bfloat16>(ws, w.hgS), aT.E, aT.linv, at<float>(ws, w.lseT),
        at<float>(ws, w.lseS), kl);
    return launch_status();
}

// Backward (teacher stopped), c = lam dloss: dH_S = c (Ebar_S - Ebar_T) at
// the student rows; dW = c sum_m (p_S - p_T) h_S as two dW passes over the
// same rows' product: softmax-only with the student's logits, then with the
// teacher's logits added in.
mw_status kl_bwd_tc(const int32_t* rowsS, int M, const void* W, int N_S, int d, int V, float c, void* ws,
                    int accumulate, void* dHS, float* dW, cudaStream_t s) {
    if (!lm_bwd_tc_supported(d)) return MW_ESHAPE;
    mw_status st = MW_OK;
    if (!accumulate && (st = cuda_status(cudaMemsetAsync(dHS, 0, (size_t)N_S * d * 2, s))) != MW_OK) return st;
    if (M == 0) return accumulate ? MW_OK : cuda_status(cudaMemsetAsync(dW, 0, (size_t)V * d * 4, s));
    const KlWs w = kl_ws_layout(M, d);
    const int M_pad = (int)ceil_div(M, 128) * 128;
    const GrpArrays aT = grp_arrays(at<char>(ws, w.fwdT), M, d), aS = grp_arrays(at<char>(ws, w.fwdS), M, d);
    count_launches(1);
    k_kl_dh_from_e<<<(unsigned)std::min(M, 8 * 152), 128, 0, s>>>(M, d, N_S, aS.E, aS.linv, aT.E, aT.linv, c, rowsS,
                                                                  accumulate, (__nv_bfloat16*)dHS,
                                                                  at<int32_t>(ws, w.status));
    if ((st = launch_status()) != MW_OK) return st;
    for (int side = 0; side < 2; ++side) {   // student: dz = c p_S; teacher: dz = -c p_T
        count_launches(1);
        k_kl_par<<<(unsigned)ceil_div(M_pad, 256), 256, 0, s>>>(M, M_pad, side == 0 ? -c : c,
                                                                at<float>(ws, side == 0 ? w.lseS : w.lseT),
                                                                at<float4>(ws, w.scratch));
        if ((st = launch_status()) != MW_OK) return st;
        LmBwdParams p = {};
        p.mode = 1;
        p.add = accumulate || side;
        p.M = M;
        p.V = V;
        p.dW = dW;
        p.status = at<int32_t>(ws, w.status);
        if ((st = launch_group(p, W, d, at<char>(ws, side == 0 ? w.hgS : w.hgT), at<char>(ws, w.scratch), s,
                               at<char>(ws, w.hgS))) != MW_OK)
            return st;
    }
    return MW_OK;
}

int32_t* kl_tc_status(int M, int d, void* ws) { return at<int32_t>(ws, kl_ws_layout(M, d).status); }

}  // namespace mw
