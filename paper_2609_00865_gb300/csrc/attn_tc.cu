// Tensor-core masked GQA attention, bf16 in / fp32 accumulate, head dim 128.
//
// Each segment's rows are scored against the segment's compact sequence: its
// live view gathered in order (§4.1's materialised branch; the visibility
// build's csrc / cpos / seg_len), so a row's visible keys are the prefix of
// that sequence up to its own index -- the 4D-masked computation (§4.2 mask,
// §4.3 Theorem "materialization equivalence") with every visible key read
// once per row and the evicted keys inside a physical tile costing nothing.
// Row i of segment s has compact index nb_s + (i - J_s), nb_s being the keys
// of view_s before the segment's rows. For rotary positions the keys are
// gathered already turned to their rank (their logical position in view_s)
// and the dK partials turned back as they are summed.
//
// q-tile kernels (forward, dQ): one CTA per (q-tile, query head) serving the
// segment of the tile's first row, heaviest q-tiles first, plus a second
// launch ("junction items") with one CTA per (segment starting inside a
// tile, head); a CTA stores only its own segment's rows. It walks compact key
// tiles 0 .. (last row's index) / 128: FULL when it covers the whole q-tile
// and every row reaches the tile's last key, otherwise PARTIAL with a
// per-row prefix mask, DEAD_HI when no row reaches the tile's second half.
//
// Forward kernel:
//   warp 0      TMA producer: Q once, then K_j / V_j of each compact tile
//               (2-stage rings, 128-byte swizzle)
//   warp 1      TMEM allocator + single-thread tcgen05.mma issuer:
//               S_j = Q K_j^T into one of two TMEM S buffers
//   warps 2..5  softmax / epilogue, one query row per thread: online softmax
//               in the exp2 domain with lazy rescaling of O (only when the
//               running max grows by more than 2^8), P written as bf16 over
//               its own S buffer, O / l and the log-sum-exp written at the end
//   warp 6      O += P_{j} V_{j} once the softmax has written P_{j}
//
// dK / dV kernel: one CTA per (compact key tile, segment, KV head) over the
// run of q-tiles whose rows see its keys, writing float32 partials per
// compact row; k_cmp_reduce sums each key's partials over the segments
// holding it, in segment order (deterministic, no atomics).
//
// All waits are bounded (tc::mbar_wait); a timeout ends the CTA and is
// reported through the visibility status word.

#include <math.h>

#include <type_traits>

#include "common.cuh"
#include "tc.cuh"
#include "tmap.cuh"

namespace mw {
namespace {

using namespace tc;

constexpr int DH = 128;
constexpr uint32_t TILE_B = 128 * DH * 2;  // one 128 x 128 bf16 tile: two [128][64] swizzled halves
constexpr uint32_t HALF_B = TILE_B / 2;
// Each kernel issues its tensor-core work from two threads in two warps: one
// thread issues about one tcgen05.mma per 57-114 cycles, and a 128 x 128 x 16
// MMA is only 64 cycles of work, so a single issuer leaves the tensor pipe idle
// (measured: two issuing warps double the issue rate, reaching the MMA's own rate
// at N = 128). The two streams are independent except through the barriers.
// Forward: warp 0 TMA, warp 1 S = Q K^T, warps 2..5 softmax (one row per thread),
// warp 6 O += P V.
constexpr int NT_FWD = 224;
constexpr int FWD_PV_WARP = 6;
// Backward kernels: warp 0 TMA, warp 1 the recomputed products, warps 2..9
// elementwise, warp 10 the gradient accumulation. Two elementwise warps per TMEM
// lane quarter split each row's columns, which hides the latency of the exp /
// scale / pack chains that bound the kernels with one warp per quarter. The two
// MMA warps issue warp-converged (tc::mma_*_w: the whole warp runs the loop, one
// elected lane issues), which cuts the issue cost of their many N = 64 / N = 128
// products; the forward keeps single-lane issue, measured faster there.
constexpr int NT_BWD = 352;
constexpr int BWD_ACC_WARP = 10;
constexpr int NEW = 256;   // elementwise threads
constexpr float LOG2E = 1.4426950408889634f;
constexpr float RESCALE_T = 8.0f;          // lazy-rescale threshold (log2 units)

// dynamic shared memory map (bytes from the 1024-aligned base)
constexpr uint32_t SM_Q = 0;
constexpr uint32_t SM_K = SM_Q + TILE_B;
constexpr uint32_t SM_V = SM_K + 2 * TILE_B;
constexpr uint32_t SM_TOTAL = SM_V + 2 * TILE_B;   // P lives in TMEM
constexpr uint32_t SMEM_FWD = SM_TOTAL + 1024;

// TMEM columns
constexpr uint32_t TM_S0 = 0, TM_O = 256;

struct FwdParams {
    VisView v;
    int64_t total;
    int n_traj, max_tiles, Hq, Hkv;
    float scale_log2;
    __nv_bfloat16* O;
    float* LSE;
    int junction_items;   // 0 = main launch, 1 = one CTA per (segment starting inside a tile, head)
};

// Work item of a q-tile kernel: trajectory b, local q-tile qt, query head h
// and the segment s whose rows the CTA stores. Main launch: one trajectory
// after another, its heaviest (largest) q-tiles first, query heads of one KV
// group adjacent; s = segment of the tile's first row. Taking trajectories in
// turn keeps the resident CTAs on one trajectory's compact K / V, whose
// working set then stays in L2. Junction items: blockIdx.x / Hq is a global
// segment index; a segment that starts inside a tile (not at its first row)
// gets a CTA there.
struct QItem {
    int b, qt, h, s;
    bool ok;
};
__device__ __forceinline__ QItem q_item(const VisView& v, int Hq, int max_tiles, int n_traj, int junction_items) {
    QItem it;
    it.h = blockIdx.x % Hq;
    const int r = blockIdx.x / Hq;
    it.s = 0;
    if (!junction_items) {
        it.b = r / max_tiles;
        it.qt = max_tiles - 1 - (r - it.b * max_tiles);
        it.ok = it.qt < v.traj_tile[it.b + 1] - v.traj_tile[it.b];
        if (it.ok) it.s = v.seg[v.traj_tok[it.b] + it.qt * 128];
    } else {
        int lo = 0, hi = n_traj;   // largest b with traj_seg[b] <= r
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (v.traj_seg[mid] <= r) lo = mid; else hi = mid;
        }
        it.b = lo;
        it.s = r - v.traj_seg[lo];
        const int J = v.seg_start[r];
        it.qt = J >> 7;
        it.ok = it.s > 0 && (J & 127) != 0;
    }
    return it;
}

// Compact views: keys come from each segment's compact sequence
// (view_s gathered in order, §4.1 LogitTree), stored at rows
// (traj_km[b] + s nt) 128 + c of a compact K / V buffer. A q-tile item serves
// the rows of one segment, whose compact index is nb + (i - seg_lo) with nb
// the keys of view_s before the segment's own rows; row i sees compact keys
// 0 .. its own index, so a compact tile is FULL (every row of a whole tile
// sees every key), or PARTIAL with a prefix of keys visible to each row
// (DEAD_HI when no row reaches its second half).
struct CPiece {
    int r0, r1;          // the item's rows (trajectory-local) [r0, r1)
    int seg_lo, nb;      // first row of the segment; keys of view_s before it
    int cfirst, clast;   // compact indices of rows r0 and r1 - 1
    bool whole;          // the item covers all 128 rows of its q-tile
};
__device__ __forceinline__ CPiece cmp_piece(const VisView& v, int b, int s, int qt, int T) {
    CPiece c;
    const int gs = v.traj_seg[b] + s;
    const int nseg = v.traj_seg[b + 1] - v.traj_seg[b];
    c.seg_lo = v.seg_start[gs];
    const int seg_hi = s + 1 < nseg ? v.seg_start[gs + 1] : T;
    c.nb = v.seg_len[gs] - (seg_hi - c.seg_lo);
    c.r0 = max(c.seg_lo, qt * 128);
    c.r1 = min(seg_hi, qt * 128 + 128);
    c.cfirst = c.nb + c.r0 - c.seg_lo;
    c.clast = c.nb + c.r1 - 1 - c.seg_lo;
    c.whole = c.r0 == qt * 128 && c.r1 == qt * 128 + 128;
    return c;
}
// list entry (tile << 4) | code of compact key tile j for a piece
__device__ __forceinline__ int cmp_entry(const CPiece& c, int j) {
    if (c.whole && j * 128 + 127 <= c.cfirst) return (j << 4) | MW_TILE_FULL;
    return (j << 4) | MW_TILE_PARTIAL | (c.clast - j * 128 < 64 ? MW_TILE_DEAD_HI : 0);
}
// 128-bit mask with keys 0 .. lim set (none for lim < 0)
__device__ __forceinline__ uint4 prefix_words(int lim) {
    uint32_t w[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int hi = lim - 32 * q;
        w[q] = hi >= 31 ? 0xffffffffu : (hi < 0 ? 0u : ((2u << hi) - 1u));
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Softmax-gradient elements of the backward, two at a time: p = 2^(s c + n)
// with n = -LSE_i log2 e, masked pairs (bit clear in vm) entering the exp2 as
// -inf (so p = +0, no branch); ds = p (dp - Delta_i). MASKED = false when the
// caller knows every pair is visible.
template <bool MASKED>
__device__ __forceinline__ void soft_pair(float s0, float s1, float dp0, float dp1, uint64_t c2, uint64_t n2,
                                          uint64_t dl2, uint32_t vm, int bit, uint32_t& p_pk, uint32_t& ds_pk) {
    const uint64_t a = fma2(f2(s0, s1), c2, n2);
    float a0 = f2_lo(a), a1 = f2_hi(a);
    if (MASKED) {
        a0 = ((vm >> bit) & 1u) ? a0 : -INFINITY;
        a1 = ((vm >> (bit + 1)) & 1u) ? a1 : -INFINITY;
    }
    const float p0 = ex2(a0), p1 = ex2(a1);
    const uint64_t d = mul2(f2(p0, p1), sub2(f2(dp0, dp1), dl2));
    p_pk = pack_bf16(p0, p1);
    ds_pk = pack_bf16(f2_lo(d), f2_hi(d));
}

// float index of n for padded row r of the (n, Delta) row-pair array; Delta
// sits 2 floats further
__device__ __forceinline__ int64_t lsd_index(int64_t r) { return ((r >> 1) << 2) + (r & 1); }

__device__ __forceinline__ void load_tile(uint8_t* dst, const CUtensorMap* map, uint64_t* bar, int head, int row) {
    tma_load_3d(dst, map, bar, 0, head, row);
    tma_load_3d(dst + HALF_B, map, bar, 64, head, row);
}

// K-major operand descriptor for k-step ks (16 elements) of a [128][128] tile.
__device__ __forceinline__ uint64_t kmaj(uint32_t base, int ks) {
    return sdesc_sw128(base + (ks >> 2) * HALF_B + (ks & 3) * 32, 16, 1024);
}
// MN-major operand descriptor (rows = K dim, 128 contiguous N elements split in
// two 64-wide halves) for k-step ks.
__device__ __forceinline__ uint64_t mnmaj(uint32_t base, int ks) {
    return sdesc_sw128(base + ks * 2048, HALF_B, 1024);
}

__global__ void __launch_bounds__(NT_FWD, 1)
    k_attn_fwd_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                  const __grid_constant__ CUtensorMap tmV, FwdParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t q_full, k_full[2], k_empty[2], v_full[2], v_empty[2], s_full[2], s_free[2],
        p_full[2], o_done, o_fin;
    __shared__ uint32_t tmem_base;
    __shared__ int abort_flag;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const VisView& v = p.v;
    const QItem it = q_item(v, p.Hq, p.max_tiles, p.n_traj, p.junction_items);
    if (!it.ok) return;
    const int h = it.h, qt = it.qt, b = it.b;
    const int nt = v.traj_tile[b + 1] - v.traj_tile[b];
    const int64_t tok0 = v.traj_tok[b];
    const int T = v.traj_tok[b + 1] - (int)tok0;
    const int kvh = h / (p.Hq / p.Hkv);
    const CPiece cp = cmp_piece(v, b, it.s, qt, T);
    const int n = cp.clast / 128 + 1;   // compact key tiles 0 .. (last row's index) / 128
    auto entry = [&](int j) -> int { return cmp_entry(cp, j); };
    int32_t* status = v.status;

    if (threadIdx.x == 0) {
        mbar_init(&q_full, 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&k_empty[s], 1);
            mbar_init(&v_full[s], 1);
            mbar_init(&v_empty[s], 1);
            mbar_init(&s_full[s], 1);
            mbar_init(&s_free[s], 1);     // PV's completion: P lives in the S buffer until then
            mbar_init(&p_full[s], 128);   // per S buffer
        }
        mbar_init(&o_done, 1);
        mbar_init(&o_fin, 1);   // one phase: the last PV's completion
        abort_flag = 0;
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

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            prefetch_tmap(&tmQ);
            prefetch_tmap(&tmK);
            prefetch_tmap(&tmV);
            mbar_expect_tx(&q_full, TILE_B);
            load_tile(sm + SM_Q, &tmQ, &q_full, h, (int)(tok0 + qt * 128));
            // first K / V row of the item's segment's compact sequence
            const int64_t krow0 = (v.traj_km[b] + (int64_t)it.s * nt) * 128;
            for (int j = 0; j < n; ++j) {
                const int kt = entry(j) >> 4;
                const int s = j & 1;
                const int row = (int)(krow0 + kt * 128);
                if (j >= 2 && !mbar_wait(&k_empty[s], ((j - 2) >> 1) & 1, status, 101)) { abort_flag = 1; break; }
                mbar_expect_tx(&k_full[s], TILE_B);
                load_tile(sm + SM_K + s * TILE_B, &tmK, &k_full[s], kvh, (int)(krow0 + kt * 128));
                if (j >= 2 && !mbar_wait(&v_empty[s], ((j - 2) >> 1) & 1, status, 102)) { abort_flag = 1; break; }
                mbar_expect_tx(&v_full[s], TILE_B);
                load_tile(sm + SM_V + s * TILE_B, &tmV, &v_full[s], kvh, row);
                if (*(volatile int*)&abort_flag) break;
            }
        }
    } else if (warp == 1 || warp == FWD_PV_WARP) {
        // ------------------------------------------------------------ MMA issuers
        // warp 1: S_j = Q K_j^T; warp FWD_PV_WARP: O += P_t V_t
        if (lane == 0) {
            const uint32_t iS = idesc_bf16(128, 128, 0, 0);   // S = Q K^T: both K-major
            const uint32_t iO = idesc_bf16(128, 128, 0, 1);   // O += P V: V is MN-major
            const uint32_t sq = smem_u32(sm + SM_Q), sk = smem_u32(sm + SM_K), sv = smem_u32(sm + SM_V);
            bool ok = mbar_wait(&q_full, 0, status, 201);
            // O += P_t V_t with P_t (bf16, two keys per 32-bit column) read from
            // the first 64 columns of S buffer t & 1
            auto pv = [&](int t) -> bool {
                const int e = entry(t);
                if (!mbar_wait(&p_full[t & 1], (t >> 1) & 1, status, 202)) return false;
                if (!mbar_wait(&v_full[t & 1], (t >> 1) & 1, status, 203)) return false;
                tc_fence_after();
                const uint32_t vb = sv + (t & 1) * TILE_B;
                const uint32_t pa = tmem + TM_S0 + (t & 1) * 128;
                if (e & (MW_TILE_DEAD_LO | MW_TILE_DEAD_HI)) {
                    // K = 64: the live half's keys (16-row k-steps 4 lh .. 4 lh + 3 of V)
                    const int kh = (e & MW_TILE_DEAD_LO) ? 4 : 0;
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks)
                        mma_ts(tmem + TM_O, pa + 8 * ks, mnmaj(vb, ks + kh), iO, (t > 0 || ks > 0));
                } else {
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)
                        mma_ts(tmem + TM_O, pa + 8 * ks, mnmaj(vb, ks), iO, (t > 0 || ks > 0));
                }
                mma_commit(&v_empty[t & 1]);
                mma_commit(&s_free[t & 1]);
                mma_commit(&o_done);
                if (t == n - 1) mma_commit(&o_fin);
                return true;
            };
            if (warp == 1) {
                const uint32_t iS64 = idesc_bf16(128, 64, 0, 0);   // S over one live key half
                for (int j = 0; ok && j < n; ++j) {
                    const int s = j & 1;
                    const int e = entry(j);
                    if (!mbar_wait(&k_full[s], (j >> 1) & 1, status, 204)) { ok = false; break; }
                    if (j >= 2 && !mbar_wait(&s_free[s], ((j - 2) >> 1) & 1, status, 205)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t kb = sk + s * TILE_B;
                    if (e & (MW_TILE_DEAD_LO | MW_TILE_DEAD_HI)) {
                        // keys 64 lh .. 64 lh + 63: rows 64 lh.. of each 64-column panel
                        const uint32_t kh = kb + ((e & MW_TILE_DEAD_LO) ? 64u * 128u : 0u);
#pragma unroll
                        for (int ks = 0; ks < 8; ++ks)
                            mma_ss(tmem + TM_S0 + s * 128, kmaj(sq, ks), kmaj(kh, ks), iS64, ks > 0);
                    } else {
#pragma unroll
                        for (int ks = 0; ks < 8; ++ks)
                            mma_ss(tmem + TM_S0 + s * 128, kmaj(sq, ks), kmaj(kb, ks), iS, ks > 0);
                    }
                    mma_commit(&k_empty[s]);
                    mma_commit(&s_full[s]);
                }
            } else {
                for (int t = 0; ok && t < n; ++t) ok = pv(t);
            }
            if (!ok) abort_flag = 1;
        }
    } else {
        // ------------------------------------------------------------ softmax + epilogue
        const int qw = warp & 3;
        const int rl = qw * 32 + lane;          // row inside the q-tile = TMEM lane
        const int i = qt * 128 + rl;
        const int ie = min(i, T - 1);
        // this row's compact index (rows outside the item see no key)
        const bool in_piece = i >= cp.r0 && i < cp.r1;
        const int crow = in_piece ? cp.cfirst + i - cp.r0 : -(1 << 30);
        auto mask_words = [&](int e) -> uint4 { return prefix_words(crow - (e >> 4) * 128); };
        const uint32_t lane_base = tmem + ((uint32_t)(qw * 32) << 16);
        float m = -INFINITY, l = 0.f;
        bool ok = true;
        // list entries and view-mask words are loaded ahead (an entry two
        // tiles, a mask word one tile), so no step waits on a global load once
        // its S is ready
        int e_cur = n > 0 ? entry(0) : 0;
        int e_nxt = n > 1 ? entry(1) : 0;
        uint4 w_cur = n > 0 ? mask_words(e_cur) : make_uint4(0u, 0u, 0u, 0u);
        // One tile of the online softmax over NC 32-column chunks of S (4: the
        // whole tile; 2: a live key half): mask, row max, P = 2^(S c - m) into
        // the first NC * 16 columns of the buffer as bf16 pairs, row sum.
        // `lim`: keys c <= lim are causal (diagonal tile); returns the factor
        // by which O must be rescaled.
        auto soft_tile = [&](auto ncc, uint32_t sbuf, bool masked, int lim, uint32_t w0, uint32_t w1, uint32_t w2,
                             uint32_t w3) -> float {
            constexpr int NC = decltype(ncc)::value;
            constexpr int NS = NC * 32;
            float s[NS];
            {   // all loads in flight before one wait
                uint32_t rr[NC][32];
#pragma unroll
                for (int c = 0; c < NC; ++c) tmem_ld32(sbuf + c * 32, rr[c]);
                tmem_wait_ld();
#pragma unroll
                for (int c = 0; c < NC; ++c)
#pragma unroll
                    for (int x = 0; x < 32; ++x) s[c * 32 + x] = __uint_as_float(rr[c][x]);
            }
            if (masked) {
                uint32_t wd[4] = {w0, w1, w2, w3};
#pragma unroll
                for (int q = 0; q < NC; ++q) {   // causal inside the diagonal tile: keys c <= lim
                    const int hi = lim - 32 * q;   // keep bits 0..hi
                    wd[q] &= hi >= 31 ? 0xffffffffu : (hi < 0 ? 0u : ((2u << hi) - 1u));
                }
#pragma unroll
                for (int c = 0; c < NS; ++c)
                    if (!((wd[c >> 5] >> (c & 31)) & 1u)) s[c] = -INFINITY;
            }
            // row max as 8 independent partial chains (a single dependency chain
            // bounds the warp's latency), two new elements per instruction
            float pm[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) pm[k] = s[k];
            constexpr int NPAIR = (NS - 8) / 16;
#pragma unroll
            for (int c = 8; c < 8 + 16 * NPAIR; c += 16)
#pragma unroll
                for (int k = 0; k < 8; ++k) pm[k] = max3(pm[k], s[c + k], s[c + 8 + k]);
#pragma unroll
            for (int k = 0; k < 8; ++k) pm[k] = fmaxf(pm[k], s[8 + 16 * NPAIR + k]);   // the last 8
            const float mx = max3(max3(pm[0], pm[1], pm[2]), max3(pm[3], pm[4], pm[5]), fmaxf(pm[6], pm[7]));
            const float mx2 = mx * p.scale_log2;
            float alpha = 1.f;
            if (mx2 > m + RESCALE_T) {
                alpha = ex2(m - mx2);   // 0 when m = -inf
                m = mx2;
            }
            const float mu = (m == -INFINITY) ? 0.f : m;
            // P = 2^(S c - mu) and its row sum, two elements per FMA / add
            const uint64_t c2 = f2(p.scale_log2, p.scale_log2), n2 = f2(-mu, -mu);
            uint64_t ps[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
            for (int c = 0; c < NS; c += 2) {
                const uint64_t a = fma2(f2(s[c], s[c + 1]), c2, n2);
                s[c] = ex2(f2_lo(a));
                s[c + 1] = ex2(f2_hi(a));
                ps[(c >> 1) & 3] = add2(ps[(c >> 1) & 3], f2(s[c], s[c + 1]));
            }
            const uint64_t ps2 = add2(add2(ps[0], ps[1]), add2(ps[2], ps[3]));
            l = l * alpha + (f2_lo(ps2) + f2_hi(ps2));
            // P (bf16 pairs) over the first NC * 16 columns of its own S buffer;
            // the PV MMA reads it from there, so P never touches shared memory
#pragma unroll
            for (int q = 0; q < NC; ++q) {
                uint32_t pk[16];
#pragma unroll
                for (int x = 0; x < 16; ++x) pk[x] = pack_bf16(s[32 * q + 2 * x], s[32 * q + 2 * x + 1]);
                tmem_st16(sbuf + 16 * q, pk);
            }
            tmem_wait_st();
            return alpha;
        };
        for (int j = 0; j < n; ++j) {
            const int e = e_cur;
            const uint4 wv = w_cur;
            if (j + 1 < n) {
                w_cur = mask_words(e_nxt);
                e_cur = e_nxt;
                e_nxt = j + 2 < n ? entry(j + 2) : 0;
            }
            const int cls = e & 3;
            if (!mbar_wait(&s_full[j & 1], (j >> 1) & 1, status, 301)) { ok = false; break; }
            tc_fence_after();
            // a tile whose first or second key half no row sees was computed as
            // S = Q K_half^T (N = 64) over the first 64 columns of its buffer
            const int lh = (e & MW_TILE_DEAD_LO) ? 1 : 0;
            const uint32_t sbuf = lane_base + TM_S0 + (j & 1) * 128;
            float alpha;
            if (e & (MW_TILE_DEAD_LO | MW_TILE_DEAD_HI)) {
                const uint32_t w0 = lh ? wv.z : wv.x, w1 = lh ? wv.w : wv.y;
                alpha = soft_tile(std::integral_constant<int, 2>(), sbuf, true, 127, w0, w1, 0u, 0u);
            } else {
                alpha = soft_tile(std::integral_constant<int, 4>(), sbuf, cls != MW_TILE_FULL, 127, wv.x, wv.y,
                                  wv.z, wv.w);
            }
            // O was last written by PV_{j-1}; rescale it when the max moved
            if (j >= 1 && __any_sync(0xffffffffu, alpha != 1.f)) {
                if (!mbar_wait(&o_done, (j - 1) & 1, status, 302)) { ok = false; break; }
                tc_fence_after();
                uint32_t o[32];
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    tmem_ld32(lane_base + TM_O + c * 32, o);
                    tmem_wait_ld();
#pragma unroll
                    for (int x = 0; x < 32; ++x) o[x] = __float_as_uint(__uint_as_float(o[x]) * alpha);
                    uint32_t lo[16], hi[16];
#pragma unroll
                    for (int x = 0; x < 16; ++x) { lo[x] = o[x]; hi[x] = o[16 + x]; }
                    tmem_st16(lane_base + TM_O + c * 32, lo);
                    tmem_st16(lane_base + TM_O + c * 32 + 16, hi);
                }
                tmem_wait_st();
            }
            tc_fence_before();
            mbar_arrive(&p_full[j & 1]);
        }
        // epilogue: O / l, LSE (natural log). The final PV is awaited on its
        // own one-phase barrier: a parity wait on o_done for phase n - 1 would
        // also pass while o_done is still in phase n - 2 (same parity as n),
        // i.e. before the last two PVs have completed.
        if (ok && n > 0 && mbar_wait(&o_fin, 0, status, 303)) {
            tc_fence_after();
            const float inv = 1.f / l;
            __nv_bfloat16* orow = p.O + ((tok0 + ie) * p.Hq + h) * DH;
            uint32_t o[32];
            const bool store = in_piece && MW_DBG_IN(tok0 + i, v.total, status, 203);
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                tmem_ld32(lane_base + TM_O + c * 32, o);
                tmem_wait_ld();
                if (store) {
#pragma unroll
                    for (int x = 0; x < 4; ++x) {
                        uint4 pk;
                        pk.x = pack_bf16(__uint_as_float(o[8 * x + 0]) * inv, __uint_as_float(o[8 * x + 1]) * inv);
                        pk.y = pack_bf16(__uint_as_float(o[8 * x + 2]) * inv, __uint_as_float(o[8 * x + 3]) * inv);
                        pk.z = pack_bf16(__uint_as_float(o[8 * x + 4]) * inv, __uint_as_float(o[8 * x + 5]) * inv);
                        pk.w = pack_bf16(__uint_as_float(o[8 * x + 6]) * inv, __uint_as_float(o[8 * x + 7]) * inv);
                        *reinterpret_cast<uint4*>(orow + c * 32 + 8 * x) = pk;
                    }
                }
            }
            if (store) p.LSE[(int64_t)h * p.total + tok0 + i] = (m + __log2f(l)) * 0.6931471805599453f;
        } else {
            abort_flag = 1;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// ----------------------------------------------------------------------------
// dQ kernel (Q-stationary, one CTA per (q-tile, q-head), same item order as the
// forward). Per listed k-tile j:
//   S_j = Q K_j^T (TMEM, double-buffered), dP_j = dO V_j^T (TMEM, single),
//   P = exp2(S c - LSE2) on visible pairs, dS = P (dP - Delta) -> bf16 over
//   its own S buffer in TMEM, dQ += dS K_j (dS a TMEM operand, K_j MN-major in
//   smem; TMEM accumulator).
// dQ = scale * accumulator, written as bf16. No atomics: each dQ row is owned
// by one CTA.
constexpr uint32_t DQ_Q = 0;
constexpr uint32_t DQ_DO = DQ_Q + TILE_B;
constexpr uint32_t DQ_K = DQ_DO + TILE_B;
constexpr uint32_t DQ_V = DQ_K + 2 * TILE_B;
constexpr uint32_t DQ_DS = DQ_V + 2 * TILE_B;
constexpr uint32_t SMEM_DQ = DQ_DS + 1024;   // dS lives in TMEM
constexpr uint32_t TM_DP = 256, TM_DQ = 384;

struct BwdParams {
    VisView v;
    int64_t total;
    int n_traj, max_tiles, Hq, Hkv;
    float scale, scale_log2;
    const float* lsd;      // [Hq][n_tiles * 64] float4 (n_i, n_i+1, Delta_i, Delta_i+1), n = -LSE log2 e;
                           // rows padded to whole tiles
    int64_t n_rows;        // n_tiles * 128
    __nv_bfloat16* dQ;
    int junction_items;    // dQ: as FwdParams
    float* dKseg;          // dK/dV: float32 partials per compact row [rows][Hkv][DH]
    float* dVseg;
};

__global__ void __launch_bounds__(NT_BWD, 1)
    k_attn_dq_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmDO,
                 const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV, BwdParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t q_full, k_full[2], k_empty[2], v_full[2], v_empty[2], s_full[2], s_free[2],
        dp_full, dp_free, ds_full[2], dq_fin;
    __shared__ uint32_t tmem_base;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const VisView& v = p.v;
    const QItem it = q_item(v, p.Hq, p.max_tiles, p.n_traj, p.junction_items);
    if (!it.ok) return;
    const int h = it.h, qt = it.qt, b = it.b;
    const int nt = v.traj_tile[b + 1] - v.traj_tile[b];
    const int64_t g = v.traj_tile[b] + qt;
    const int64_t tok0 = v.traj_tok[b];
    const int T = v.traj_tok[b + 1] - (int)tok0;
    const int kvh = h / (p.Hq / p.Hkv);
    const CPiece cp = cmp_piece(v, b, it.s, qt, T);
    const int n = cp.clast / 128 + 1;   // compact key tiles 0 .. (last row's index) / 128
    auto entry = [&](int j) -> int { return cmp_entry(cp, j); };
    int32_t* status = v.status;
    if (*(volatile int32_t*)&status[1]) return;

    if (threadIdx.x == 0) {
        mbar_init(&q_full, 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&k_empty[s], 1);
            mbar_init(&v_full[s], 1);
            mbar_init(&v_empty[s], 1);
            mbar_init(&s_full[s], 1);
            mbar_init(&s_free[s], 1);     // dQ's completion: dS lives in the S buffer until then
            mbar_init(&ds_full[s], NEW);  // per S buffer
        }
        mbar_init(&dp_full, 1);
        mbar_init(&dp_free, NEW);
        mbar_init(&dq_fin, 1);   // one phase: the last dQ MMA's completion
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

    if (warp == 0) {
        if (lane == 0) {
            prefetch_tmap(&tmQ);
            prefetch_tmap(&tmDO);
            prefetch_tmap(&tmK);
            prefetch_tmap(&tmV);
            const int row0 = (int)(tok0 + qt * 128);
            mbar_expect_tx(&q_full, 2 * TILE_B);
            load_tile(sm + DQ_Q, &tmQ, &q_full, h, row0);
            load_tile(sm + DQ_DO, &tmDO, &q_full, h, row0);
            // first K / V row of the item's segment's compact sequence
            const int64_t krow0 = (v.traj_km[b] + (int64_t)it.s * nt) * 128;
            for (int j = 0; j < n; ++j) {
                const int kt = entry(j) >> 4;
                const int s = j & 1;
                const int row = (int)(krow0 + kt * 128);
                if (j >= 2 && !mbar_wait(&v_empty[s], ((j - 2) >> 1) & 1, status, 111)) break;
                mbar_expect_tx(&v_full[s], TILE_B);
                load_tile(sm + DQ_V + s * TILE_B, &tmV, &v_full[s], kvh, row);
                if (j >= 2 && !mbar_wait(&k_empty[s], ((j - 2) >> 1) & 1, status, 112)) break;
                mbar_expect_tx(&k_full[s], TILE_B);
                load_tile(sm + DQ_K + s * TILE_B, &tmK, &k_full[s], kvh, (int)(krow0 + kt * 128));
            }
        }
    } else if (warp == 1 || warp == BWD_ACC_WARP) {
        const uint32_t iKK = idesc_bf16(128, 128, 0, 0);  // both operands K-major
        const uint32_t iMN = idesc_bf16(128, 128, 0, 1);  // B MN-major
        const uint32_t sq = smem_u32(sm + DQ_Q), sdo = smem_u32(sm + DQ_DO), sk = smem_u32(sm + DQ_K),
                       sv = smem_u32(sm + DQ_V);
        bool ok = mbar_wait_warp(&q_full, 0, status, 211);
        // S_j (needs K_j and a free S buffer)
        // A tile whose first or second key half no row sees is computed over
        // the live half only: S and dP with N = 64, dQ += dS K with K = 64
        const uint32_t iKK64 = idesc_bf16(128, 64, 0, 0);
        auto issue_s = [&](int j, int e) -> bool {
            const int s = j & 1;
            if (!mbar_wait_warp(&k_full[s], (j >> 1) & 1, status, 212)) return false;
            if (j >= 2 && !mbar_wait_warp(&s_free[s], ((j - 2) >> 1) & 1, status, 213)) return false;
            tc_fence_after();
            if (e & (MW_TILE_DEAD_LO | MW_TILE_DEAD_HI)) {
                // the live half's 64 keys: rows 64 lh.. of each 64-column panel
                const uint32_t kh = sk + s * TILE_B + ((e & MW_TILE_DEAD_LO) ? 64u * 128u : 0u);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) mma_ss_w(tmem + TM_S0 + s * 128, kmaj(sq, ks), kmaj(kh, ks), iKK64, ks > 0);
            } else {
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    mma_ss_w(tmem + TM_S0 + s * 128, kmaj(sq, ks), kmaj(sk + s * TILE_B, ks), iKK, ks > 0);
            }
            mma_commit_w(&s_full[s]);
            return true;
        };
        // dP_j (needs V_j and the softmax to have read dP_{j-1})
        auto issue_dp = [&](int j, int e) -> bool {
            const int s = j & 1;
            if (!mbar_wait_warp(&v_full[s], (j >> 1) & 1, status, 214)) return false;
            if (j >= 1 && !mbar_wait_warp(&dp_free, (j - 1) & 1, status, 215)) return false;
            tc_fence_after();
            if (e & (MW_TILE_DEAD_LO | MW_TILE_DEAD_HI)) {
                const uint32_t vh = sv + s * TILE_B + ((e & MW_TILE_DEAD_LO) ? 64u * 128u : 0u);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) mma_ss_w(tmem + TM_DP, kmaj(sdo, ks), kmaj(vh, ks), iKK64, ks > 0);
            } else {
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    mma_ss_w(tmem + TM_DP, kmaj(sdo, ks), kmaj(sv + s * TILE_B, ks), iKK, ks > 0);
            }
            mma_commit_w(&v_empty[s]);
            mma_commit_w(&dp_full);
            return true;
        };
        // dQ += dS_t K_t, dS_t (bf16 pairs) read from TMEM: keys 0..63 in
        // columns 0..31 and keys 64..127 in columns 64..95 of S buffer t & 1
        // (half tile: the live half's keys 0..31 in columns 0..15, keys
        // 32..63 in columns 32..47; K rows from 16-row k-step 4 lh on)
        auto issue_dq = [&](int t) -> bool {
            const int e = entry(t);
            if (!mbar_wait_warp(&ds_full[t & 1], (t >> 1) & 1, status, 216)) return false;
            tc_fence_after();
            const uint32_t da = tmem + TM_S0 + (t & 1) * 128;
            if (e & (MW_TILE_DEAD_LO | MW_TILE_DEAD_HI)) {
                const int kh = (e & MW_TILE_DEAD_LO) ? 4 : 0;
#pragma unroll
                for (int ks = 0; ks < 4; ++ks)
                    mma_ts_w(tmem + TM_DQ, da + (ks < 2 ? 8 * ks : 32 + 8 * (ks - 2)),
                           mnmaj(sk + (t & 1) * TILE_B, ks + kh), iMN, (t > 0 || ks > 0));
            } else {
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    mma_ts_w(tmem + TM_DQ, da + (ks < 4 ? 8 * ks : 64 + 8 * (ks - 4)),
                           mnmaj(sk + (t & 1) * TILE_B, ks), iMN, (t > 0 || ks > 0));
            }
            mma_commit_w(&k_empty[t & 1]);
            mma_commit_w(&s_free[t & 1]);
            if (t == n - 1) mma_commit_w(&dq_fin);
            return true;
        };
        if (warp == 1) {
            for (int j = 0; ok && j < n; ++j) {
                const int e = entry(j);
                ok = issue_s(j, e) && issue_dp(j, e);
            }
        } else {
            // dQ's K-stage release also covers S_j: dS_j exists only once S_j is done
            for (int j = 0; ok && j < n; ++j) ok = issue_dq(j);
        }
    } else {
        // row rl = TMEM lane; this warp's 64 of the 128 key columns: [64 ch, 64 ch + 64)
        const int qw = warp & 3;
        const int ch = (warp - 2) >> 2;
        const int rl = qw * 32 + lane;
        const int i = qt * 128 + rl;
        const int ie = min(i, T - 1);
        // this row's compact index (rows outside the item see no key)
        const bool in_piece = i >= cp.r0 && i < cp.r1;
        const int crow = in_piece ? cp.cfirst + i - cp.r0 : -(1 << 30);
        auto mask_words = [&](int e) -> uint4 { return prefix_words(crow - (e >> 4) * 128); };
        const uint32_t lane_base = tmem + ((uint32_t)(qw * 32) << 16);
        const float* ld = p.lsd + lsd_index((int64_t)h * p.n_rows + g * 128 + rl);
        const uint64_t c2 = f2(p.scale_log2, p.scale_log2), n2 = f2(ld[0], ld[0]), dl2 = f2(ld[2], ld[2]);
        bool ok = true;
        // list entries and view-mask words are loaded ahead (an entry two
        // tiles, a mask word one tile), so no step waits on a global load once
        // its S is ready
        int e_cur = n > 0 ? entry(0) : 0;
        int e_nxt = n > 1 ? entry(1) : 0;
        uint4 w_cur = n > 0 ? mask_words(e_cur) : make_uint4(0u, 0u, 0u, 0u);
        // One k-tile for this thread's NC 32-key chunks (2: its 64 keys of a
        // full tile; 1: its 32 of a live half), S and dP read at columns scol /
        // dcol: P = 2^(S c - LSE2), two elements per instruction, masked pairs
        // entering the exp2 as -inf (P = +0) instead of branching around it;
        // dS = P (dP - Delta) as bf16 pairs over the first NC * 16 of its own S
        // columns, which only this thread has read.
        auto dq_step = [&](auto ncc, int j, uint32_t scol, uint32_t dcol, uint32_t w0, uint32_t w1) -> bool {
            constexpr int NC = decltype(ncc)::value;
            float s[NC * 32];
            {   // all loads in flight before one wait
                uint32_t rr[NC][32];
#pragma unroll
                for (int c = 0; c < NC; ++c) tmem_ld32(scol + c * 32, rr[c]);
                tmem_wait_ld();
#pragma unroll
                for (int c = 0; c < NC; ++c)
#pragma unroll
                    for (int x = 0; x < 32; ++x) s[c * 32 + x] = __uint_as_float(rr[c][x]);
            }
            if (__all_sync(0xffffffffu, (NC == 2 ? (w0 & w1) : w0) == 0xffffffffu)) {
#pragma unroll
                for (int x = 0; x < NC * 16; ++x) {
                    const uint64_t a = fma2(f2(s[2 * x], s[2 * x + 1]), c2, n2);
                    s[2 * x] = ex2(f2_lo(a));
                    s[2 * x + 1] = ex2(f2_hi(a));
                }
            } else {
#pragma unroll
                for (int x = 0; x < NC * 16; ++x) {
                    const uint32_t wm = x < 16 ? w0 : w1;
                    const int bit = (2 * x) & 31;
                    const uint64_t a = fma2(f2(s[2 * x], s[2 * x + 1]), c2, n2);
                    s[2 * x] = ex2(((wm >> bit) & 1u) ? f2_lo(a) : -INFINITY);
                    s[2 * x + 1] = ex2(((wm >> (bit + 1)) & 1u) ? f2_hi(a) : -INFINITY);
                }
            }
            if (!mbar_wait(&dp_full, j & 1, status, 312)) return false;
            tc_fence_after();
            uint32_t dpr[NC][32];   // all dP loads in flight before one wait
#pragma unroll
            for (int cc = 0; cc < NC; ++cc) tmem_ld32(dcol + cc * 32, dpr[cc]);
            tmem_wait_ld();
            tc_fence_before();
            mbar_arrive(&dp_free);
#pragma unroll
            for (int cc = 0; cc < NC; ++cc) {
                const uint32_t* dp = dpr[cc];
                uint32_t pk[16];
#pragma unroll
                for (int x = 0; x < 16; ++x) {
                    const int c0 = cc * 32 + 2 * x;
                    const uint64_t d = mul2(f2(s[c0], s[c0 + 1]),
                                            sub2(f2(__uint_as_float(dp[2 * x]), __uint_as_float(dp[2 * x + 1])), dl2));
                    pk[x] = pack_bf16(f2_lo(d), f2_hi(d));
                }
                tmem_st16(scol + 16 * cc, pk);
            }
            tmem_wait_st();
            return true;
        };
        for (int j = 0; j < n; ++j) {
            const int e = e_cur;
            const uint4 wv = w_cur;
            if (j + 1 < n) {
                w_cur = mask_words(e_nxt);
                e_cur = e_nxt;
                e_nxt = j + 2 < n ? entry(j + 2) : 0;
            }
            const int cls = e & 3;
            if (!mbar_wait(&s_full[j & 1], (j >> 1) & 1, status, 311)) { ok = false; break; }
            tc_fence_after();
            const uint32_t sbuf = lane_base + TM_S0 + (j & 1) * 128;
            bool stepok;
            if (e & (MW_TILE_DEAD_LO | MW_TILE_DEAD_HI)) {
                // the live half's 64 keys, 32 per warp of the lane quarter
                const bool hi_half = (e & MW_TILE_DEAD_LO) != 0;
                const uint32_t wm = hi_half ? (ch ? wv.w : wv.z) : (ch ? wv.y : wv.x);
                stepok = dq_step(std::integral_constant<int, 1>(), j, sbuf + 32 * ch, lane_base + TM_DP + 32 * ch, wm, 0u);
            } else {
                uint32_t wd[4] = {0xffffffffu, 0xffffffffu, 0xffffffffu, 0xffffffffu};
                if (cls != MW_TILE_FULL) {
                    wd[0] = wv.x; wd[1] = wv.y; wd[2] = wv.z; wd[3] = wv.w;
                }
                stepok = dq_step(std::integral_constant<int, 2>(), j, sbuf + 64 * ch, lane_base + TM_DP + 64 * ch,
                                 ch ? wd[2] : wd[0], ch ? wd[3] : wd[1]);
            }
            if (!stepok) { ok = false; break; }
            tc_fence_before();
            mbar_arrive(&ds_full[j & 1]);
        }
        // awaited on a one-phase barrier (a parity wait on a per-tile barrier
        // could pass one phase early, before the last dQ MMAs complete)
        if (ok && n > 0 && mbar_wait(&dq_fin, 0, status, 314)) {
            tc_fence_after();
            __nv_bfloat16* qrow = p.dQ + ((tok0 + ie) * p.Hq + h) * DH;
            uint32_t o[32];
            const bool store = in_piece && MW_DBG_IN(tok0 + i, v.total, status, 204);
#pragma unroll
            for (int cc = 0; cc < 2; ++cc) {
                const int c = 2 * ch + cc;
                tmem_ld32(lane_base + TM_DQ + c * 32, o);
                tmem_wait_ld();
                if (store) {
#pragma unroll
                    for (int x = 0; x < 4; ++x) {
                        uint4 pk;
                        pk.x = pack_bf16(__uint_as_float(o[8 * x + 0]) * p.scale, __uint_as_float(o[8 * x + 1]) * p.scale);
                        pk.y = pack_bf16(__uint_as_float(o[8 * x + 2]) * p.scale, __uint_as_float(o[8 * x + 3]) * p.scale);
                        pk.z = pack_bf16(__uint_as_float(o[8 * x + 4]) * p.scale, __uint_as_float(o[8 * x + 5]) * p.scale);
                        pk.w = pack_bf16(__uint_as_float(o[8 * x + 6]) * p.scale, __uint_as_float(o[8 * x + 7]) * p.scale);
                        *reinterpret_cast<uint4*>(qrow + c * 32 + 8 * x) = pk;
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// ----------------------------------------------------------------------------
// dK / dV kernel (KV-stationary, one CTA per (compact key tile, kv-head,
// segment), smallest key tiles -- the longest runs -- first). Steps run over
// the run of q-tiles whose rows see the tile's keys (last q-tile first) x the
// group's query heads x two 64-row halves:
//   S^T = K Q^T, dP^T = V dO^T   (M=128 keys, N=64 rows; TMEM, double-buffered)
//   P^T = exp2(S^T c - LSE2_i), dS^T = P^T (dP^T - Delta_i) on visible pairs,
//   written as bf16 over their own S^T / dP^T TMEM buffers
//   dV += P^T dO, dK += dS^T Q   (P^T, dS^T TMEM operands; dO, Q MN-major in smem)
// The segment's rows that see compact key c form the interval
// [J_s + max(0, c - nb_s), J_{s+1}), so the mask is two compares per element.
constexpr uint32_t HT_B = 64 * DH * 2;     // 64-row half tile: two [64][64] swizzled halves
constexpr uint32_t HT_HALF = HT_B / 2;
constexpr uint32_t KV_K = 0;
constexpr uint32_t KV_V = KV_K + TILE_B;
constexpr int QD_ST = 5;                           // (Q half, dO half) stages
constexpr uint32_t KV_Q = KV_V + TILE_B;
constexpr uint32_t SMEM_KV = KV_Q + QD_ST * 2 * HT_B + 1024;   // P^T, dS^T live in TMEM
constexpr uint32_t TM_ST = 0, TM_DPT = 128, TM_DV = 256, TM_DK = 384;

// K-major descriptor, k-step ks, of a 64-row half tile ([64][128] as two [64][64]).
__device__ __forceinline__ uint64_t kmaj_ht(uint32_t base, int ks) {
    return sdesc_sw128(base + (ks >> 2) * HT_HALF + (ks & 3) * 32, 16, 1024);
}
// MN-major descriptor, k-step ks (16 rows), of a 64-row half tile.
__device__ __forceinline__ uint64_t mnmaj_ht(uint32_t base, int ks) {
    return sdesc_sw128(base + ks * 2048, HT_HALF, 1024);
}

__global__ void __launch_bounds__(NT_BWD, 1)
    k_attn_dkdv_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmDO,
                   const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV, BwdParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t kv_full, qd_full[QD_ST], qd_empty[QD_ST], sd_full[2], sd_free[2], pd_full[2];
    __shared__ uint32_t tmem_base;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int grp = p.Hq / p.Hkv;
    // KV head outermost, then trajectory by trajectory: the CTAs resident at
    // one time hold the key tiles of one or two trajectories under one head,
    // and walk the same Q / dO tiles from the trajectory's end (L2 reuse
    // across key tiles; with the trajectories interleaved instead, a record of
    // many short trajectories spread the resident CTAs over all of them and
    // read Q / dO from DRAM again for nearly every key tile)
    const int kvh = blockIdx.x / (p.max_tiles * p.n_traj);
    const int r = blockIdx.x % (p.max_tiles * p.n_traj);
    const int b = r / p.max_tiles;
    const int kt = r % p.max_tiles;
    const VisView& v = p.v;
    const int nt = v.traj_tile[b + 1] - v.traj_tile[b];
    if (kt >= nt) return;
    const int64_t tok0 = v.traj_tok[b];
    const int T = v.traj_tok[b + 1] - (int)tok0;
    // item (compact key tile kt, segment blockIdx.y): keys kt*128.. of view_s;
    // the rows that see one of them are the segment's rows whose compact index
    // reaches kt*128, a contiguous run of q-tiles
    const int sgb = v.traj_seg[b];
    const int sk = blockIdx.y;
    if (sk >= v.traj_seg[b + 1] - sgb) return;
    const int clen = v.seg_len[sgb + sk];                  // |view_s|
    if (kt * 128 >= clen) return;
    const int seg_lo = v.seg_start[sgb + sk];
    const int seg_hi = sgb + sk + 1 < v.traj_seg[b + 1] ? v.seg_start[sgb + sk + 1] : T;
    const int nb = clen - (seg_hi - seg_lo);               // keys of view_s before the segment's rows
    const int qlo = (seg_lo + max(0, kt * 128 - nb)) >> 7;
    const int nlist = ((seg_hi - 1) >> 7) - qlo + 1;
    const int64_t krow0 = (v.traj_km[b] + (int64_t)sk * nt + kt) * 128;   // first compact K / V row
    const int nsteps = nlist * grp * 2;
    int32_t* status = v.status;
    if (*(volatile int32_t*)&status[1]) return;

    if (threadIdx.x == 0) {
        mbar_init(&kv_full, 1);
        for (int s = 0; s < QD_ST; ++s) {
            mbar_init(&qd_full[s], 1);
            mbar_init(&qd_empty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&sd_full[s], 1);
            mbar_init(&sd_free[s], 1);     // the accumulation's completion: P^T / dS^T live there until then
            mbar_init(&pd_full[s], NEW);
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
    // step t -> (list entry e, head in group, half), kept as a running cursor
    // (integer division on these threads costs more than a step's work). The
    // list is walked from its last q-tile down, so CTAs of one KV head that
    // started together stream the same Q / dO tiles at the same time (L2 reuse
    // across k-tiles); rem = 2 * (head in group) + half.
    // The q-tiles of the current and the next list entry are cached, so that
    // no step waits on a load of the list.
    struct Cursor {
        int e, rem, qt, qt_next;
    };
    auto list_qt = [&](int e) -> int { return e >= 0 ? qlo + e : 0; };
    const Cursor first{nlist - 1, 0, list_qt(nlist - 1), list_qt(nlist - 2)};
    auto advance = [&](Cursor& c) {
        if (++c.rem == 2 * grp) {
            c.rem = 0;
            --c.e;
            c.qt = c.qt_next;
            c.qt_next = list_qt(c.e - 1);
        }
    };
    auto cur_q0 = [&](const Cursor& c, int& hq) -> int {
        hq = kvh * grp + (c.rem >> 1);
        return c.qt * 128 + (c.rem & 1) * 64;
    };

    if (warp == 0) {
        if (lane == 0) {
            prefetch_tmap(&tmQ);
            prefetch_tmap(&tmDO);
            prefetch_tmap(&tmK);
            prefetch_tmap(&tmV);
            mbar_expect_tx(&kv_full, 2 * TILE_B);
            load_tile(sm + KV_K, &tmK, &kv_full, kvh, (int)krow0);
            load_tile(sm + KV_V, &tmV, &kv_full, kvh, (int)krow0);
            Cursor c = first;
            int s = 0;
            uint32_t ph = 0;
            for (int t = 0; t < nsteps; ++t, advance(c)) {
                int hq;
                const int q0 = cur_q0(c, hq);
                if (t >= QD_ST && !mbar_wait(&qd_empty[s], ph ^ 1u, status, 121)) break;
                mbar_expect_tx(&qd_full[s], 2 * HT_B);
                uint8_t* dst = sm + KV_Q + s * 2 * HT_B;
                tma_load_3d(dst, &tmQ, &qd_full[s], 0, hq, (int)(tok0 + q0));
                tma_load_3d(dst + HT_HALF, &tmQ, &qd_full[s], 64, hq, (int)(tok0 + q0));
                tma_load_3d(dst + HT_B, &tmDO, &qd_full[s], 0, hq, (int)(tok0 + q0));
                tma_load_3d(dst + HT_B + HT_HALF, &tmDO, &qd_full[s], 64, hq, (int)(tok0 + q0));
                if (++s == QD_ST) {
                    s = 0;
                    ph ^= 1u;
                }
            }
        }
    } else if (warp == 1 || warp == BWD_ACC_WARP) {
        const uint32_t iSD = idesc_bf16(128, 64, 0, 0);
        const uint32_t iAC = idesc_bf16(128, 128, 0, 1);
        const uint32_t sk = smem_u32(sm + KV_K), sv = smem_u32(sm + KV_V), sq = smem_u32(sm + KV_Q);
        bool ok = mbar_wait_warp(&kv_full, 0, status, 221);
        auto issue_sd = [&](int t) -> bool {
            const int s = t & 1, qs = t % QD_ST;
            if (!mbar_wait_warp(&qd_full[qs], (t / QD_ST) & 1, status, 222)) return false;
            if (t >= 2 && !mbar_wait_warp(&sd_free[s], ((t - 2) >> 1) & 1, status, 223)) return false;
            tc_fence_after();
            const uint32_t qb = sq + qs * 2 * HT_B, db = qb + HT_B;
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) mma_ss_w(tmem + TM_ST + s * 64, kmaj(sk, ks), kmaj_ht(qb, ks), iSD, ks > 0);
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) mma_ss_w(tmem + TM_DPT + s * 64, kmaj(sv, ks), kmaj_ht(db, ks), iSD, ks > 0);
            mma_commit_w(&sd_full[s]);
            return true;
        };
        auto issue_acc = [&](int t) -> bool {
            const int s = t & 1, qs = t % QD_ST;
            if (!mbar_wait_warp(&pd_full[s], (t >> 1) & 1, status, 224)) return false;
            tc_fence_after();
            const uint32_t qb = sq + qs * 2 * HT_B, db = qb + HT_B;
            // P^T, dS^T (bf16 pairs of query rows) in TMEM: rows 0..31 of the
            // half-step in columns 0..15, rows 32..63 in columns 32..47 of
            // their S^T / dP^T buffer
#pragma unroll
            for (int ks = 0; ks < 4; ++ks)
                mma_ts_w(tmem + TM_DV, tmem + TM_ST + s * 64 + 32 * (ks >> 1) + 8 * (ks & 1), mnmaj_ht(db, ks), iAC,
                       (t > 0 || ks > 0));
#pragma unroll
            for (int ks = 0; ks < 4; ++ks)
                mma_ts_w(tmem + TM_DK, tmem + TM_DPT + s * 64 + 32 * (ks >> 1) + 8 * (ks & 1), mnmaj_ht(qb, ks), iAC,
                       (t > 0 || ks > 0));
            mma_commit_w(&qd_empty[qs]);
            mma_commit_w(&sd_free[s]);
            return true;
        };
        if (warp == 1) {
            for (int t = 0; ok && t < nsteps; ++t) ok = issue_sd(t);
        } else {
            // the Q/dO stage release also covers S^T_t, dP^T_t: P^T_t, dS^T_t
            // exist only once those are done
            for (int t = 0; ok && t < nsteps; ++t) ok = issue_acc(t);
        }
    } else {
        // key row rl = TMEM lane; this warp's 32 of a half-step's 64 query
        // columns: [32 ch, 32 ch + 32)
        const int qw = warp & 3;
        const int ch = (warp - 2) >> 2;
        const int rl = qw * 32 + lane;               // key row inside the k-tile = TMEM lane
        const int jk = kt * 128 + rl;                // this thread's compact key
        // compact key jk of view_s is seen by the segment's rows whose compact
        // index reaches it: [jlo, iend)
        const bool kin = jk < clen;
        const int jlo = kin ? seg_lo + max(0, jk - nb) : 0;
        const int iend = kin ? seg_hi : 0;
        const uint32_t lane_base = tmem + ((uint32_t)(qw * 32) << 16);
        bool ok = true;
        // (-LSE2, Delta) of this warp's 32 query rows of a step: 256 contiguous
        // bytes of the tile-padded row-pair array, read by every lane
        // (broadcast) at the start of the step, after a prefetch into L1 one
        // step earlier. A float4 holds two rows' (n, n', Delta, Delta'), so its
        // halves are the register pairs the paired arithmetic takes.
        const int64_t lsd_k = (int64_t)v.traj_tile[b] * 128 + 32 * ch;
        auto lsd_row = [&](const Cursor& c) -> const float4* {
            int hq;
            const int q0 = cur_q0(c, hq);
            return reinterpret_cast<const float4*>(p.lsd + lsd_index(lsd_k + (int64_t)hq * p.n_rows + q0));
        };
        Cursor cur = first, nxt = first;   // steps t and t + 1
        advance(nxt);
        for (int t = 0; t < nsteps; ++t) {
            const int s = t & 1;
            int hq;
            const int q0 = cur_q0(cur, hq);
            float4 lv[16];
            {
                const float4* l4 = lsd_row(cur);
#pragma unroll
                for (int q = 0; q < 16; ++q) lv[q] = l4[q];
            }
            if (t + 1 < nsteps && lane < 2)
                asm volatile("prefetch.global.L1 [%0];" ::"l"(reinterpret_cast<const char*>(lsd_row(nxt)) + 128 * lane));
            if (!mbar_wait(&sd_full[s], (t >> 1) & 1, status, 321)) { ok = false; break; }
            tc_fence_after();
            float sv[32], dp[32];
            {   // both loads in flight before one wait
                uint32_t ra[32], rb[32];
                tmem_ld32(lane_base + TM_ST + s * 64 + ch * 32, ra);
                tmem_ld32(lane_base + TM_DPT + s * 64 + ch * 32, rb);
                tmem_wait_ld();
#pragma unroll
                for (int x = 0; x < 32; ++x) {
                    sv[x] = __uint_as_float(ra[x]);
                    dp[x] = __uint_as_float(rb[x]);
                }
            }
            // visible columns [lo, hi) of this warp's 32, as a bit mask
            const int lo = min(max(jlo, q0 + 32 * ch) - q0 - 32 * ch, 32);
            const int hi = max(min(min(iend, q0 + 64) - q0 - 32 * ch, 32), lo);
            const uint32_t vm = (hi >= 32 ? 0xffffffffu : ((1u << hi) - 1u)) & ~(lo >= 32 ? 0xffffffffu : ((1u << lo) - 1u));
            {   // P^T, dS^T (bf16 pairs) over the first 16 of this warp's own 32
                // columns of the S^T / dP^T buffers, which only this thread has read
                uint32_t pa[16], pd[16];
                const uint64_t c2 = f2(p.scale_log2, p.scale_log2);
                if (__all_sync(0xffffffffu, vm == 0xffffffffu)) {
#pragma unroll
                    for (int x = 0; x < 16; ++x)
                        soft_pair<false>(sv[2 * x], sv[2 * x + 1], dp[2 * x], dp[2 * x + 1], c2, f2(lv[x].x, lv[x].y),
                                         f2(lv[x].z, lv[x].w), vm, 2 * x, pa[x], pd[x]);
                } else {
#pragma unroll
                    for (int x = 0; x < 16; ++x)
                        soft_pair<true>(sv[2 * x], sv[2 * x + 1], dp[2 * x], dp[2 * x + 1], c2, f2(lv[x].x, lv[x].y),
                                        f2(lv[x].z, lv[x].w), vm, 2 * x, pa[x], pd[x]);
                }
                tmem_st16(lane_base + TM_ST + s * 64 + 32 * ch, pa);
                tmem_st16(lane_base + TM_DPT + s * 64 + 32 * ch, pd);
                tmem_wait_st();
            }
            tc_fence_before();
            mbar_arrive(&pd_full[s]);
            cur = nxt;
            advance(nxt);
        }
        if (ok && mbar_wait(&sd_free[(nsteps - 1) & 1], ((nsteps - 1) >> 1) & 1, status, 323)) {
            // float32 partials of this segment, unscaled dV and scaled dK
            // per compact row
            tc_fence_after();
            const int64_t row = ((krow0 + rl) * p.Hkv + kvh) * DH;
            const bool kstore = kin && MW_DBG_IN(krow0 + rl, v.n_keymask * 128, status, 205);
            uint32_t o[32];
#pragma unroll
            for (int pass = 0; pass < 2; ++pass) {
                float* dst = (pass == 0 ? p.dVseg : p.dKseg) + row;
                const float mul = pass == 0 ? 1.f : p.scale;
                const uint32_t col = pass == 0 ? TM_DV : TM_DK;
#pragma unroll
                for (int cc = 0; cc < 2; ++cc) {
                    const int c = 2 * ch + cc;
                    tmem_ld32(lane_base + col + c * 32, o);
                    tmem_wait_ld();
                    if (kstore) {
#pragma unroll
                        for (int x = 0; x < 8; ++x)
                            *reinterpret_cast<float4*>(dst + c * 32 + 4 * x) =
                                make_float4(__uint_as_float(o[4 * x + 0]) * mul, __uint_as_float(o[4 * x + 1]) * mul,
                                            __uint_as_float(o[4 * x + 2]) * mul, __uint_as_float(o[4 * x + 3]) * mul);
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

}  // namespace

// Whether TMA's int32 row coordinates reach every compact K / V row (128 per
// (segment, k-tile) entry) and the junction-item and dK/dV grids fit.
static bool cmp_fits(const mw_vis_layout* L, int Hq) {
    return L->n_keymask * 128 <= INT32_MAX && L->n_segs * (int64_t)Hq <= INT32_MAX && L->max_segs <= 65535;
}

namespace {

// (n_i = -LSE_i log2 e, Delta_i = rowsum(dO_i * O_i)) per (head, row) in the
// tile-padded layout [Hq][n_tiles * 128 rows]: padded row r = h n_rows + g 128
// + (row in tile g) sits in float4 r / 2 as (n_r, n_r+1, Delta_r, Delta_r+1)
// (r even), so any 32 rows of a tile are 256 contiguous, 16-byte aligned
// bytes. Rows past a trajectory's end hold zeros. One warp per (row, head).
__global__ void k_attn_lsd(VisView v, int64_t total, int64_t n_rows, int Hq, const __nv_bfloat16* __restrict__ O,
                           const __nv_bfloat16* __restrict__ dO, const float* __restrict__ LSE,
                           float* __restrict__ lsd) {
    const int lane = threadIdx.x & 31;
    const int64_t nw = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t w = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; w < n_rows * Hq; w += nw) {
        const int64_t gr = w / Hq;
        const int h = (int)(w - gr * Hq);
        const int g = (int)(gr >> 7);
        const int b = v.tile_traj[g];
        const int64_t tok0 = v.traj_tok[b];
        const int i = (g - v.traj_tile[b]) * 128 + (int)(gr & 127);
        float2 out = make_float2(0.f, 0.f);
        if (i < v.traj_tok[b + 1] - (int)tok0) {
            const int64_t row = ((tok0 + i) * Hq + h) * DH + 4 * lane;
            const uint2 o = *reinterpret_cast<const uint2*>(O + row), d = *reinterpret_cast<const uint2*>(dO + row);
            const float2 o0 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&o.x));
            const float2 o1 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&o.y));
            const float2 d0 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&d.x));
            const float2 d1 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&d.y));
            const float acc = warp_sum(fmaf(o0.x, d0.x, fmaf(o0.y, d0.y, fmaf(o1.x, d1.x, o1.y * d1.y))));
            out = make_float2(-LSE[(int64_t)h * total + tok0 + i] * LOG2E, acc);
        }
        if (lane == 0) {
            const int64_t at = lsd_index((int64_t)h * n_rows + gr);
            lsd[at] = out.x;
            lsd[at + 2] = out.y;
        }
    }
}

// Compact K / V: row (traj_km[b] + s nt) 128 + c of Kc, Vc holds the key at
// rank c of view_s (csrc) for c < |view_s|, zeros up to the end of that
// tile. With a rotary table the K row is also turned to position c, its
// logical position in view_s (§4.2): feature f pairs with f + 64 and turns by
// table[c][f] = (cos, sin). One block per (segment, tile) entry with keys in
// it; 16-byte vectors.
__device__ __forceinline__ int cmp_entry_traj(const VisView& v, int n_traj, int64_t e, int& s, int& kt, int& nt) {
    int lo = 0, hi = n_traj;   // the trajectory holding entry e: largest b with traj_km[b] <= e
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (v.traj_km[mid] <= e) lo = mid; else hi = mid;
    }
    nt = v.traj_tile[lo + 1] - v.traj_tile[lo];
    const int64_t rel = e - v.traj_km[lo];
    s = (int)(rel / nt);
    kt = (int)(rel - (int64_t)s * nt);
    return lo;
}

__global__ void __launch_bounds__(256) k_cmp_gather(VisView v, int n_traj, int Hkv,
                                                    const __nv_bfloat16* __restrict__ K,
                                                    const __nv_bfloat16* __restrict__ V, __nv_bfloat16* __restrict__ Kc,
                                                    __nv_bfloat16* __restrict__ Vc, const float2* __restrict__ table) {
    const int64_t e = blockIdx.x;
    int s, kt, nt;
    const int b = cmp_entry_traj(v, n_traj, e, s, kt, nt);
    if (kt * 128 >= v.seg_len[v.traj_seg[b] + s]) return;
    const int64_t tok0 = v.traj_tok[b];
    const int T_b = v.traj_tok[b + 1] - (int)tok0;
    const int vec = Hkv * (DH / 8);   // 16-byte vectors per key row
    for (int x = threadIdx.x; x < 128 * vec; x += blockDim.x) {
        const int r = x / vec, k = x - r * vec;
        int j = v.csrc[e * 128 + r];
        if (j >= 0 && !MW_DBG_IN(j, T_b, v.status, 201)) j = -1;
        uint4 vv = make_uint4(0u, 0u, 0u, 0u);
        if (j >= 0) vv = reinterpret_cast<const uint4*>(V + (tok0 + j) * Hkv * DH)[k];
        reinterpret_cast<uint4*>(Vc + (e * 128 + r) * Hkv * DH)[k] = vv;
        if (!table) {
            uint4 kv = make_uint4(0u, 0u, 0u, 0u);
            if (j >= 0) kv = reinterpret_cast<const uint4*>(K + (tok0 + j) * Hkv * DH)[k];
            reinterpret_cast<uint4*>(Kc + (e * 128 + r) * Hkv * DH)[k] = kv;
        } else if ((k & 15) < 8) {
            // vector k of head k / 16 holds features 8 (k % 16) ..; with its
            // partner 64 features on, it is one rotated 16-element unit
            const int h = k >> 4, f0 = 8 * (k & 15);
            const int64_t c = (int64_t)kt * 128 + r;   // the key's rank in view_s
            uint4 lo = make_uint4(0u, 0u, 0u, 0u), hi = lo;
            if (j >= 0) {
                const __nv_bfloat16* src = K + ((tok0 + j) * Hkv + h) * DH;
                const uint4 x0 = *reinterpret_cast<const uint4*>(src + f0);
                const uint4 x1 = *reinterpret_cast<const uint4*>(src + 64 + f0);
                const uint32_t a[4] = {x0.x, x0.y, x0.z, x0.w}, bq[4] = {x1.x, x1.y, x1.z, x1.w};
                uint32_t ya[4], yb[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    float y[4];
#pragma unroll
                    for (int u = 0; u < 2; ++u) {
                        const float2 cs = table[c * 64 + f0 + 2 * q + u];
                        const float p0 = u ? __uint_as_float(a[q] & 0xffff0000u) : __uint_as_float(a[q] << 16);
                        const float p1 = u ? __uint_as_float(bq[q] & 0xffff0000u) : __uint_as_float(bq[q] << 16);
                        y[u] = fmaf(p0, cs.x, -p1 * cs.y);
                        y[2 + u] = fmaf(p1, cs.x, p0 * cs.y);
                    }
                    ya[q] = pack_bf16(y[0], y[1]);
                    yb[q] = pack_bf16(y[2], y[3]);
                }
                lo = make_uint4(ya[0], ya[1], ya[2], ya[3]);
                hi = make_uint4(yb[0], yb[1], yb[2], yb[3]);
            }
            __nv_bfloat16* dst = Kc + ((e * 128 + r) * Hkv + h) * DH;
            *reinterpret_cast<uint4*>(dst + f0) = lo;
            *reinterpret_cast<uint4*>(dst + 64 + f0) = hi;
        }
    }
}

// dK, dV of every key from the compact float32 partials: the sum, in segment
// order, over the segments whose views hold the key, each taken at the key's
// rank there (cpos); dKc carries the softmax scale already. With a rotary
// table each dK partial is first turned back by the key's position in that
// segment (its rank). A key enters the views at its own segment, so the scan
// starts there. One block per key tile; the order of the additions is fixed,
// so the result is deterministic.
__global__ void __launch_bounds__(256) k_cmp_reduce(VisView v, int Hkv, const float* __restrict__ dKc,
                                                    const float* __restrict__ dVc, __nv_bfloat16* __restrict__ dK,
                                                    __nv_bfloat16* __restrict__ dV, const float2* __restrict__ table) {
    const int64_t g = blockIdx.x;
    const int b = v.tile_traj[g];
    const int nt = v.traj_tile[b + 1] - v.traj_tile[b];
    const int kt = (int)(g - v.traj_tile[b]);
    const int64_t tok0 = v.traj_tok[b];
    const int T = v.traj_tok[b + 1] - (int)tok0;
    const int nseg = v.traj_seg[b + 1] - v.traj_seg[b];
    const int vec = Hkv * (DH / 8);   // 8-element chunks per key row
    for (int x = threadIdx.x; x < 128 * vec; x += blockDim.x) {
        const int r = x / vec, k = x - r * vec;
        const int j = kt * 128 + r;
        if (j >= T) continue;
        // dV: chunk k; dK: chunk k, or (rotary) the pair of chunks k, k + 8
        // of one head when k is in the first half of its head
        const bool rot = table != nullptr;
        const bool kdo = !rot || (k & 15) < 8;
        const int kk = rot ? ((k >> 4) << 4) + (k & 15) + 8 : k;   // partner chunk (rotary)
        float ak[8], ak2[8], av[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) ak[q] = ak2[q] = av[q] = 0.f;
        for (int s = v.seg[tok0 + j]; s < nseg; ++s) {
            const int64_t base = (v.traj_km[b] + (int64_t)s * nt) * 128;
            const int c = v.cpos[base + j];
            if (c < 0 || !MW_DBG_IN(c, (int64_t)nt * 128, v.status, 202)) continue;
            const float4* pv = reinterpret_cast<const float4*>(dVc + (base + c) * Hkv * DH) + 2 * k;
            const float4 v0 = pv[0], v1 = pv[1];
            av[0] += v0.x; av[1] += v0.y; av[2] += v0.z; av[3] += v0.w;
            av[4] += v1.x; av[5] += v1.y; av[6] += v1.z; av[7] += v1.w;
            if (!kdo) continue;
            const float4* pk = reinterpret_cast<const float4*>(dKc + (base + c) * Hkv * DH);
            const float4 k0 = pk[2 * k], k1 = pk[2 * k + 1];
            const float x0[8] = {k0.x, k0.y, k0.z, k0.w, k1.x, k1.y, k1.z, k1.w};
            if (!rot) {
#pragma unroll
                for (int q = 0; q < 8; ++q) ak[q] += x0[q];
            } else {
                const float4 m0 = pk[2 * kk], m1 = pk[2 * kk + 1];
                const float x1[8] = {m0.x, m0.y, m0.z, m0.w, m1.x, m1.y, m1.z, m1.w};
                const int f0 = 8 * (k & 15);
#pragma unroll
                for (int q = 0; q < 8; ++q) {   // turn back: the transpose of the rotation
                    const float2 cs = table[(int64_t)c * 64 + f0 + q];
                    ak[q] += fmaf(x0[q], cs.x, x1[q] * cs.y);
                    ak2[q] += fmaf(x1[q], cs.x, -x0[q] * cs.y);
                }
            }
        }
        reinterpret_cast<uint4*>(dV + (tok0 + j) * Hkv * DH)[k] =
            make_uint4(pack_bf16(av[0], av[1]), pack_bf16(av[2], av[3]), pack_bf16(av[4], av[5]), pack_bf16(av[6], av[7]));
        if (kdo) {
            reinterpret_cast<uint4*>(dK + (tok0 + j) * Hkv * DH)[k] =
                make_uint4(pack_bf16(ak[0], ak[1]), pack_bf16(ak[2], ak[3]), pack_bf16(ak[4], ak[5]),
                           pack_bf16(ak[6], ak[7]));
            if (rot)
                reinterpret_cast<uint4*>(dK + (tok0 + j) * Hkv * DH)[kk] =
                    make_uint4(pack_bf16(ak2[0], ak2[1]), pack_bf16(ak2[2], ak2[3]), pack_bf16(ak2[4], ak2[5]),
                               pack_bf16(ak2[6], ak2[7]));
        }
    }
}

}  // namespace

// Compact key rows: one 128-row region per (segment, k-tile) entry, of which
// each segment uses its first ceil(|view_s| / 128) tiles.
static int64_t cmp_rows(const mw_vis_layout* L) { return L->n_keymask * 128; }

// Forward workspace: the compact K and V (bf16).
int64_t attn_fwd_tc_ws(const mw_vis_layout* L, int Hkv) { return align256(4 * cmp_rows(L) * Hkv * DH); }

// Backward workspace: the (-LSE2, Delta) pair array, the compact K and V, and
// the float32 dK / dV partials per compact row.
int64_t attn_bwd_tc_ws(const mw_vis_layout* L, int Hq, int Hkv) {
    return align256(8 * L->n_tiles * 128 * (int64_t)Hq) + attn_fwd_tc_ws(L, Hkv) +
           align256(8 * cmp_rows(L) * Hkv * DH);
}

static mw_status cmp_gather(const mw_vis_layout* L, const VisView& v, int Hkv, const void* K, const void* V, void* Kc,
                            void* Vc, const float* table, cudaStream_t s) {
    count_launches(1);
    k_cmp_gather<<<(unsigned)L->n_keymask, 256, 0, s>>>(v, L->n_traj, Hkv, (const __nv_bfloat16*)K,
                                                        (const __nv_bfloat16*)V, (__nv_bfloat16*)Kc,
                                                        (__nv_bfloat16*)Vc, reinterpret_cast<const float2*>(table));
    return launch_status();
}

// Compact forward: gather every segment's view into Kc / Vc (in `ws`), then
// one CTA per (q-tile, segment of its first row, head) plus one per (segment
// starting inside a q-tile, head), each over its segment's compact keys.
mw_status attn_fwd_tc(const mw_vis_layout* L, const void* vis, const void* Q, const void* K, const void* V, void* O,
                      float* LSE, int Hq, int Hkv, float scale, void* ws, cudaStream_t s, const float* table) {
    if (L->n_tiles == 0) return MW_OK;
    if (!cmp_fits(L, Hq)) return MW_ESHAPE;
    const VisView view = make_view(L, vis);
    const int64_t KR = cmp_rows(L);
    void* Kc = ws;
    void* Vc = at<char>(ws, 2 * KR * Hkv * DH);
    mw_status st = cmp_gather(L, view, Hkv, K, V, Kc, Vc, table, s);
    if (st != MW_OK) return st;
    CUtensorMap tq, tk, tv;
    const uint64_t T = (uint64_t)L->total_tokens;
    if (!tmap_bf16_3d(&tq, Q, T, Hq, DH, 128, 64) || !tmap_bf16_3d(&tk, Kc, (uint64_t)KR, Hkv, DH, 128, 64) ||
        !tmap_bf16_3d(&tv, Vc, (uint64_t)KR, Hkv, DH, 128, 64))
        return MW_ECUDA;
    FwdParams p;
    p.v = view;
    p.total = L->total_tokens;
    p.n_traj = L->n_traj;
    p.max_tiles = L->max_tiles;
    p.Hq = Hq;
    p.Hkv = Hkv;
    p.scale_log2 = scale * LOG2E;
    p.O = (__nv_bfloat16*)O;
    p.LSE = LSE;
    p.junction_items = 0;
    if ((st = cuda_status(cudaFuncSetAttribute(k_attn_fwd_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)SMEM_FWD))) != MW_OK)
        return st;
    count_launches(1);
    k_attn_fwd_tc<<<(unsigned)((int64_t)L->max_tiles * L->n_traj * Hq), NT_FWD, SMEM_FWD, s>>>(tq, tk, tv, p);
    if ((st = launch_status()) != MW_OK || L->n_junc == 0) return st;
    p.junction_items = 1;
    count_launches(1);
    k_attn_fwd_tc<<<(unsigned)(L->n_segs * Hq), NT_FWD, SMEM_FWD, s>>>(tq, tk, tv, p);
    return launch_status();
}

// Compact backward: (-LSE2, Delta) pairs, the compact gather, dQ (main +
// junction launches), dK / dV per (compact key tile, segment) into float32
// partials per compact row, and their deterministic sum per key.
mw_status attn_bwd_tc(const mw_vis_layout* L, const void* vis, const void* Q, const void* K, const void* V,
                      const void* O, const void* dO, const float* LSE, void* dQ, void* dK, void* dV, int Hq, int Hkv,
                      float scale, void* ws, cudaStream_t s, const float* table) {
    if (L->n_tiles == 0) return MW_OK;
    if (!cmp_fits(L, Hq)) return MW_ESHAPE;
    const int64_t n_rows = L->n_tiles * 128;
    const int64_t KR = cmp_rows(L);
    float* lsd = reinterpret_cast<float*>(ws);
    void* Kc = at<char>(ws, align256(8 * n_rows * (int64_t)Hq));
    void* Vc = at<char>(Kc, 2 * KR * Hkv * DH);
    float* dKc = at<float>(Kc, attn_fwd_tc_ws(L, Hkv));
    float* dVc = dKc + KR * Hkv * DH;
    const VisView view = make_view(L, vis);
    count_launches(1);
    k_attn_lsd<<<(unsigned)std::min<int64_t>(ceil_div(n_rows * Hq, 8), 152 * 64), 256, 0, s>>>(
        view, L->total_tokens, n_rows, Hq, (const __nv_bfloat16*)O, (const __nv_bfloat16*)dO, LSE, lsd);
    mw_status st = launch_status();
    if (st == MW_OK) st = cmp_gather(L, view, Hkv, K, V, Kc, Vc, table, s);
    if (st != MW_OK) return st;
    const uint64_t T = (uint64_t)L->total_tokens;
    CUtensorMap tq, tdo, tk, tv, tq64, tdo64;
    if (!tmap_bf16_3d(&tq, Q, T, Hq, DH, 128, 64) || !tmap_bf16_3d(&tdo, dO, T, Hq, DH, 128, 64) ||
        !tmap_bf16_3d(&tk, Kc, (uint64_t)KR, Hkv, DH, 128, 64) || !tmap_bf16_3d(&tv, Vc, (uint64_t)KR, Hkv, DH, 128, 64) ||
        !tmap_bf16_3d(&tq64, Q, T, Hq, DH, 64, 64) || !tmap_bf16_3d(&tdo64, dO, T, Hq, DH, 64, 64))
        return MW_ECUDA;
    BwdParams p;
    p.v = view;
    p.total = L->total_tokens;
    p.n_traj = L->n_traj;
    p.max_tiles = L->max_tiles;
    p.Hq = Hq;
    p.Hkv = Hkv;
    p.scale = scale;
    p.scale_log2 = scale * LOG2E;
    p.lsd = lsd;
    p.n_rows = n_rows;
    p.dQ = (__nv_bfloat16*)dQ;
    p.dKseg = dKc;
    p.dVseg = dVc;
    p.junction_items = 0;
    if ((st = cuda_status(cudaFuncSetAttribute(k_attn_dq_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)SMEM_DQ))) != MW_OK)
        return st;
    if ((st = cuda_status(cudaFuncSetAttribute(k_attn_dkdv_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)SMEM_KV))) != MW_OK)
        return st;
    count_launches(1);
    k_attn_dq_tc<<<(unsigned)((int64_t)L->max_tiles * L->n_traj * Hq), NT_BWD, SMEM_DQ, s>>>(tq, tdo, tk, tv, p);
    if ((st = launch_status()) != MW_OK) return st;
    if (L->n_junc > 0) {
        p.junction_items = 1;
        count_launches(1);
        k_attn_dq_tc<<<(unsigned)(L->n_segs * Hq), NT_BWD, SMEM_DQ, s>>>(tq, tdo, tk, tv, p);
        if ((st = launch_status()) != MW_OK) return st;
        p.junction_items = 0;
    }
    const dim3 gk((unsigned)((int64_t)L->max_tiles * L->n_traj * Hkv), (unsigned)L->max_segs);
    count_launches(2);
    k_attn_dkdv_tc<<<gk, NT_BWD, SMEM_KV, s>>>(tq64, tdo64, tk, tv, p);
    k_cmp_reduce<<<(unsigned)L->n_tiles, 256, 0, s>>>(view, Hkv, dKc, dVc, (__nv_bfloat16*)dK, (__nv_bfloat16*)dV,
                                                      reinterpret_cast<const float2*>(table));
    return launch_status();
}

}  // namespace mw
