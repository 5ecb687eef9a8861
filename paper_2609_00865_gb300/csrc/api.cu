// extern "C" entry points of libmw: host-side argument checks and dispatch.
// See include/mw.h for the contract of every function.

#include <algorithm>
#include <math.h>

#include "common.cuh"

namespace mw {
mw_status attn_fwd_simt(const mw_vis_layout*, const void*, const void*, const void*, const void*, void*, float*,
                        int, int, int, int, float, cudaStream_t);
mw_status attn_bwd_simt(const mw_vis_layout*, const void*, const void*, const void*, const void*, const void*,
                        const void*, const float*, void*, void*, void*, int, int, int, int, float, float*,
                        cudaStream_t);
mw_status lm_fwd_simt(const void*, const void*, const int32_t*, const int32_t*, int, int, int, int, int, float*,
                      float*, float*, int32_t*, cudaStream_t);
mw_status lm_bwd_simt(const void*, const void*, const int32_t*, const int32_t*, int, int, int, int, int,
                      const float*, const float*, float, void*, float*, int32_t*, cudaStream_t);
mw_status attn_fwd_tc(const mw_vis_layout*, const void*, const void*, const void*, const void*, void*, float*, int,
                      int, float, void*, cudaStream_t, const float* = nullptr);
mw_status attn_bwd_tc(const mw_vis_layout*, const void*, const void*, const void*, const void*, const void*,
                      const void*, const float*, void*, void*, void*, int, int, float, void*, cudaStream_t,
                      const float* = nullptr);
int64_t attn_fwd_tc_ws(const mw_vis_layout*, int);
int64_t attn_bwd_tc_ws(const mw_vis_layout*, int, int);
mw_status attn_delta(const mw_vis_layout*, const void*, const void*, int, int, int, float*, cudaStream_t);
mw_status attn_fwd_simt_segk(const mw_vis_layout*, const void*, const void*, const void*, const void*, void*, float*,
                             int, int, int, int, float, cudaStream_t);
mw_status attn_bwd_simt_segk(const mw_vis_layout*, const void*, const void*, const void*, const void*, const void*,
                             const float*, const float*, void*, float*, void*, int, int, int, int, float,
                             cudaStream_t);
mw_status logical_positions(const mw_vis_layout*, const void*, int32_t*, cudaStream_t);
mw_status rope_table(int, int, double, float*, cudaStream_t);
mw_status rope_rows(const mw_vis_layout*, const void*, const int32_t*, const float*, int, const void*, void*, int,
                    int, int, bool, cudaStream_t);
mw_status rope_segments(const mw_vis_layout*, const void*, const int32_t*, const float*, int, const void*, void*,
                        int, int, int, cudaStream_t);
mw_status rope_segments_bwd(const mw_vis_layout*, const void*, const int32_t*, const float*, int, const float*,
                            void*, int, int, int, bool, cudaStream_t);
__global__ void k_loss_epilogue(int, const float*, const float*, const float*, float, float, const float*, float, float*,
                                float*, float*);
__global__ void k_logdiff(int, const float*, const float*, float*);

mw_status lm_ref_tc(const void*, const void*, const int32_t*, const int32_t*, int, int, int, int, void*, int32_t*,
                    float2*, float*, float4*, int32_t*, cudaStream_t);

bool lm_bwd_tc_supported(int d);
int64_t lm_bwd_tc_scratch(int M, int d);
int64_t lm_fwd_grp_bytes(int M, int d);
mw_status lm_fwd_grp_tc(const void*, int, int, int, const void*, const int32_t*, float*, float*, float*, int32_t*,
                        void*, void*, cudaStream_t);
mw_status lm_bwd_tc(const void*, int, int, int, int, const int32_t*, const void*, const int32_t*, const float*,
                    const float*, float, void*, float*, int32_t*, void*, void*, cudaStream_t);

// Tensor-core LM-head path: bf16 with d a multiple of 64 that the clustered
// backward can split (d / C <= 448 for a cluster of C <= 8 CTAs).
static bool lm_tc(int d, int dtype) { return dtype == MW_BF16 && d % 64 == 0 && lm_bwd_tc_supported(d); }

// Byte offsets inside the log-prob workspace. The bf16 path keeps, between
// forward and backward: g, the gathered rows (hg, tg) and the fused
// forward's E and 1 / l (fwd); `part` holds the reference prepass's partials,
// `bwd` the group passes' parameters, exchange ring and counters.
struct LmWs {
    int64_t g, zt, hg, tg, part, bwd, fwd, status, bytes;
};
static LmWs lm_ws_layout(int N, int M, int d, int V, int dtype) {
    (void)N; (void)V;
    LmWs w;
    int64_t o = 0;
    const int64_t M_pad = ceil_div(M, 128) * 128;
    w.g = o; o = align256(o + 4 * (int64_t)M);
    w.zt = o; o = align256(o + 4 * (int64_t)M);
    w.status = o; o = align256(o + 32);
    w.hg = w.tg = w.part = w.bwd = w.fwd = o;
    if (lm_tc(d, dtype)) {
        w.hg = o; o = align256(o + 2 * M_pad * d);
        w.tg = o; o = align256(o + 4 * M_pad);
        w.part = o; o = align256(o + 8 * 64 * M_pad);
        w.bwd = o; o = align256(o + lm_bwd_tc_scratch(M, d));
        w.fwd = o; o = align256(o + lm_fwd_grp_bytes(M, d));
    }
    w.bytes = o;
    return w;
}

static mw_status attn_args(const mw_vis_layout* L, const void* vis, int Hq, int Hkv, int Dh, int dtype,
                           float scale) {
    if (!L) return MW_EINVAL;
    if (L->total_tokens > 0 && !vis) return MW_EINVAL;
    if (dtype != MW_F32 && dtype != MW_BF16) return MW_EDTYPE;
    if (Hq <= 0 || Hkv <= 0 || Hq % Hkv != 0) return MW_ESHAPE;
    if (!(Dh == 64 || Dh == 128)) return MW_ESHAPE;
    if (!(scale > 0.f) || !isfinite(scale)) return MW_EINVAL;
    return MW_OK;
}

}  // namespace mw

using namespace mw;

extern "C" mw_status mw_masked_attn_fwd_ws(const mw_vis_layout* L, int Hkv, int Dh, int dtype, size_t* bytes) {
    if (!L || !bytes) return MW_EINVAL;
    if (Hkv <= 0) return MW_ESHAPE;
    *bytes = dtype == MW_BF16 && Dh == 128 ? (size_t)attn_fwd_tc_ws(L, Hkv) : 0;
    return MW_OK;
}

extern "C" mw_status mw_masked_attn_fwd(const mw_vis_layout* L, const void* vis, const void* Q, const void* K,
                                        const void* V, void* O, float* LSE, int Hq, int Hkv, int Dh, int dtype,
                                        float scale, void* ws, void* stream) {
    mw_status st = attn_args(L, vis, Hq, Hkv, Dh, dtype, scale);
    if (st != MW_OK) return st;
    // views of an EVENTS record have no tile lists: only the compact path reads them
    if (L->kind != MW_VIEWS_EDITS && !(dtype == MW_BF16 && Dh == 128)) return MW_ESHAPE;
    if (L->total_tokens == 0) return MW_OK;
    if (!Q || !K || !V || !O || !LSE) return MW_EINVAL;
    if (dtype == MW_BF16 && Dh == 128) {
        if (!ws) return MW_EINVAL;
        return attn_fwd_tc(L, vis, Q, K, V, O, LSE, Hq, Hkv, scale, ws, (cudaStream_t)stream);
    }
    return attn_fwd_simt(L, vis, Q, K, V, O, LSE, Hq, Hkv, Dh, dtype, scale, (cudaStream_t)stream);
}

extern "C" mw_status mw_masked_attn_bwd_ws(const mw_vis_layout* L, int Hq, int Hkv, int Dh, int dtype,
                                           size_t* bytes) {
    if (!L || !bytes) return MW_EINVAL;
    if (Hq <= 0 || Hkv <= 0) return MW_ESHAPE;
    int64_t b = 4 * L->total_tokens * (int64_t)Hq;   // Delta per (head, row)
    if (dtype == MW_BF16 && Dh == 128) b = std::max(b, attn_bwd_tc_ws(L, Hq, Hkv));
    *bytes = (size_t)align256(b);
    return MW_OK;
}

extern "C" mw_status mw_masked_attn_bwd(const mw_vis_layout* L, const void* vis, const void* Q, const void* K,
                                        const void* V, const void* O, const void* dO, const float* LSE, void* dQ,
                                        void* dK, void* dV, int Hq, int Hkv, int Dh, int dtype, float scale,
                                        void* ws, void* stream) {
    mw_status st = attn_args(L, vis, Hq, Hkv, Dh, dtype, scale);
    if (st != MW_OK) return st;
    // views of an EVENTS record have no tile lists: only the compact path reads them
    if (L->kind != MW_VIEWS_EDITS && !(dtype == MW_BF16 && Dh == 128)) return MW_ESHAPE;
    if (L->total_tokens == 0) return MW_OK;
    if (!Q || !K || !V || !O || !dO || !LSE || !dQ || !dK || !dV || !ws) return MW_EINVAL;
    if (dtype == MW_BF16 && Dh == 128)
        return attn_bwd_tc(L, vis, Q, K, V, O, dO, LSE, dQ, dK, dV, Hq, Hkv, scale, ws, (cudaStream_t)stream);
    return attn_bwd_simt(L, vis, Q, K, V, O, dO, LSE, dQ, dK, dV, Hq, Hkv, Dh, dtype, scale, (float*)ws,
                         (cudaStream_t)stream);
}

static mw_status lm_args(int N, int M, int d, int V, int dtype) {
    if (N < 0 || M < 0 || d <= 0 || V <= 0) return MW_ESHAPE;
    if (M > N) return MW_ESHAPE;
    if (dtype != MW_F32 && dtype != MW_BF16) return MW_EDTYPE;
    if (!lm_tc(d, dtype) && d > 256) return MW_ESHAPE;
    return MW_OK;
}

extern "C" mw_status mw_logprob_ws(int N, int M, int d, int V, int dtype, size_t* bytes) {
    if (!bytes) return MW_EINVAL;
    mw_status st = lm_args(N, M, d, V, dtype);
    if (st != MW_OK) return st;
    *bytes = (size_t)lm_ws_layout(N, M, d, V, dtype).bytes;
    return MW_OK;
}

extern "C" mw_status mw_logprob_loss_fwd_kl(const void* H, const void* W, const int32_t* targets,
                                            const int32_t* rows, int M, const float* lp_old, const float* adv,
                                            float eps_lo, float eps_hi, const float* lp_ref, float beta, int N, int d,
                                            int V, int dtype, float* lp, float* ratio, float* lse, float* loss,
                                            void* ws, void* stream) {
    mw_status st = lm_args(N, M, d, V, dtype);
    if (st != MW_OK) return st;
    if (!(eps_lo >= 0.f && eps_lo < 1.f && eps_hi >= 0.f && isfinite(eps_hi))) return MW_EINVAL;
    if (!(beta >= 0.f && isfinite(beta))) return MW_EINVAL;
    if (beta > 0.f && M > 0 && !lp_ref) return MW_EINVAL;
    if (beta == 0.f) lp_ref = nullptr;
    if (!loss || !ws) return MW_EINVAL;
    if (M > 0 && (!H || !W || !targets || !rows || !lp_old || !adv || !lp || !ratio || !lse)) return MW_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    LmWs w = lm_ws_layout(N, M, d, V, dtype);
    float* g = at<float>(ws, w.g);
    float* zt = at<float>(ws, w.zt);
    int32_t* status = at<int32_t>(ws, w.status);
    if ((st = cuda_status(cudaMemsetAsync(status, 0, 32, s))) != MW_OK) return st;
    if (lm_tc(d, dtype)) {
        // references from the first vocabulary entries, then the fused pass
        // over the whole vocabulary (lse, lp, and E for the backward)
        st = lm_ref_tc(H, W, targets, rows, M, N, d, V, at<char>(ws, w.hg), at<int32_t>(ws, w.tg),
                       at<float2>(ws, w.part), zt, at<float4>(ws, w.bwd), status, s);
        if (st == MW_OK)
            st = lm_fwd_grp_tc(W, M, d, V, at<char>(ws, w.hg), at<int32_t>(ws, w.tg), zt, lse, lp, status,
                               at<char>(ws, w.bwd), at<char>(ws, w.fwd), s);
    } else {
        st = lm_fwd_simt(H, W, targets, rows, M, N, d, V, dtype, lse, zt, lp, status, s);
    }
    if (st != MW_OK) return st;
    count_launches(1);
    k_loss_epilogue<<<1, 1024, 0, s>>>(M, lp, lp_old, adv, eps_lo, eps_hi, lp_ref, beta, ratio, g, loss);
    return launch_status();
}

extern "C" mw_status mw_logprob_loss_fwd(const void* H, const void* W, const int32_t* targets, const int32_t* rows,
                                         int M, const float* lp_old, const float* adv, float eps_lo, float eps_hi,
                                         int N, int d, int V, int dtype, float* lp, float* ratio, float* lse,
                                         float* loss, void* ws, void* stream) {
    return mw_logprob_loss_fwd_kl(H, W, targets, rows, M, lp_old, adv, eps_lo, eps_hi, nullptr, 0.f, N, d, V, dtype,
                                  lp, ratio, lse, loss, ws, stream);
}

extern "C" mw_status mw_logprob_loss_bwd(const void* H, const void* W, const int32_t* targets, const int32_t* rows,
                                         int M, int N, int d, int V, int dtype, const float* lse, void* ws,
                                         float dloss, void* dH, float* dW, void* stream) {
    mw_status st = lm_args(N, M, d, V, dtype);
    if (st != MW_OK) return st;
    if (!isfinite(dloss)) return MW_EINVAL;
    if (!ws || !dW || (N > 0 && !dH)) return MW_EINVAL;
    if (M > 0 && (!H || !W || !targets || !rows || !lse)) return MW_EINVAL;
    LmWs w = lm_ws_layout(N, M, d, V, dtype);
    // the backward reads the forward's g (and on the tensor cores its gathered
    // rows, E and 1 / l); it adds to the status words the forward reset, so
    // a forward that gave up a wait ends the backward's waits at once
    int32_t* status = at<int32_t>(ws, w.status);
    if (lm_tc(d, dtype))
        return lm_bwd_tc(W, M, N, d, V, rows, at<char>(ws, w.hg), at<int32_t>(ws, w.tg), lse, at<float>(ws, w.g),
                         dloss, dH, dW, status, at<char>(ws, w.bwd), at<char>(ws, w.fwd), (cudaStream_t)stream);
    return lm_bwd_simt(H, W, targets, rows, M, N, d, V, dtype, lse, at<float>(ws, w.g), dloss, dH, dW, status,
                       (cudaStream_t)stream);
}

extern "C" mw_status mw_logdiff(const float* lp_train, const float* lp_rollout, int M, float* out, void* stream) {
    if (M < 0) return MW_ESHAPE;
    if (!out || (M > 0 && (!lp_train || !lp_rollout))) return MW_EINVAL;
    count_launches(1);
    k_logdiff<<<1, 1024, 0, (cudaStream_t)stream>>>(M, lp_train, lp_rollout, out);
    return launch_status();
}

extern "C" mw_status mw_logprob_check_status(int N, int M, int d, int V, int dtype, const void* ws, void* stream) {
    mw_status st = lm_args(N, M, d, V, dtype);
    if (st != MW_OK) return st;
    if (!ws) return MW_EINVAL;
    // timeouts come from the tensor-core kernels' barrier waits; both paths
    // raise the bounds flag for a loss row or target out of range
    LmWs w = lm_ws_layout(N, M, d, V, dtype);
    int32_t h[8];
    if ((st = cuda_status(cudaMemcpyAsync(h, at<char>(ws, w.status), sizeof(h), cudaMemcpyDeviceToHost,
                                          (cudaStream_t)stream))) != MW_OK)
        return st;
    if ((st = cuda_status(cudaStreamSynchronize((cudaStream_t)stream))) != MW_OK) return st;
    return h[1] ? MW_ETIMEOUT : h[0] ? MW_EDEVICE : MW_OK;
}

// --- row-wise logical positions and rotary attention (§4.2) -----------------

// The rotary attention's tensor-core path: bf16 with head dim 128, as the
// plain attention's.
static bool rope_tc(int Dh, int dtype) { return dtype == MW_BF16 && Dh == 128; }

// Byte offsets inside the rotary-attention workspace. Tensor-core path: the
// rotated queries, then the compact attention's own workspace (its keys are
// turned by rank as they are gathered). CUDA-core path: the rotated queries,
// the segment key rows, then (backward only) Delta and the float32 gradient
// of the segment key rows.
struct RopeWs {
    int64_t q, kseg, delta, dkseg, fwd_bytes, bwd_bytes;
};
static RopeWs rope_ws_layout(const mw_vis_layout* L, int Hq, int Hkv, int Dh, int dtype) {
    RopeWs w;
    const int64_t esz = dtype == MW_F32 ? 4 : 2;
    const int64_t krows = L->n_keymask * MW_TILE;
    const bool tc = rope_tc(Dh, dtype);
    int64_t o = 0;
    if (tc) {   // rotated queries, then the compact attention's own workspace (keys rotated by rank)
        w.q = o; o = align256(o + esz * L->total_tokens * Hq * Dh);
        w.kseg = w.delta = w.dkseg = o;
        w.fwd_bytes = o + attn_fwd_tc_ws(L, Hkv);
        w.bwd_bytes = o + attn_bwd_tc_ws(L, Hq, Hkv);
        return w;
    }
    w.q = o; o = align256(o + esz * L->total_tokens * Hq * Dh);
    w.kseg = o; o = align256(o + esz * krows * Hkv * Dh);
    w.fwd_bytes = o;
    w.delta = o; o = align256(o + 4 * L->total_tokens * Hq);
    w.dkseg = o; o = align256(o + 4 * krows * Hkv * Dh);
    w.bwd_bytes = o;
    return w;
}

static mw_status rope_args(const mw_vis_layout* L, const void* vis, const int32_t* pos, const float* table,
                           int n_pos) {
    if (!L) return MW_EINVAL;
    if (L->total_tokens == 0) return MW_OK;
    if (!vis || !pos || !table) return MW_EINVAL;
    if (n_pos < MW_TILE * (int64_t)L->max_tiles) return MW_ESHAPE;   // every position < T_b <= 128 nt_b
    return MW_OK;
}

extern "C" mw_status mw_logical_positions(const mw_vis_layout* L, const void* vis, int32_t* pos, void* stream) {
    if (!L) return MW_EINVAL;
    if (L->n_keymask == 0) return MW_OK;
    if (!vis || !pos) return MW_EINVAL;
    if (L->kind != MW_VIEWS_EDITS)   // views in list order: the positions are the build's ranks
        return cuda_status(cudaMemcpyAsync(pos, at<char>(vis, L->off_cpos), 4 * MW_TILE * (size_t)L->n_keymask,
                                           cudaMemcpyDeviceToDevice, (cudaStream_t)stream));
    return logical_positions(L, vis, pos, (cudaStream_t)stream);
}

extern "C" mw_status mw_rope_table(int n_pos, int Dh, double theta, float* table, void* stream) {
    if (n_pos < 0 || Dh <= 0 || Dh % 2 != 0) return MW_ESHAPE;
    if (!(theta > 0.0) || !isfinite(theta)) return MW_EINVAL;
    if (n_pos > 0 && !table) return MW_EINVAL;
    return rope_table(n_pos, Dh, theta, table, (cudaStream_t)stream);
}

extern "C" mw_status mw_rope_rows(const mw_vis_layout* L, const void* vis, const int32_t* pos, const float* table,
                                  int n_pos, const void* X, void* Y, int H, int Dh, int dtype, int inverse,
                                  void* stream) {
    if (dtype != MW_F32 && dtype != MW_BF16) return MW_EDTYPE;
    if (H <= 0 || Dh <= 0 || Dh % 2 != 0) return MW_ESHAPE;
    mw_status st = rope_args(L, vis, pos, table, n_pos);
    if (st != MW_OK || L->total_tokens == 0) return st;
    if (!X || !Y) return MW_EINVAL;
    return rope_rows(L, vis, pos, table, n_pos, X, Y, H, Dh, dtype, inverse != 0, (cudaStream_t)stream);
}

extern "C" mw_status mw_masked_attn_rope_ws(const mw_vis_layout* L, int Hq, int Hkv, int Dh, int dtype,
                                            size_t* fwd_bytes, size_t* bwd_bytes) {
    if (!L || !fwd_bytes || !bwd_bytes) return MW_EINVAL;
    if (dtype != MW_F32 && dtype != MW_BF16) return MW_EDTYPE;
    if (Hq <= 0 || Hkv <= 0 || Hq % Hkv != 0 || !(Dh == 64 || Dh == 128)) return MW_ESHAPE;
    RopeWs w = rope_ws_layout(L, Hq, Hkv, Dh, dtype);
    *fwd_bytes = (size_t)w.fwd_bytes;
    *bwd_bytes = (size_t)w.bwd_bytes;
    return MW_OK;
}

extern "C" mw_status mw_masked_attn_rope_fwd(const mw_vis_layout* L, const void* vis, const int32_t* pos,
                                             const float* table, int n_pos, const void* Q, const void* K,
                                             const void* V, void* O, float* LSE, int Hq, int Hkv, int Dh, int dtype,
                                             float scale, void* ws, void* stream) {
    // views of an EVENTS record have no tile lists: only the compact path reads them
    if (L && L->kind != MW_VIEWS_EDITS && !rope_tc(Dh, dtype)) return MW_ESHAPE;
    mw_status st = attn_args(L, vis, Hq, Hkv, Dh, dtype, scale);
    if (st != MW_OK) return st;
    if ((st = rope_args(L, vis, pos, table, n_pos)) != MW_OK) return st;
    if (L->total_tokens == 0) return MW_OK;
    if (!Q || !K || !V || !O || !LSE || !ws) return MW_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    RopeWs w = rope_ws_layout(L, Hq, Hkv, Dh, dtype);
    void* q = at<char>(ws, w.q);
    void* kseg = at<char>(ws, w.kseg);
    if ((st = rope_rows(L, vis, pos, table, n_pos, Q, q, Hq, Dh, dtype, false, s)) != MW_OK) return st;
    // compact path: each key turned by its rank in the segment's view (its logical position) as it is gathered
    if (rope_tc(Dh, dtype)) return attn_fwd_tc(L, vis, q, K, V, O, LSE, Hq, Hkv, scale, kseg, s, table);
    if ((st = rope_segments(L, vis, pos, table, n_pos, K, kseg, Hkv, Dh, dtype, s)) != MW_OK) return st;
    return attn_fwd_simt_segk(L, vis, q, kseg, V, O, LSE, Hq, Hkv, Dh, dtype, scale, s);
}

extern "C" mw_status mw_masked_attn_rope_bwd(const mw_vis_layout* L, const void* vis, const int32_t* pos,
                                             const float* table, int n_pos, const void* Q, const void* K,
                                             const void* V, const void* O, const void* dO, const float* LSE,
                                             void* dQ, void* dK, void* dV, int Hq, int Hkv, int Dh, int dtype,
                                             float scale, void* ws, void* stream) {
    if (L && L->kind != MW_VIEWS_EDITS && !rope_tc(Dh, dtype)) return MW_ESHAPE;
    mw_status st = attn_args(L, vis, Hq, Hkv, Dh, dtype, scale);
    if (st != MW_OK) return st;
    if ((st = rope_args(L, vis, pos, table, n_pos)) != MW_OK) return st;
    if (L->total_tokens == 0) return MW_OK;
    if (!Q || !K || !V || !O || !dO || !LSE || !dQ || !dK || !dV || !ws) return MW_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    RopeWs w = rope_ws_layout(L, Hq, Hkv, Dh, dtype);
    void* q = at<char>(ws, w.q);
    void* kseg = at<char>(ws, w.kseg);
    float* delta = at<float>(ws, w.delta);
    float* dkseg = at<float>(ws, w.dkseg);
    if ((st = rope_rows(L, vis, pos, table, n_pos, Q, q, Hq, Dh, dtype, false, s)) != MW_OK) return st;
    // dQ first holds the gradient of the rotated queries, then is turned back in place
    if (rope_tc(Dh, dtype)) {
        // compact path: keys turned by rank as they are gathered, dK partials turned back as they are summed
        if ((st = attn_bwd_tc(L, vis, q, K, V, O, dO, LSE, dQ, dK, dV, Hq, Hkv, scale, kseg, s, table)) != MW_OK)
            return st;
        return rope_rows(L, vis, pos, table, n_pos, dQ, dQ, Hq, Dh, dtype, true, s);
    }
    if ((st = rope_segments(L, vis, pos, table, n_pos, K, kseg, Hkv, Dh, dtype, s)) != MW_OK) return st;
    if ((st = attn_delta(L, O, dO, Hq, Dh, dtype, delta, s)) != MW_OK) return st;
    if ((st = attn_bwd_simt_segk(L, vis, q, kseg, V, dO, LSE, delta, dQ, dkseg, dV, Hq, Hkv, Dh, dtype, scale, s)) !=
        MW_OK)
        return st;
    if ((st = rope_rows(L, vis, pos, table, n_pos, dQ, dQ, Hq, Dh, dtype, true, s)) != MW_OK) return st;
    return rope_segments_bwd(L, vis, pos, table, n_pos, dkseg, dK, Hkv, Dh, dtype, true, s);
}
