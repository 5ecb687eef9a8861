/*
 * mw.h -- C ABI of libmw: view-consistent scoring of compressed agent rollouts
 * on one GB300 (sm_103a).
 *
 * Method: MemoryWalker (arXiv 2609.00865). Every generated token of an edited
 * (compressed) rollout is scored under the live context view the policy held
 * when it decoded that token (§3.2 live-view equation; §3.3 conditioning
 * invariant), using the packed 4D-mask form of §4.2 on the physical union of
 * all tokens, which Theorem "materialization equivalence" (§4.3) equates with
 * per-branch LogitTree forwards (§4.1).
 *
 * Conventions shared by every entry point
 * ----------------------------------------
 *  - Trajectories are packed back to back. cu_seqlens[n_traj+1] (host int32)
 *    holds their token offsets; T_b = cu_seqlens[b+1] - cu_seqlens[b].
 *  - Positions inside a trajectory are 0-based (the prompt starts at 0). The
 *    k-th edit of a trajectory fires at junction J_k = the physical index of
 *    the last token that existed before the edit; every row i >= J_k is scored
 *    under the post-edit view (App. B.4 Table "running-prefixes" pins this).
 *    Row i predicts token i+1.
 *  - Key j is visible to row i iff j <= i < omega(j), where omega(j) is the
 *    smallest junction whose evicted set contains j (never evicted: INT32_MAX)
 *    (§4.2, the M = M^causal (+) M^logical equation with lifetime [j, omega(j))).
 *    Inserted summary tokens are ordinary physical tokens placed after their
 *    junction, so causality alone hides them from earlier rows.
 *  - Tiles are 128 x 128, trajectory-local, the last one ragged. Class EMPTY
 *    (no visible in-range pair), FULL (all in-range pairs visible) or PARTIAL.
 *    Tile-list entries are int32 (tile << 4) | code, code = class plus the
 *    MW_TILE_DEAD_* bits (see below).
 *  - Every device pointer is caller-owned device memory (the library never
 *    allocates device memory, never frees, never synchronises a stream except
 *    where stated). Host pointers are read during the call only.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *  - Errors are returned as mw_status; nothing is thrown across the ABI. All
 *    argument checks run on the host before any launch; on error nothing is
 *    launched. MW_ECUDA reports a failed launch or copy (the CUDA error is
 *    available through mw_last_cuda_error()).
 */
#ifndef MW_H_
#define MW_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum mw_status {
    MW_OK = 0,
    MW_EINVAL = 1,    /* null pointer, negative size or bad scalar */
    MW_EEDITS = 2,    /* record breaks the junction / span conventions */
    MW_ESHAPE = 3,    /* unsupported or inconsistent shape */
    MW_EDTYPE = 4,    /* unsupported dtype code */
    MW_ECUDA = 5,     /* a CUDA runtime call failed */
    MW_ETIMEOUT = 6,  /* a bounded device-side wait gave up (status word) */
    MW_EDEVICE = 7,   /* a device-side consistency check failed (status word) */
    MW_ENOSPACE = 8   /* request exceeds a fixed capacity */
} mw_status;

enum { MW_F32 = 0, MW_BF16 = 1 };
enum { MW_TILE = 128 };
enum { MW_TILE_EMPTY = 0, MW_TILE_PARTIAL = 1, MW_TILE_FULL = 2 };
/* Beside its class (bits 0-1), a PARTIAL off-diagonal tile carries DEAD_LO
 * (bit 2) when no row of its q-tile sees any of the k-tile's keys 0..63, and
 * DEAD_HI (bit 3) for keys 64..127 (every key of that half evicted before the
 * q-tile starts, or past the trajectory's end). At most one is set. */
enum { MW_TILE_DEAD_LO = 4, MW_TILE_DEAD_HI = 8 };

/* Human-readable name of a status code (static string). */
const char* mw_status_str(int status);
/* Last CUDA error code seen by the library on this host thread (0 if none). */
int mw_last_cuda_error(void);
/* ABI version of this header (bumped on any signature or layout change). */
int mw_abi_version(void);
/* How this library was built: MW_BUILD_DEBUG set for libmw_debug.so, whose
 * kernels check the indices they read from memory (a record's spans, the
 * compact maps, segment tables, tile lists) against the arrays they address;
 * an index out of range is not followed and the status check of the call
 * (mw_check_status for the visibility-based calls) reports MW_EDEVICE. The
 * arithmetic is the release library's. */
#define MW_BUILD_DEBUG 1
int mw_build_flags(void);
/* Number of CUDA kernels this library has launched in this process so far
 * (all threads, all devices); lets callers count launches in a timed region. */
uint64_t mw_kernel_launches(void);

/*
 * Visibility layout: sizes and byte offsets of every array inside the
 * caller-allocated device buffer `vis` (vis_bytes) and of the build
 * workspace `ws` (ws_bytes). All offsets are multiples of 256.
 */
typedef struct mw_vis_layout {
    int32_t n_traj;
    int32_t n_junc;
    int32_t n_spans;
    int32_t max_tiles;      /* max over trajectories of ceil(T_b / 128) */
    int64_t total_tokens;   /* sum T_b */
    int64_t n_tiles;        /* sum ceil(T_b / 128): q-tiles == k-tiles */
    int64_t n_tri;          /* sum nt_b (nt_b + 1) / 2: tile pairs kt <= qt */
    int64_t n_segs;         /* n_traj + n_junc */
    int64_t n_keymask;      /* sum (1 + K_b) nt_b keymask entries */
    /* --- arrays in `vis` (byte offsets) --- */
    int64_t off_omega;      /* int32 [total_tokens] lifetime end, traj-local */
    int64_t off_seg;        /* int32 [total_tokens] segment id of each row */
    int64_t off_traj_tok;   /* int32 [n_traj + 1] token offset of each traj */
    int64_t off_traj_tile;  /* int32 [n_traj + 1] first global tile of each traj */
    int64_t off_traj_seg;   /* int32 [n_traj + 1] first global segment of each traj */
    int64_t off_traj_tri;   /* int64 [n_traj + 1] first triangle entry of each traj */
    int64_t off_traj_km;    /* int64 [n_traj + 1] first keymask entry of each traj */
    int64_t off_seg_start;  /* int32 [n_segs] first row of each segment (0, J_1..J_K per traj) */
    int64_t off_tile_traj;  /* int32 [n_tiles] trajectory of each global tile */
    int64_t off_cls;        /* uint8 [n_tri] class of (qt, kt), index qt(qt+1)/2 + kt */
    int64_t off_fwd_ptr;    /* int32 [n_tiles + 1] per global q-tile */
    int64_t off_fwd_idx;    /* int32 [n_tri] ascending k-tiles (capacity n_tri) */
    int64_t off_bwd_ptr;    /* int32 [n_tiles + 1] per global k-tile */
    int64_t off_bwd_idx;    /* int32 [n_tri] ascending q-tiles (capacity n_tri) */
    int64_t off_pairs;      /* int64 [n_traj + 1] visible pairs per traj, then total */
    int64_t off_keymask;    /* uint32 [n_keymask][4] per (segment, k-tile) view bits */
    int64_t off_status;     /* int32 [8] device status words (0 = ok) */
    int64_t vis_bytes;
    /* --- arrays in `ws` (build workspace; byte offsets) --- */
    int64_t ws_off_spans;   /* int32 [n_spans][3] (global a, global b, J) */
    int64_t ws_off_tstat;   /* int32 [n_tiles][2] per k-tile min / max lifetime */
    int64_t ws_off_cnt;     /* int32 [2][n_tiles] fwd / bwd list lengths */
    int64_t ws_bytes;
    int64_t max_segs;       /* max over trajectories of 1 + K_b (segments per trajectory) */
    /* --- compact views (in `vis`; byte offsets). Segment s of trajectory b
     * owns the 128 nt_b entries starting at (traj_km[b] + s nt_b) 128, the
     * same indexing as the keymask entries times 128. --- */
    int64_t off_seg_len;    /* int32 [n_segs] |view_s|, the length of each segment's compact sequence */
    int64_t off_cpos;       /* int32 [n_keymask][128] rank of key j in view_s (the compact index), -1 if absent */
    int64_t off_csrc;       /* int32 [n_keymask][128] key (traj-local) at compact index c of view_s;
                               -1 from |view_s| to the end of its last 128-entry tile, unset after */
    int64_t kind;           /* MW_VIEWS_EDITS (mw_visibility_layout) or MW_VIEWS_EVENTS (mw_events_layout) */
} mw_vis_layout;

/* Record kinds. EDITS: each edit only evicts (one lifetime interval per key),
 * every array of `vis` is built. EVENTS: an edit may also bring earlier
 * evicted spans back (offload / retrieve), so a view is an ordered list that
 * need not follow physical order; `vis` then holds the segments, the compact
 * views (seg_len, cpos, csrc), the view bits and the pair counts, and no
 * lifetimes (omega reads INT32_MAX), tile classes or tile lists (empty). */
enum { MW_VIEWS_EDITS = 0, MW_VIEWS_EVENTS = 1 };

/*
 * Fill `out` for a record shape. Host-only; launches nothing.
 *   n_traj >= 0; cu_seqlens[n_traj+1] non-decreasing from 0;
 *   junc_traj[n_junc] non-decreasing in [0, n_traj); n_spans >= 0.
 * Returns MW_EINVAL / MW_EEDITS on malformed input.
 */
mw_status mw_visibility_layout(int n_traj, const int32_t* cu_seqlens, int n_junc,
                               const int32_t* junc_traj, int n_spans, mw_vis_layout* out);

/*
 * Layout of an EVENTS record (offload / retrieve): the same shape arguments as
 * mw_visibility_layout, n_spans counting out- and in-spans together. Sets
 * kind = MW_VIEWS_EVENTS and sizes the build workspace for the event replay.
 */
mw_status mw_events_layout(int n_traj, const int32_t* cu_seqlens, int n_junc, const int32_t* junc_traj,
                           int n_spans, mw_vis_layout* out);

/*
 * Views of an EVENTS record (the paper's MemexRL harness, App. F: offload
 * evicts a span, retrieve brings it back). Event k fires at junction J_k like
 * an edit (rows i >= J_k see the post-event view): first the out-spans
 * spans[out_off[k] .. out_off[k+1]) leave the view, then the in-spans
 * spans[in_off[k] .. in_off[k+1]) -- positions out of the view at J_k --
 * re-enter at its end in the given order, before the segment's own rows
 * (the harness figure's MemexRL panel draws retrieved tokens after the ones
 * decoded meanwhile). A row sees the members of its segment's list up to and
 * including itself.
 *   junctions, junc_traj as for mw_build_visibility; out_off, in_off host
 *   int32 [n_junc + 1] (CSR into spans, non-decreasing, within [0, n_spans]);
 *   spans host int32 [n_spans][2] half-open [a, b) with 0 <= a < b <= J_k.
 * MW_EEDITS if a retrieved position is not out of the view when its event
 * fires, or on any convention of mw_build_visibility. `layout` must come from
 * mw_events_layout; `ws` and `vis` as for mw_build_visibility. The masked
 * attention (bf16, Dh 128) accepts such views; entry points that need
 * single-interval lifetimes return MW_ESHAPE for them.
 */
mw_status mw_build_views_events(const mw_vis_layout* layout, const int32_t* cu_seqlens, int n_junc,
                                const int32_t* junctions, const int32_t* junc_traj, const int32_t* out_off,
                                const int32_t* in_off, const int32_t* spans, void* ws, void* vis, void* stream);

/*
 * Build every visibility artefact of a record (§4.2 lifetimes; App. B.1
 * segments) into `vis` (layout->vis_bytes, device) using `ws`
 * (layout->ws_bytes, device). Both must be 256-byte aligned (every array of
 * the layout sits at a 256-byte offset; cudaMalloc's alignment suffices), else
 * MW_EINVAL.
 *   junctions[n_junc]      host int32, traj-local J_k, strictly ascending
 *                          within a trajectory, 1 <= J_k <= T_b - 1
 *   junc_traj[n_junc]      host int32, owning trajectory, non-decreasing
 *   junc_span_off[n_junc+1] host int32 CSR offsets into spans
 *   spans[n_spans][2]      host int32 half-open [a, b), 0 <= a < b <= J_k
 * The record is validated on the host (MW_EEDITS) and packed into one of two
 * page-locked, device-mapped host buffers the library keeps per device (grown
 * as records grow, kept for the life of the process); a kernel on `stream`
 * reads it into place over the host link (no copy engine, no host-side
 * staging copy). Before a buffer is reused, the call waits for the build that
 * last used it, so the host runs at most two builds ahead of the GPU.
 * Everything else runs asynchronously. (mw_build_visibility_noalloc copies
 * from pageable memory.)
 */
mw_status mw_build_visibility(const mw_vis_layout* layout, const int32_t* cu_seqlens,
                              int n_junc, const int32_t* junctions, const int32_t* junc_traj,
                              const int32_t* junc_span_off, const int32_t* spans,
                              void* ws, void* vis, void* stream);

/*
 * Same result as mw_build_visibility, but allocation-free: for callers that
 * are handed their input and output buffers and may not allocate device
 * memory (e.g. a plugin inside a host framework that owns all device memory
 * through its own pool, where cudaMalloc would synchronise the device or
 * bypass the pool's accounting). The paper has no counterpart; this is a
 * library convenience.
 *   The build workspace is a fixed 1 MiB device array inside libmw, resident
 *   on every GPU that loads the library until process exit. Records whose
 *   layout->ws_bytes exceeds 1 MiB are rejected with MW_ENOSPACE (nothing is
 *   launched). The first call on a device looks up the array's address with
 *   that device current. With CUDA's lazy module loading (the default) that
 *   first lookup also loads libmw's device code on the device, which places
 *   the fixed array and may synchronise the device: make one warm-up call at
 *   set-up time, before any stream capture. The address is kept for the life
 *   of the process; after cudaDeviceReset on a device it is stale, so a
 *   process that resets a device must not call this entry point on it again.
 *   All calls on a device share the array: calls whose GPU work overlaps
 *   (other streams or threads) race and must be serialised by the caller.
 *   The caller still provides `vis` (layout->vis_bytes, device). No device
 *   memory is allocated or freed.
 */
mw_status mw_build_visibility_noalloc(const mw_vis_layout* layout, const int32_t* cu_seqlens,
                                      int n_junc, const int32_t* junctions, const int32_t* junc_traj,
                                      const int32_t* junc_span_off, const int32_t* spans,
                                      void* vis, void* stream);

/* Bytes of device workspace mw_masked_attn_fwd needs for these sizes (0 for
 * the fp32 path). bf16 with Dh 128: the compact K and V, 2 x 2 bytes per
 * element of [128 n_keymask, Hkv, Dh]. */
mw_status mw_masked_attn_fwd_ws(const mw_vis_layout* layout, int Hkv, int Dh, int dtype, size_t* ws_bytes);

/*
 * Eviction-aware masked GQA attention forward (§4.2 mask; §4.3 equivalence).
 *   Q, O  [total_tokens, Hq, Dh]   K, V [total_tokens, Hkv, Dh]   (dtype)
 *   LSE   [Hq, total_tokens] float32, natural-log row log-sum-exp (saved for bwd)
 *   O_i = sum_{j visible} softmax_j(scale q_i . k_j) v_j;  q-head h reads
 *   kv-head h / (Hq / Hkv).
 * dtype MW_BF16 requires Dh == 128 (tensor-core path); MW_F32 accepts Dh 64
 * or 128 (exact-fp32 SIMT path, which visits the non-EMPTY tiles of the
 * lists). Hq % Hkv == 0.
 * The bf16 path gathers each segment's live view into its compact sequence
 * (the segment's view_s in order, as §4.1 materialises a branch; the compact
 * maps of `vis`) in `ws` (mw_masked_attn_fwd_ws bytes, device, overwritten)
 * and runs causal attention of the segment's rows over it; a q-tile holding
 * rows of several segments is computed once per segment.
 */
mw_status mw_masked_attn_fwd(const mw_vis_layout* layout, const void* vis,
                             const void* Q, const void* K, const void* V, void* O, float* LSE,
                             int Hq, int Hkv, int Dh, int dtype, float scale, void* ws, void* stream);

/* Bytes of device workspace mw_masked_attn_bwd needs for these sizes. */
mw_status mw_masked_attn_bwd_ws(const mw_vis_layout* layout, int Hq, int Hkv, int Dh, int dtype,
                                size_t* ws_bytes);

/*
 * Backward of mw_masked_attn_fwd for upstream dO (same layout as O).
 * Writes dQ (like Q), dK, dV (like K, V), all in `dtype`, overwriting them.
 * `ws` (mw_masked_attn_bwd_ws bytes, device, overwritten) holds Delta_i =
 * rowsum(dO_i * O_i); for bf16 with Dh 128 the pair (-LSE_i log2 e, Delta_i)
 * per row (rows padded to whole 128-row tiles), the compact K and V, and
 * float32 dK / dV partials per compact row, which are summed per key in
 * segment order (deterministic; no atomics).
 */
mw_status mw_masked_attn_bwd(const mw_vis_layout* layout, const void* vis,
                             const void* Q, const void* K, const void* V, const void* O,
                             const void* dO, const float* LSE, void* dQ, void* dK, void* dV,
                             int Hq, int Hkv, int Dh, int dtype, float scale,
                             void* ws, void* stream);

/*
 * Row-wise logical positions (§4.2: position ids reassigned so that the keys a
 * row sees form a gap-free sequence; condition (ii) of the 4D-mask equivalence
 * proposition, App. C).
 *   pos  int32 [layout->n_keymask * 128] (device, overwritten). Entry
 *        (traj_km[b] + s * nt_b) * 128 + j, for trajectory b with nt_b tiles,
 *        its segment s and key j < 128 nt_b, is the rank of key j in segment
 *        s's live view (the number of view members before j), or -1 when j is
 *        not a member (evicted by an edit <= s, after the segment, or past
 *        T_b). traj_km is the vis array at layout->off_traj_km. A row i of
 *        segment s is a member of its own view; its entry is its position.
 * Computed from the view bits of `vis` (one prefix popcount per segment).
 */
mw_status mw_logical_positions(const mw_vis_layout* layout, const void* vis, int32_t* pos, void* stream);

/*
 * Rotary-embedding table (RoFormer rotate-half pairing; the paper fixes no
 * positional encoding, only that it depend on the logical offset):
 *   table float32 [n_pos][Dh/2][2] (device, overwritten) =
 *   (cos, sin)(p * theta^(-2f/Dh)) for position p < n_pos and pair f < Dh/2,
 *   evaluated in double precision and rounded once.
 * Dh even and > 0; theta > 0 and finite (MW_ESHAPE / MW_EINVAL).
 */
mw_status mw_rope_table(int n_pos, int Dh, double theta, float* table, void* stream);

/*
 * Rotate every row by its own logical position: for row i of segment s with
 * p = pos[(traj_km[b] + s nt_b) 128 + i], pair f of every head turns by the
 * table angle of p (inverse != 0: by minus that angle, the transpose):
 *   y_f = x_f cos - x_(f+Dh/2) sin,  y_(f+Dh/2) = x_(f+Dh/2) cos + x_f sin.
 *   X, Y [total_tokens, H, Dh] (dtype); Y may equal X (in place).
 * pos from mw_logical_positions, table from mw_rope_table with
 * n_pos >= 128 * layout->max_tiles (else MW_ESHAPE).
 */
mw_status mw_rope_rows(const mw_vis_layout* layout, const void* vis, const int32_t* pos, const float* table,
                       int n_pos, const void* X, void* Y, int H, int Dh, int dtype, int inverse, void* stream);

/* Workspace bytes of mw_masked_attn_rope_fwd and of mw_masked_attn_rope_bwd. */
mw_status mw_masked_attn_rope_ws(const mw_vis_layout* layout, int Hq, int Hkv, int Dh, int dtype,
                                 size_t* fwd_bytes, size_t* bwd_bytes);

/*
 * mw_masked_attn_fwd with rotary positions reassigned per row (§4.2): the
 * score of row i (segment s) and visible key j is
 *   scale * (R(p_s(i)) q_i) . (R(p_s(j)) k_j),
 * so it depends only on the logical offset p_s(i) - p_s(j), the number of
 * keys of view_s in [j, i). Q, K are NOT rotated by the caller. The rotated
 * queries and, for every segment, the keys of its view rotated to their
 * positions in it (layout->n_keymask * 128 rows of [Hkv, Dh]) are written to
 * `ws` (mw_masked_attn_rope_ws fwd_bytes). Other arguments as
 * mw_masked_attn_fwd; pos and table as mw_rope_rows. bf16 with Dh 128 runs
 * on the tensor-core kernels (one CTA per q-tile and segment it serves:
 * tiles that a junction splits get one CTA per segment); float32, and bf16
 * with Dh 64, on the CUDA-core kernels. MW_ESHAPE when n_keymask * 128 or
 * the segment count exceeds the tensor-core kernels' int32 coordinates.
 */
mw_status mw_masked_attn_rope_fwd(const mw_vis_layout* layout, const void* vis, const int32_t* pos,
                                  const float* table, int n_pos, const void* Q, const void* K, const void* V,
                                  void* O, float* LSE, int Hq, int Hkv, int Dh, int dtype, float scale,
                                  void* ws, void* stream);

/*
 * Backward of mw_masked_attn_rope_fwd: dQ, dK, dV of the un-rotated inputs
 * (dQ = R^T dQ_rot per row; dK_j = sum over the segments whose view holds j
 * of R(p_s(j))^T times that segment's key-row gradient, accumulated in
 * float32), all in dtype, overwritten. dV_j likewise sums the per-segment
 * parts on the tensor-core path. `ws`: mw_masked_attn_rope_ws bwd_bytes
 * (recomputes the rotations; need not hold the forward's).
 */
mw_status mw_masked_attn_rope_bwd(const mw_vis_layout* layout, const void* vis, const int32_t* pos,
                                  const float* table, int n_pos, const void* Q, const void* K, const void* V,
                                  const void* O, const void* dO, const float* LSE, void* dQ, void* dK, void* dV,
                                  int Hq, int Hkv, int Dh, int dtype, float scale, void* ws, void* stream);

/*
 * Diverging rows of SDCC (§5; App. B Def. "trajectory tree": a node whose
 * live prefix differs from its prefix on the final compressed walk):
 *   out uint8 [total_tokens] (device, overwritten) = 1 where row i saw a key
 *   that a later edit evicts (some j <= i with i < omega(j) < INT32_MAX),
 *   else 0. Row i scores token i + 1, so these are the leaves where SDCC adds
 *   its KL term. One prefix-max scan of the lifetimes per trajectory.
 */
mw_status mw_diverging_rows(const mw_vis_layout* layout, const void* vis, uint8_t* out, void* stream);

/*
 * The final compressed walk of every trajectory (§5: the replay sequence left
 * after every edit, the student's input): its never-evicted positions in order.
 *   walk_index  int32 [total_tokens]: position of token j on its trajectory's
 *               walk (0-based), -1 if some edit evicts j;
 *   student_row int32 [total_tokens]: for row r, the walk index of the last
 *               surviving position <= r, -1 if none (when token r+1 survives,
 *               the walk row whose prediction is the student's for it);
 *   walk_len    int32 [n_traj]: the walk's length per trajectory.
 * All device, overwritten. One prefix count of survivors per trajectory.
 * student_row is defined for every row, including rows whose leaf y_(r+1) is
 * evicted; SDCC scores a leaf on the student side only when its token survives
 * on the walk, so a caller keeps loss row r only where walk_index[r + 1] >= 0
 * (and r + 1 lies inside the trajectory).
 */
mw_status mw_final_walk(const mw_vis_layout* layout, const void* vis, int32_t* walk_index, int32_t* student_row,
                        int32_t* walk_len, void* stream);

/* Workspace bytes of the forward-KL pair (kept from forward to backward). */
mw_status mw_forward_kl_ws(int M, int d, int Vocab, int dtype, size_t* ws_bytes);

/*
 * SDCC's consistency term (§5, Eq. "soft_loss"), forward: for pair m the
 * teacher row HT[rows_T[m]] and the student row HS[rows_S[m]],
 *   zT = hT W^T, zS = hS W^T (never stored),
 *   kl[m] = KL(softmax(zT) || softmax(zS)) = sum_v pT (log pT - log pS),
 *   loss  = lam * sum_m kl[m]  (one float32, device),
 * the forward KL with the teacher first. HT [N_T, d], HS [N_S, d], W [Vocab, d]
 * (dtype, W in torch Linear layout), rows_T / rows_S int32 [M] (device),
 * rows_S distinct (M <= N_S), rows_T may repeat. lam >= 0 and finite
 * (MW_EINVAL). M = 0 gives loss = 0.
 * bf16 with d a multiple of 64 that the LM head's CTA groups split (as for
 * mw_logprob_loss_fwd): tensor cores. For the teacher rows and then the
 * student rows, one fused pass over the vocabulary gives lse and
 * E = sum_v p_v W_v; since z = h W^T, E_pT[zT - zS] = (hT - hS) . E_T, so
 * kl = (hT - hS) . E_T - lse_T + lse_S. Otherwise (fp32; bf16 with d <= 256
 * not split that way): float32 on CUDA cores. `ws` keeps lse (and E) for the
 * backward.
 */
mw_status mw_forward_kl_fwd(const void* HT, const int32_t* rows_T, const void* HS, const int32_t* rows_S, int M,
                            const void* W, int N_T, int N_S, int d, int Vocab, int dtype, float lam,
                            float* kl, float* loss, void* ws, void* stream);

/*
 * Backward of mw_forward_kl_fwd scaled by dloss, the teacher held fixed
 * (stop-gradient): dzS = lam * dloss * (softmax(zS) - softmax(zT)),
 *   dHS[rows_S[m]] = dzS_m W (other rows of dHS = 0),  dW = sum_m dzS_m^T hS_m.
 * dHS [N_S, d] in dtype and dW [Vocab, d] float32 are overwritten
 * (accumulate = 0) or added to (accumulate = 1: rows of dHS without a pair
 * are left as they are), so the KL's gradients can join the task loss's in
 * one buffer. Needs the forward's `ws` (the tensor-core path also uses it as
 * scratch). Tensor cores:
 * dHS = lam dloss (E_S - E_T) from the forward, dW by two vocabulary-
 * stationary passes (the student's softmax, then the teacher's added in).
 */
mw_status mw_forward_kl_bwd(const void* HT, const int32_t* rows_T, const void* HS, const int32_t* rows_S, int M,
                            const void* W, int N_T, int N_S, int d, int Vocab, int dtype, float lam, float dloss,
                            int accumulate, void* ws, void* dHS, float* dW, void* stream);

/* Synchronise `stream` and report, from `ws`, the last mw_forward_kl_fwd /
 * mw_forward_kl_bwd on it: MW_ETIMEOUT if a bounded device wait of the
 * tensor-core passes gave up, MW_EDEVICE if a pair's row index lay outside
 * [0, N_T) (rows_T) or [0, N_S) (rows_S), else MW_OK. Such a row is never
 * read or written (it counts as a zero row); the call's other outputs are
 * then unspecified. */
mw_status mw_forward_kl_check_status(int M, int d, int Vocab, int dtype, void* ws, void* stream);

/*
 * Branch-replicated packing for stacked layers (App. G). From the second layer
 * on a token's state differs between the segments' branches that hold it, so
 * the exact multi-layer step runs every branch's compact sequence (its live
 * view in order, §4.1) through all layers. Packed rows: the branches back to
 * back in global segment order, branch g at rows off_g = sum of the earlier
 * seg_len values, |view_g| rows (total: the sum of seg_len); a packed record
 * of those lengths with no edits is what the layers attend over.
 *   mw_branch_pack:       Xp[off_g + c] = X[csrc_g(c)]  (c < |view_g|)
 *   mw_branch_unpack_add: dX[j] = sum over the segments g holding j, in
 *                         segment order, of dXp[off_g + cpos_g(j)]
 *                         (float32 accumulation, written in dtype)
 * X, dX [total_tokens, row_elems], Xp, dXp [sum seg_len, row_elems] (dtype,
 * device); row_elems * element size a multiple of 16 bytes (MW_ESHAPE).
 * `vis` from either builder.
 */
mw_status mw_branch_pack(const mw_vis_layout* layout, const void* vis, const void* X, void* Xp, int row_elems,
                         int dtype, void* stream);
mw_status mw_branch_unpack_add(const mw_vis_layout* layout, const void* vis, const void* dXp, void* dX,
                               int row_elems, int dtype, void* stream);

/* Bytes of device workspace the log-prob loss forward/backward pair needs. */
mw_status mw_logprob_ws(int N, int M, int d, int Vocab, int dtype, size_t* ws_bytes);

/*
 * Fused LM-head log-prob + clipped policy loss, forward. No logits tensor is
 * materialised. For loss row m (physical row t = rows[m]):
 *   z_v = H_t . W_v,  lse_m = log sum_v exp z_v,  lp_m = z_{targets[t]} - lse_m,
 *   ratio_m = exp(lp_m - lp_old_m),
 *   loss = (1/M) sum_m -min(ratio_m A_m, clip(ratio_m, 1-eps_lo, 1+eps_hi) A_m)
 * (App. B.4 "Pitfall A, RL view" ratio; PPO/GRPO clipping, App. F.1).
 *   H [N, d], W [Vocab, d] (dtype; W in torch Linear layout); targets[N],
 *   rows[M] distinct physical rows (int32, device); lp_old, adv [M] float32.
 *   An index out of range (rows[m] outside [0, N), a target outside
 *   [0, Vocab)) is not followed; mw_logprob_check_status reports it.
 *   Outputs lp, ratio, lse [M] float32, loss: one float32 (device).
 * `ws` (mw_logprob_ws bytes) keeps dL/dlp per row for the backward.
 * M = 0 is allowed: the loss is 0 (and the backward writes zero gradients).
 * dtype MW_BF16 requires d % 64 == 0; MW_F32 requires d <= 256.
 */
mw_status mw_logprob_loss_fwd(const void* H, const void* W, const int32_t* targets,
                              const int32_t* rows, int M, const float* lp_old, const float* adv,
                              float eps_lo, float eps_hi, int N, int d, int Vocab, int dtype,
                              float* lp, float* ratio, float* lse, float* loss,
                              void* ws, void* stream);

/*
 * mw_logprob_loss_fwd plus the KL-to-reference term of GRPO training (App. F.1:
 * coefficient beta, "low-variance estimator"), read as the k3 estimate per loss
 * row with d_m = lp_ref_m - lp_m:
 *   loss += beta * (1/M) sum_m (exp(d_m) - d_m - 1),
 *   dL/dlp_m gains beta * (1 - exp(d_m)) / M (kept in `ws` for the backward,
 *   which is unchanged).
 *   lp_ref [M] float32 (device): the reference policy's log-prob of each loss
 *   row's target. beta >= 0 and finite, else MW_EINVAL; beta > 0 with M > 0
 *   requires lp_ref (MW_EINVAL); beta = 0 ignores lp_ref and equals
 *   mw_logprob_loss_fwd. The paper has no closed form for the estimator; k3 is
 *   the standard low-variance one.
 */
mw_status mw_logprob_loss_fwd_kl(const void* H, const void* W, const int32_t* targets,
                                 const int32_t* rows, int M, const float* lp_old, const float* adv,
                                 float eps_lo, float eps_hi, const float* lp_ref, float beta,
                                 int N, int d, int Vocab, int dtype,
                                 float* lp, float* ratio, float* lse, float* loss,
                                 void* ws, void* stream);

/*
 * Backward of mw_logprob_loss_fwd, scaled by the upstream gradient dloss:
 *   dz_{m,v} = dloss * g_m * (1[v = target] - softmax_v(z_m)),
 *   dH_t = sum_v dz_{m,v} W_v (rows outside `rows` get 0),
 *   dW_v = sum_m dz_{m,v} H_{rows[m]}.
 * Needs the forward's lse and `ws`. dH [N, d] in dtype; dW [Vocab, d] float32.
 * Both are overwritten. The backward keeps the forward's part of `ws` intact
 * (it may run again with another dloss) and uses the rest as scratch, so two
 * backward calls on one `ws` must not overlap in time.
 */
mw_status mw_logprob_loss_bwd(const void* H, const void* W, const int32_t* targets,
                              const int32_t* rows, int M, int N, int d, int Vocab, int dtype,
                              const float* lse, void* ws, float dloss,
                              void* dH, float* dW, void* stream);

/*
 * Train-inference logits drift (Eq. "logdiff", §3): out = (1/M) sum_m
 * |lp_train[m] - lp_rollout[m]| over the loss-carrying tokens, one float32
 * (device). lp_train, lp_rollout float32 [M] (device), e.g. this library's
 * log-probs and the rollout's (the lp_old of the loss). M = 0 gives 0.
 * Fixed reduction order (deterministic).
 */
mw_status mw_logdiff(const float* lp_train, const float* lp_rollout, int M, float* out, void* stream);

/*
 * Copy the device status words of a visibility buffer to the host after
 * synchronising `stream`; returns MW_OK, MW_ETIMEOUT or MW_EDEVICE.
 */
mw_status mw_check_status(const mw_vis_layout* layout, const void* vis, void* stream);

/*
 * Dense visibility of trajectory `traj`, bit-packed (Eq. 7's 4D mask, for
 * checking against a dense-mask implementation on small trajectories): row i
 * sees key j iff j is in the live view of i's segment at or before i's own
 * place in it -- j <= i and j in view_s for an edits record, the view-order
 * prefix for an offload / retrieve record (§4.1: the row attends to its
 * segment's compact sequence up to itself).
 *   cu_seqlens[n_traj+1]  host int32, the record's offsets (as for the build)
 *   mask                  device uint32 [T][ceil(T / 32)], T = the trajectory's
 *                         length; bit k of word w of row i is key 32 w + k
 * T > MW_DENSE_MASK_MAX_T is MW_ESHAPE (the mask is T^2 / 8 bytes); T = 0
 * writes nothing. Reads only `vis`; asynchronous on `stream`.
 */
#define MW_DENSE_MASK_MAX_T 65536
mw_status mw_export_dense_mask(const mw_vis_layout* layout, const void* vis, const int32_t* cu_seqlens, int traj,
                               uint32_t* mask, void* stream);

/*
 * Status of the last mw_logprob_loss_fwd / mw_logprob_loss_bwd on `ws` (same
 * shape arguments): synchronises `stream`, then returns MW_ETIMEOUT if a
 * tensor-core kernel gave up a bounded wait, MW_EDEVICE if some rows[m] lay
 * outside [0, N) or its target outside [0, Vocab), else MW_OK. rows and
 * targets are device arrays no host check sees: the kernels read each index
 * once, never follow one out of range (that row reads as zero and its dH row
 * is not written), and raise this flag; lp, lse, the loss and the gradients
 * are then unspecified. No counterpart in the paper: failure detection of
 * this implementation.
 */
mw_status mw_logprob_check_status(int N, int M, int d, int Vocab, int dtype, const void* ws, void* stream);

/*
 * Self-test of the bounded-wait failure path (no counterpart in the paper):
 * launches one kernel that waits on an mbarrier nothing arrives on, gives up
 * after `limit_ns` (0 < limit_ns <= 1e9), records the timeout in `status`
 * (device int32[8], overwritten) and returns. Synchronises `stream` and
 * returns MW_ETIMEOUT when the timeout was recorded (the expected outcome);
 * the CUDA context stays usable.
 */
mw_status mw_selftest_wait_timeout(int64_t limit_ns, int32_t* status, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* MW_H_ */
