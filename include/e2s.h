/*
 * e2s.h -- C ABI of the GB300 (sm_103a) E2S-Pruner pruning decision.
 *
 * One pruning step of Algorithm 1 (E2S-Pruner) for a packed batch of images:
 *
 *   e2s_score    text-to-visual attention score a[l][h][n]       (Sec. 3.1, Eq. 1)
 *   e2s_fuse     support, reliability, layer mass, Dempster-Shafer
 *                fusion across layers, plausibility and priority q (Sec. 4.1-4.2,
 *                Eqs. 8-19)
 *   e2s_select   spatial-novelty bonus and global Top-K            (Sec. 4.3, Eqs. 20-23)
 *   e2s_compact  gather of the retained hidden / K / V rows so that the next
 *                layer runs on the shortened sequence (Sec. 4, opening
 *                paragraph; Sec. 5.1.2 pruning settings)
 *
 * Conventions shared by every call:
 *   - Every array argument is a DEVICE pointer unless its comment says host.
 *     The caller owns all memory, including the workspace; the library never
 *     allocates and never synchronises (except e2s_read_status).
 *   - Calls are asynchronous and ordered on the given stream (a cudaStream_t
 *     passed as void*, NULL = legacy default stream).  They keep no state
 *     between calls and may be issued from several host threads.
 *   - The return value reports host-side argument validation and launch
 *     errors only.  Errors found on the device (inconsistent layout arrays,
 *     a bounded wait that ran out) are OR-ed into a status word at the start
 *     of the workspace; e2s_read_status fetches it.
 *   - bf16 tensors are raw 16-bit bfloat16 patterns.  Results are
 *     deterministic: reductions run in a fixed order, and ties in the cell
 *     arg-max and in Top-K go to the lower index.
 *
 * Token layout of image b (Sec. 3.1): [system S_b][visual N_V,b on an
 * h_b x w_b grid, raster order][text N_T,b].  T_b = S_b + N_V,b + N_T,b.
 * Images are packed back to back; tok_off / vis_off / text_off are the
 * exclusive prefix sums of T_b / N_V,b / N_T,b (length B+1).
 */
#ifndef E2S_H_
#define E2S_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  E2S_OK = 0,
  E2S_ERR_INVALID_ARG = 1,   /* null pointer, bad enum value, bad parameter   */
  E2S_ERR_SHAPE = 2,         /* inconsistent sizes (host or device detected)   */
  E2S_ERR_ALIGNMENT = 3,     /* pointer or stride not 16-byte aligned          */
  E2S_ERR_UNSUPPORTED = 4,   /* valid but not implemented (e.g. d != 128)      */
  E2S_ERR_WORKSPACE = 5,     /* workspace missing, too small or misaligned     */
  E2S_ERR_CUDA = 6,          /* a CUDA runtime/driver call failed              */
  E2S_ERR_TIMEOUT = 7        /* a bounded device wait ran out (device status)  */
} e2s_status;

/* Batch layout.  Pointer members are device arrays of int32. */
typedef struct {
  int32_t B;                 /* images in the batch, >= 1                         */
  int32_t L;                 /* evidence layers, >= 1                             */
  int32_t H;                 /* query heads                                       */
  int32_t H_kv;              /* key/value heads; H % H_kv == 0 (GQA group H/H_kv) */
  int32_t d;                 /* head dimension; 128 is the only supported value   */
  const int32_t* tok_off;    /* [B+1] packed row offset of image b (K, V, hidden) */
  const int32_t* n_sys;      /* [B]   S_b                                         */
  const int32_t* n_vis;      /* [B]   N_V,b = grid_h[b] * grid_w[b]               */
  const int32_t* n_text;     /* [B]   N_T,b >= 1                                  */
  const int32_t* grid_h;     /* [B]   visual grid height                          */
  const int32_t* grid_w;     /* [B]   visual grid width                           */
  const int32_t* vis_off;    /* [B+1] packed offset into per-visual-token arrays  */
  const int32_t* text_off;   /* [B+1] packed offset into text-query rows          */
  int32_t max_T, max_vis, max_text;    /* HOST values: maxima over the batch      */
  int32_t sum_T, sum_vis, sum_text;    /* HOST values: tok_off[B], vis_off[B], text_off[B] */
} e2s_layout;

/* Score modes.  EQ1 is Eq. 1 as printed: the mean over text queries of the
 * pre-softmax logit Q_t K_n / sqrt(d).  CAUSAL_PROB is the attention
 * probability the model itself computes: softmax of Q_t K^T / sqrt(d) over
 * the text row's full causal key prefix (keys 0 .. S+N_V+t), visual columns
 * kept, mean over the text rows. */
enum { E2S_SCORE_EQ1 = 0, E2S_SCORE_CAUSAL_PROB = 1 };

/* Normalisation of Eq. 8 over the candidate tokens.  DEFAULT = SOFTMAX for
 * EQ1 and RENORM (r = a / sum a, which keeps r = 1/N_l as "average") for
 * CAUSAL_PROB, where a softmax of probabilities would be nearly uniform. */
enum { E2S_NORM_DEFAULT = 0, E2S_NORM_SOFTMAX = 1, E2S_NORM_RENORM = 2 };

/* Flags.  The first five are the ablations of Table 2 (A1-A5). */
enum {
  E2S_NO_RELIABILITY = 1u << 0,   /* A2: rho = 1 (Bayesian masses)                      */
  E2S_NO_LAYER_FUSION = 1u << 1,  /* A3: only the last evidence layer, no prior         */
  E2S_NO_CONFLICT = 1u << 2,      /* A4: q = Pl                                         */
  E2S_NO_NOVELTY = 1u << 3,       /* A5: lambda = 0                                     */
  E2S_VANILLA = 1u << 4,          /* A1: q = mean over layers and heads of a, lambda = 0 */
  E2S_SIMT_SCORE = 1u << 8        /* e2s_score: plain SIMT kernel instead of tcgen05    */
};

typedef struct {
  float lambda;        /* spatial novelty weight, Eq. 22; paper value 0.1         */
  int32_t G;           /* G x G spatial cells, Sec. 4.3; paper value 4; 1..8      */
  int32_t score_mode;  /* E2S_SCORE_*                                            */
  int32_t norm_mode;   /* E2S_NORM_*                                             */
  uint32_t flags;      /* E2S_* flags                                            */
} e2s_params;

/* Bytes of workspace every call below needs: the status word, one float4 of
 * normalisation statistics per (image, layer, head) written by e2s_score and
 * e2s_decide, and one arrival counter per image (e2s_decide).  The workspace
 * must be 256-byte aligned and its first 32 bytes zero before the first call
 * (e2s_clear_status zeroes them; bytes 4..11 hold the attention kernel's item
 * counter and bytes 12..19 the streaming score kernel's unit counter, which
 * every call leaves zero); the rest needs no initialisation. */
size_t e2s_workspace_size(const e2s_layout* layout, const e2s_params* params);

/* Text-to-visual score (Sec. 3.1, Eq. 1; Algorithm 1 "Compute a_{l,h,n}").
 *   q_text  bf16 [L][sum_text] rows of (H x d), row stride q_row_stride elements
 *           (>= H*d, multiple of 8); layer l starts at row l*sum_text.
 *   k       bf16 [L][sum_T] rows of (H_kv x d), row stride k_row_stride elements
 *           (>= H_kv*d, multiple of 8); layer l starts at row l*sum_T.
 *           Query head h uses key head h / (H / H_kv).
 *   a_out   fp32 [L][H][sum_vis]: a[l][h][vis_off[b] + n].
 * q_text and k must be 16-byte aligned.  The default path is a tcgen05/TMEM
 * kernel with TMA-staged K tiles; flag E2S_SIMT_SCORE selects a plain SIMT
 * kernel with the same results (used to cross-check). */
e2s_status e2s_score(const e2s_layout* layout, const e2s_params* params,
                     const void* q_text, int64_t q_row_stride,
                     const void* k, int64_t k_row_stride,
                     float* a_out, void* ws, size_t ws_bytes, void* stream);

/* Text-to-visual score reusing the pruning layer's own attention pass (Sec. 6
 * names lower-overhead evidence caching as future work; taking the attention
 * pass's row normalisers is this library's reading of it).  A flash-attention forward of the layer already
 * returns, for every query row, the natural-log log-sum-exp of its scaled
 * logits Q_t K_j / sqrt(d) over the row's causal prefix (j = 0 .. S+N_V+t).
 * Given those of the text rows, the CAUSAL_PROB score needs only the visual
 * key tiles, in one pass: a[l][h][n] = mean over t of
 * exp(Q_t K_n / sqrt(d) - lse_t), with no sweep over the whole prefix for the
 * row normalisers.
 *   lse_text  fp32 [L][H][sum_text], device, 4-byte aligned:
 *             lse_text[(l*H + h)*sum_text + text_off[b] + t] for text row t of
 *             image b, query head h, layer l; finite for every text row.  Its
 *             accuracy bounds that of a (a relative error e in exp(-lse)
 *             scales a by 1 + e), so it should be float32-exact.
 * Other arguments, the results and the Eq. 8 statistics left in the workspace
 * are those of e2s_score.  E2S_ERR_UNSUPPORTED unless score_mode is
 * CAUSAL_PROB, E2S_SIMT_SCORE is clear and max_text <= 128. */
e2s_status e2s_score_lse(const e2s_layout* layout, const e2s_params* params,
                         const void* q_text, int64_t q_row_stride,
                         const void* k, int64_t k_row_stride, const float* lse_text,
                         float* a_out, void* ws, size_t ws_bytes, void* stream);

/* The pruning layer's own causal self-attention, with the decision's score
 * as a by-product (Sec. 3.1; Sec. 6 names lower-overhead evidence caching as
 * future work, and reading the score off the layer's attention pass is this
 * library's reading of it).  Every row attends to the keys of its own image
 * at positions up to its own (causal mask per image, images packed as in the
 * layout); query head h uses key/value head h / (H / H_kv).
 *   q        bf16 [L][sum_T] rows of (H x d): the queries of EVERY row (not
 *            only the text rows), row stride q_row_stride elements.
 *   k, v     bf16 [L][sum_T] rows of (H_kv x d), strides k_/v_row_stride.
 *   o_out    bf16 [L][sum_T] rows of (H x d), stride o_row_stride: the
 *            attention output softmax(Q K^T / sqrt(d)) V of every row.
 *   lse_out  nullable fp32 [L][H][sum_T]: natural-log normaliser of every row
 *            (the value e2s_score_lse takes for the text rows).
 *   a_out    nullable fp32 [L][H][sum_vis]: the CAUSAL_PROB score of
 *            e2s_score, computed from the final normalisers of the text rows
 *            inside the same launch (no other pass reads K for it); the Eq. 8
 *            statistics go to the workspace and the decision scratch is
 *            zeroed, as e2s_score does, so e2s_fuse / e2s_fuse_select /
 *            e2s_select may follow.  Requires max_text <= 128
 *            (E2S_ERR_UNSUPPORTED otherwise).
 * Pointers 16-byte aligned (lse_out, a_out 4), strides multiples of 8 and at
 * least H*d (q, o) or H_kv*d (k, v).  P is rounded to bf16 before P V, as in
 * flash-attention forwards, so O carries bf16 rounding of the weights; lse
 * and a are computed from the fp32 logits.  The CTAs share an item counter in
 * the workspace (bytes 4..15, zero before and after the call), so calls that
 * may run concurrently need separate workspaces. */
e2s_status e2s_attention(const e2s_layout* layout, const void* q, int64_t q_row_stride,
                         const void* k, int64_t k_row_stride, const void* v, int64_t v_row_stride,
                         void* o_out, int64_t o_row_stride, float* lse_out, float* a_out,
                         void* ws, size_t ws_bytes, void* stream);


/* The whole pruning decision from the pruning layer's own attention pass, in
 * two launches: e2s_attention with a_out (the layer's O and lse, the score a
 * and its Eq. 8 statistics), then the evidence, fusion and selection of
 * e2s_decide from them -- no pass of its own over K.  Arguments are those of
 * e2s_attention and e2s_decide; a_out is required and params->score_mode must
 * be E2S_SCORE_CAUSAL_PROB (the attention pass defines that score).  Results
 * equal e2s_decide's up to the rounding order of the score's sums. */
e2s_status e2s_decide_attn(const e2s_layout* layout, const e2s_params* params, const void* q,
                           int64_t q_row_stride, const void* k, int64_t k_row_stride,
                           const void* v, int64_t v_row_stride, void* o_out, int64_t o_row_stride,
                           float* lse_out, const int32_t* cand, const float* prior, float* a_out,
                           float* mass_out, float* fused_out, float* q_out,
                           const int32_t* keep_count, const int32_t* keep_off, int32_t sum_keep,
                           int32_t* keep_idx, float* q_tilde_out, void* ws, size_t ws_bytes,
                           void* stream);

/* The whole pruning decision of one step in two launches: e2s_score, then
 * evidence, fusion and selection (Sec. 3.1 and 4.1-4.3, Eqs. 1 and 8-23).
 * Arguments have the meaning they have in e2s_score, e2s_fuse and e2s_select;
 * a_out is required (it carries a[l][h][n] from the first launch to the
 * second).  The score kernel also leaves the Eq. 8 normalisation statistics
 * of every (image, layer, head) in the workspace, so the second kernel treats
 * every visual token independently (no cross-CTA reduction) and the last CTA to
 * finish an image runs that image's Top-K.  Results are identical to
 * e2s_score, e2s_fuse and e2s_select called in sequence, up to the rounding
 * order of the normalisation sums.  keep_count and keep_off are required;
 * keep_idx may be NULL only when sum_keep == 0.  Concurrent e2s_decide calls
 * must use separate workspaces.  E2S_ERR_UNSUPPORTED when H > 128 or when
 * L * H * 84 + 5 * max_vis bytes exceed 160 KiB (L * H > 1900 or so). */
e2s_status e2s_decide(const e2s_layout* layout, const e2s_params* params,
                      const void* q_text, int64_t q_row_stride,
                      const void* k, int64_t k_row_stride,
                      const int32_t* cand, const float* prior, float* a_out,
                      float* mass_out, float* fused_out, float* q_out,
                      const int32_t* keep_count, const int32_t* keep_off, int32_t sum_keep,
                      int32_t* keep_idx, float* q_tilde_out,
                      void* ws, size_t ws_bytes, void* stream);

/* e2s_decide with its score taken as e2s_score_lse takes it (same lse_text
 * argument and restrictions). */
e2s_status e2s_decide_lse(const e2s_layout* layout, const e2s_params* params,
                          const void* q_text, int64_t q_row_stride,
                          const void* k, int64_t k_row_stride, const float* lse_text,
                          const int32_t* cand, const float* prior, float* a_out,
                          float* mass_out, float* fused_out, float* q_out,
                          const int32_t* keep_count, const int32_t* keep_off, int32_t sum_keep,
                          int32_t* keep_idx, float* q_tilde_out,
                          void* ws, size_t ws_bytes, void* stream);

/* One complete pruning step: e2s_decide followed by e2s_compact, three
 * launches (Algorithm 1, one pruning layer; Sec. 3.1 and 4.1-4.3).  Arguments
 * are those of the two calls.  The score kernel is launched with programmatic
 * dependence on the kernel before it on the stream: its blocks may be
 * scheduled while that kernel finishes, but they wait for its completion
 * before touching memory, and only then let the decision and the compaction
 * be scheduled.  So all earlier work on the stream is complete before the
 * compaction copies the system and text rows (which do not depend on the
 * selection) while the decision is still running; it waits only before the
 * kept visual rows.  The src tensors, keep_count and keep_off must therefore
 * be written by earlier work on the same stream (or be complete before the
 * call), and nothing else may write them while the call runs.  Give it
 * device-memory sources (it prefetches every candidate row into L2 on small
 * batches).  Results are identical to e2s_decide then e2s_compact. */
e2s_status e2s_prune(const e2s_layout* layout, const e2s_params* params,
                     const void* q_text, int64_t q_row_stride,
                     const void* k, int64_t k_row_stride,
                     const int32_t* cand, const float* prior, float* a_out,
                     float* mass_out, float* fused_out, float* q_out,
                     const int32_t* keep_count, const int32_t* keep_off, int32_t sum_keep,
                     int32_t* keep_idx, float* q_tilde_out,
                     int32_t n_tensors, const void* const* src, void* const* dst,
                     const int64_t* row_bytes, int32_t* pos_ids_out,
                     void* ws, size_t ws_bytes, void* stream);

/* e2s_prune with its score taken as e2s_score_lse takes it (lse_text
 * required, same restrictions). */
e2s_status e2s_prune_lse(const e2s_layout* layout, const e2s_params* params,
                         const void* q_text, int64_t q_row_stride,
                         const void* k, int64_t k_row_stride, const float* lse_text,
                         const int32_t* cand, const float* prior, float* a_out,
                         float* mass_out, float* fused_out, float* q_out,
                         const int32_t* keep_count, const int32_t* keep_off, int32_t sum_keep,
                         int32_t* keep_idx, float* q_tilde_out,
                         int32_t n_tensors, const void* const* src, void* const* dst,
                         const int64_t* row_bytes, int32_t* pos_ids_out,
                         void* ws, size_t ws_bytes, void* stream);

/* Evidence and fusion (Sec. 4.1-4.2, Eqs. 8-19; Algorithm 1 inner loops).
 *   a          fp32 [L][H][sum_vis] from e2s_score.
 *   cand       nullable int32 [sum_vis]: original raster index of visual slot n
 *              (a later progressive step); NULL = identity.  Only the spatial
 *              cells of the Top-K read it; e2s_fuse accepts it for symmetry.
 *   prior      nullable fp32 [sum_vis][4] (m~(I), m~(U), m~(Theta), -): fused
 *              mass carried from an earlier pruning step.  NULL: the first
 *              layer initialises the fusion (Eq. 12) and K^(1) = 0.
 *   mass_out   nullable fp32 [L][sum_vis][4]: (m(I), m(U), m(Theta), p_bar) (Eq. 11).
 *   fused_out  fp32 [sum_vis][4]: (m~(I), m~(U), m~(Theta), K) after the last layer;
 *              K is the conflict of the latest combination (Eq. 13).
 *   q_out      fp32 [sum_vis]: retention priority q (Eq. 19).
 * Total conflict (1 - K <= 0) gives the vacuous mass (0, 0, 1) and K = 1. */
e2s_status e2s_fuse(const e2s_layout* layout, const e2s_params* params,
                    const float* a, const int32_t* cand, const float* prior,
                    float* mass_out, float* fused_out, float* q_out,
                    void* ws, size_t ws_bytes, void* stream);

/* e2s_fuse followed by e2s_select in a single launch (one thread-block cluster
 * per image; Sec. 4.1-4.3, Eqs. 8-23).  Arguments and outputs are those of the
 * two calls; results are identical to calling them in sequence. */
e2s_status e2s_fuse_select(const e2s_layout* layout, const e2s_params* params,
                           const float* a, const int32_t* cand, const float* prior,
                           float* mass_out, float* fused_out, float* q_out,
                           const int32_t* keep_count, const int32_t* keep_off, int32_t sum_keep,
                           int32_t* keep_idx, float* q_tilde_out,
                           void* ws, size_t ws_bytes, void* stream);

/* e2s_fuse without a workspace (the paper has no counterpart; this is a
 * deployment convenience).  Some callers cannot allocate device memory: code
 * running inside a host framework whose memory pool owns the whole device
 * heap, plug-ins reached through a foreign-function interface that has no
 * allocator, or real-time loops where cudaMalloc is not allowed.  This entry
 * point takes the same inputs and outputs as e2s_fuse, and its results equal
 * e2s_fuse's up to the rounding order of the normalisation sums.  It uses a
 * two-kernel formulation (a statistics kernel, then one thread per token)
 * whose scratch -- the per-(image, layer, head) normalisation statistics --
 * lives in a static device array inside the library, so it allocates
 * nothing and needs no workspace.
 *   - Capacity: B * L * H <= 8192; larger batches return E2S_ERR_WORKSPACE
 *     before anything is launched.  The array (about 64 KiB) is held by every
 *     GPU that loads the library until the process exits.
 *   - The first call on a device looks up the array's device address (once
 *     per device, with that device current); make that first call before any
 *     stream capture.
 *   - Every call shares the one array: calls whose kernels overlap on the GPU
 *     (different streams, or different host threads on one device) race and
 *     must be serialised by the caller.  Each call rewrites every statistic it
 *     reads, so the contents left by an earlier call do no harm.
 *   - Device-side layout errors are not reported (there is no status word to
 *     read back); use e2s_fuse with a workspace and e2s_read_status to
 *     diagnose them.  The tokens of an image whose device layout arrays
 *     disagree get defined placeholder outputs: every layer mass and the
 *     fused mass (0, 0, 1, 0) and q = 0. */
e2s_status e2s_fuse_noalloc(const e2s_layout* layout, const e2s_params* params,
                            const float* a, const int32_t* cand, const float* prior,
                            float* mass_out, float* fused_out, float* q_out, void* stream);

/* Spatial novelty and Top-K (Sec. 4.3, Eqs. 20-23).
 *   q            fp32 [sum_vis] priorities (e2s_fuse q_out).
 *   cand         nullable int32 [sum_vis] original raster index of each slot
 *                (ascending per image); NULL = identity.  Cells follow the
 *                original grid: cell(i, j) = (i*G/h, j*G/w), integer division.
 *   keep_count   int32 [B] K_b >= 0.
 *   keep_off     int32 [B+1] exclusive prefix sum of keep_count.
 *   sum_keep     HOST int: keep_off[B].
 *   keep_idx     int32 [sum_keep] out: image-local visual slot indices, ascending
 *                per image.  If K_b > N_V,b all slots are kept and the spare
 *                entries are -1.
 *   q_tilde_out  nullable fp32 [sum_vis]: q~ of Eq. 22. */
e2s_status e2s_select(const e2s_layout* layout, const e2s_params* params,
                      const float* q, const int32_t* cand,
                      const int32_t* keep_count, const int32_t* keep_off, int32_t sum_keep,
                      int32_t* keep_idx, float* q_tilde_out,
                      void* ws, size_t ws_bytes, void* stream);

/* Row compaction of the shortened sequence.  Output rows of image b, in
 * order: system rows [0, S_b), visual rows S_b + keep_idx (ascending), text
 * rows [S_b + N_V,b, T_b).  Output image b starts at row
 * tok_off[b] - vis_off[b] + keep_off[b]; total rows sum_T - sum_vis + sum_keep.
 *   src[i], dst[i]  n_tensors (1..32) HOST arrays of DEVICE pointers to
 *                   row-major [sum_T][row] and [sum_T - sum_vis + sum_keep][row]
 *                   tensors (e.g. hidden states and each layer's K and V).
 *                   A source may also be page-locked host memory the device
 *                   can address (cudaHostAlloc, or cudaHostRegister with
 *                   mapping, under unified addressing): the kernel then reads
 *                   only the rows it keeps across the host link.  (e2s_prune
 *                   prefetches every candidate row into L2: give it device
 *                   sources.)
 *   row_bytes[i]    HOST array; each a positive multiple of 16; pointers
 *                   16-byte aligned.
 *   pos_ids_out     nullable int32 [total rows]: image-local original position
 *                   of every output row.
 * Requires 0 <= K_b <= N_V,b (device-checked; a violating image is skipped and
 * E2S_ERR_SHAPE is raised in the status word).  Rows are copied bit-exactly. */
e2s_status e2s_compact(const e2s_layout* layout, const int32_t* keep_idx,
                       const int32_t* keep_off, int32_t sum_keep, int32_t n_tensors,
                       const void* const* src, void* const* dst, const int64_t* row_bytes,
                       int32_t* pos_ids_out, void* ws, size_t ws_bytes, void* stream);

/* Synchronises `stream`, reads and returns the device status word (E2S_OK if
 * no device-side error was recorded; otherwise the lowest-numbered recorded
 * error).  Does not clear it. */
e2s_status e2s_read_status(const void* ws, void* stream);

/* Zeroes the first 32 bytes of the workspace: the device status word and the
 * attention and streaming score kernels' work counters (stream-ordered,
 * asynchronous). */
e2s_status e2s_clear_status(void* ws, void* stream);

/* Human-readable name of a status value (static string). */
const char* e2s_status_string(e2s_status s);

/* Self-test of the bounded device waits (no counterpart in the paper).
 * Every mbarrier wait in this library's kernels gives up after a wall-clock
 * limit, records E2S_ERR_TIMEOUT in the status word and lets the kernel
 * return, so a lost arrival is reported instead of hanging the GPU.  This
 * call launches one thread that initialises a barrier expecting two
 * arrivals, arrives once (twice when `complete` is non-zero) and waits on it
 * with that same bounded wait, nothing else in flight.
 *   complete  0: the phase never completes; after limit_ns the wait gives up
 *             and E2S_ERR_TIMEOUT is OR-ed into the status word.
 *             1: the phase completes and nothing is recorded.
 *   limit_ns  HOST value, 1e6 .. 2e9 (1 ms .. 2 s), else E2S_ERR_INVALID_ARG.
 *   ws        256-byte aligned workspace; only its status word is used.
 * Read the outcome with e2s_read_status. */
e2s_status e2s_selftest_bounded_wait(int32_t complete, int64_t limit_ns, void* ws, void* stream);

/* Library ABI version (major * 100 + minor). */
int32_t e2s_version(void);

#ifdef __cplusplus
}
#endif
#endif /* E2S_H_ */
