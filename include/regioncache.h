/*
 * regioncache.h -- C ABI of the GB300 (sm_103a) region-sparse DiT step.
 *
 * The library implements the hot path of RegionCache (semantic-aware region
 * reuse for multi-turn image editing): a cross-attention localisation pass
 * turns the prompt-delta text tokens into a token-level dirty mask
 * (Section 3.2, R_edit); only dirty image tokens are recomputed through each
 * PixArt-alpha-shaped block, their queries attending over every token's
 * keys/values, where clean tokens' K/V and hidden states come from a
 * per-(layer, timestep) cache (Section 3.3, Region-Level Sparse Attention);
 * fresh K/V rows are written straight to their cache rows by the projection
 * GEMM (Section 3.4, Kernel Fusing); a step follows a per-step reuse
 * schedule given as input (Section 3.3, Eq. 2).
 *
 * Conventions for every entry point:
 *   - Return value: rc_status; RC_OK (0) on success.  No C++ exception ever
 *     crosses this boundary.  rc_last_error() gives a thread-local message
 *     for the last failing call on the calling thread.
 *   - Host arguments are validated before anything is launched; a failing
 *     validation launches nothing and changes no memory.
 *   - Pointers named *_host are host memory.  Every other tensor pointer is a
 *     device pointer owned by the caller, who keeps it alive and unmodified
 *     until the work queued on `stream` has finished.  Weights are borrowed
 *     for the lifetime of the rc_ctx.
 *   - Work is queued asynchronously on `stream` (a cudaStream_t; 0 is the
 *     legacy default stream).  Device-side argument errors (an index out of
 *     range, a count above its bound) are recorded in a library-owned error
 *     word and reported by rc_sync().
 *   - Dtypes: "bf16" = bfloat16 (2 bytes), "f32" = IEEE float.  Matrices are
 *     row-major.  Linear weights are [out][in]: y = x W^T + b.
 */
#ifndef REGIONCACHE_H
#define REGIONCACHE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int rc_status;
#define RC_OK 0
#define RC_ERR_INVALID_ARG 1   /* null pointer, value out of range           */
#define RC_ERR_SHAPE 2         /* sizes inconsistent with the rc_dims         */
#define RC_ERR_OOM 3           /* device allocation failed                    */
#define RC_ERR_CUDA 4          /* a CUDA runtime call failed                  */
#define RC_ERR_TIMEOUT 5       /* a bounded device wait gave up               */
#define RC_ERR_DEVICE_ASSERT 6 /* a kernel found a bad index / count          */
#define RC_ERR_STATE 7         /* call order violated (e.g. no weights set)   */
#define RC_ERR_IO 8            /* a file could not be opened, read or written */

/* Per-step modes of a reuse schedule (Section 3.3, Eq. 2). */
#define RC_MODE_DENSE 0  /* every token recomputed; cache rows overwritten    */
#define RC_MODE_SPARSE 1 /* only the dirty tokens recomputed                  */
#define RC_MODE_REUSE 2  /* no block runs; the last hidden state is cached    */

typedef void* rc_stream; /* cudaStream_t */

/* Model and problem sizes.  PixArt-alpha: hidden 1152, heads 16 (head_dim
 * 72), mlp 4608, layers 28, patch 2, in_ch 4, out_ch 8, text_len 120,
 * freq_dim 256.  N = grid_h * grid_w image tokens.  max_batch = most items
 * of one rc_step_batched call (1 .. RC_MAX_BATCH; 0 means 1): the context's
 * row scratch is sized for max_batch * N rows. */
#define RC_MAX_BATCH 16
typedef struct rc_dims {
  int hidden, heads, mlp, layers;
  int grid_h, grid_w, patch, in_ch, out_ch;
  int text_len, timesteps, freq_dim;
  int max_batch;
} rc_dims;

/* One block's weights (device pointers, borrowed).  W_* bf16 [out][in];
 * b_* f32 [out]; table f32 [6][hidden] = the adaLN-single scale-shift table
 * whose rows are (shift_msa, scale_msa, gate_msa, shift_mlp, scale_mlp,
 * gate_mlp).  W_qkv's outputs are q | k | v; W_xkv's are k | v. */
typedef struct rc_layer_weights {
  const void* W_qkv; const float* b_qkv;  /* [3h][h], [3h] */
  const void* W_o;   const float* b_o;    /* [h][h],  [h]  */
  const void* W_xq;  const float* b_xq;   /* [h][h],  [h]  */
  const void* W_xkv; const float* b_xkv;  /* [2h][h], [2h] */
  const void* W_xo;  const float* b_xo;   /* [h][h],  [h]  */
  const void* W_1;   const float* b_1;    /* [F][h],  [F]  */
  const void* W_2;   const float* b_2;    /* [h][F],  [h]  */
  const float* table;                     /* [6][h]        */
} rc_layer_weights;

/* Model-level weights (device pointers, borrowed).  W_e: patch embedding as a
 * linear map of the patch vector ordered (channel, py, px), bf16
 * [h][in_ch*p*p]; pos f32 [N][h] fixed positional table; timestep MLP
 * W_t1 [h][freq_dim], W_t2 [h][h]; adaLN-single W_tb [6h][h]; final layer
 * table_f f32 [2][h] (shift, scale), W_f bf16 [p*p*out_ch][h] with outputs
 * ordered (py, px, channel). */
typedef struct rc_global_weights {
  const void* W_e;  const float* b_e;  const float* pos;
  const void* W_t1; const float* b_t1;
  const void* W_t2; const float* b_t2;
  const void* W_tb; const float* b_tb;
  const float* table_f;
  const void* W_f;  const float* b_f;
} rc_global_weights;

typedef struct rc_ctx rc_ctx;     /* model + device scratch, one per stream user */
typedef struct rc_cache rc_cache; /* library-owned per-(session, t, layer) cache */

/* ---------------------------------------------------------------- context */

/* Creates a context on the current CUDA device and allocates its scratch
 * (sized for N tokens).  Errors: RC_ERR_INVALID_ARG (null, a dimension <= 0),
 * RC_ERR_SHAPE (hidden % heads != 0, head_dim not 72 or 64, hidden not a
 * multiple of 128 or above 1536, mlp not a multiple of 128, N > 16384,
 * in_ch * patch^2 > 16, out_ch < in_ch), RC_ERR_OOM.  Validation happens
 * before any CUDA call. */
rc_status rc_create(const rc_dims* dims, rc_ctx** out);
void rc_destroy(rc_ctx* ctx);

/* Registers (borrows) the weights of block `layer` / of the model.  The text
 * keys / values of every session (and the cross-query keys folded from them,
 * see rc_set_text) depend on a layer's W_xkv, b_xkv, W_xq and b_xq:
 * rc_set_layer_weights therefore marks the text of every session of every
 * cache of this context stale, and steps of a session return RC_ERR_STATE
 * until rc_set_text (or rc_cache_import) runs for it again. */
rc_status rc_set_layer_weights(rc_ctx* ctx, int layer, const rc_layer_weights* w);
/* The timestep embedding and t_block modulation of every scheduled timestep
 * depend only on W_t1 .. b_tb and the schedule: they are computed once, at
 * the first step or graph capture after rc_set_global_weights or
 * rc_set_schedule, and reused by every later step.  Weights changed in place
 * therefore need rc_set_global_weights again.  (A step captured by the
 * caller into a graph before they exist computes its own.) */
rc_status rc_set_global_weights(rc_ctx* ctx, const rc_global_weights* w);

/* Sampling schedule, copied: timestep values t_values_host[timesteps] fed to
 * the timestep embedding, and cumulative alphas alpha_bar_host[timesteps+1]
 * (entry timesteps is the value after the last step, normally 1) for the
 * DDIM (eta = 0) update after step t: alpha_bar[t] -> alpha_bar[t+1]. */
rc_status rc_set_schedule(rc_ctx* ctx, const float* t_values_host, const float* alpha_bar_host);

/* Reproducible sums.  By default the three gated-residual projections of a
 * block (x += g (y W^T + b) after attention, cross-attention and the MLP,
 * Section 3.3's region block) may split their reduction over k between
 * CTAs that add their partial products into x with atomic reductions, so a
 * step's result can differ in the last bits from run to run (always within
 * the documented tolerances).  With on != 0 every such GEMM runs on whole
 * output tiles (one reduction per element, k summed in a fixed order), and
 * rc_step, rc_step_batched, rc_step_dense, rc_block_forward_region and the
 * graphs captured from them give bit-identical results for bit-identical
 * inputs on the same GPU and build.  It costs about a tenth of the step
 * rate at 831 dirty tokens of 4096 (fewer CTAs share the residual GEMMs).
 * The score sums of rc_step_capture and rc_localize_scores (over heads, with
 * atomic adds) stay order-dependent either way.  Takes effect at the next
 * launch; graphs keep the schedule they were captured with.  Never fails
 * except on a null context. */
rc_status rc_set_deterministic(rc_ctx* ctx, int on);

/* ------------------------------------------------------------------ cache */

/* Cache pool of Section 3.2 (Hidden-State-Oriented Caching): for every
 * session s, timestep t and layer l, the block output H^{l+1}, keys K^l and
 * values V^l of all N tokens, bf16 [N][hidden] each, plus the per-session
 * text keys/values of every layer.  Library-owned device memory:
 * sessions * timesteps * layers * 3 * N * hidden * 2 bytes (15.85 GB for one
 * PixArt-alpha session at 4096 tokens and 20 steps). */
rc_status rc_cache_create(rc_ctx* ctx, int sessions, rc_cache** out);

/* The same pool in pinned, device-mapped host memory (Section 3.4, Pipelined
 * Execution): for pools larger than HBM.  The text keys/values and two HBM
 * windows of 3 * N * hidden bf16 stay on the device.  rc_step and
 * rc_step_capture on such a cache load each layer's cached K, V (plus H for the
 * last layer) into a window on a library-owned copy stream while the previous
 * layer computes, then write the dirty rows' H, K, V back to host memory; the
 * results equal those of a device-tier cache.  rc_step_batched takes one item
 * and rc_block_forward_region is refused (RC_ERR_INVALID_ARG).  Steps on one
 * host-tier cache must be issued from one host thread.  rc_cache_fill /
 * rc_cache_read work as for a device-tier cache.  Errors: RC_ERR_OOM when the
 * pinned allocation or a window fails. */
rc_status rc_cache_create_host(rc_ctx* ctx, int sessions, rc_cache** out);
void rc_cache_destroy(rc_cache* cache);

/* Copies caller bf16 [N][hidden] device buffers into / out of the (session,
 * layer, t) slot.  Any of H, K, V may be null to skip it. */
rc_status rc_cache_fill(rc_cache* cache, int session, int layer, int t,
                        const void* H, const void* K, const void* V, rc_stream stream);
rc_status rc_cache_read(rc_cache* cache, int session, int layer, int t,
                        void* H, void* K, void* V, rc_stream stream);

/* One session's whole cache to / from a file, so that an editing session
 * outlives the process (the paper keeps the pool in host memory between
 * turns, Section 3.4): every (t, layer) H, K, V slot and the text
 * keys/values, after a header with N, hidden, layers, timesteps and
 * text_len.  Synchronous (the device is synchronised first); the file is
 * raw little-endian bf16, about timesteps * layers * 3 * N * hidden * 2
 * bytes.  Import requires a header equal to the cache's dimensions
 * (RC_ERR_SHAPE otherwise) and marks the session's text as set when the
 * exported session had it; the folded text keys (see rc_set_text) are not
 * in the file but recomputed on import, so a session with text needs every
 * layer's weights set first (RC_ERR_STATE otherwise).  Errors:
 * RC_ERR_INVALID_ARG, RC_ERR_IO (open, short read / write, bad magic),
 * RC_ERR_SHAPE, RC_ERR_STATE, RC_ERR_CUDA.  An import that fails after the
 * header check has overwritten part of the session: its text is then marked
 * unset (steps return RC_ERR_STATE) until rc_set_text or a successful import. */
rc_status rc_cache_export(rc_cache* cache, int session, const char* path);
rc_status rc_cache_import(rc_cache* cache, int session, const char* path);

/* Text conditioning of one session for an editing turn: ctx_bf16 is the
 * text context, bf16 [text_len][hidden].  Computes every layer's
 * cross-attention keys/values (ctx W_xkv^T + b_xkv) into the session's
 * cache, and from them the keys with the cross-query projection folded in
 * (G_h = K_h W_xq,h, kb_h = K_h b_xq,h per head, device memory owned by the
 * cache) that sparse steps use instead of a separate query projection.
 * Must precede rc_step / rc_block_forward_region for the session. */
rc_status rc_set_text(rc_ctx* ctx, rc_cache* cache, int session, const void* ctx_bf16,
                      rc_stream stream);

/* ----------------------------------------------------------- localisation */

/* Bytes of device workspace rc_localize_mask needs for N tokens and
 * n_delta delta tokens. */
size_t rc_localize_workspace_size(int N, int n_delta);

/* Edit region R_edit of Section 3.2 as a dirty mask and a compact list.
 *   xattn        f32 [S][N][M] cross-attention scores (S slices, e.g. heads
 *                x layers, averaged: summed in ascending s, divided by S).
 *   delta_ids_host  int32 [n_delta], the new/modified text tokens, each in
 *                [0, M); 1 <= n_delta <= 64.
 *   threshold    per delta token j the scores are min-max normalised over the
 *                N tokens and token i is in j's region iff the normalised
 *                value is >= threshold; a constant column gives no token,
 *                and so does a column whose averaged scores hold a
 *                non-finite value (NaN, +-Inf), where the normalisation is
 *                undefined.
 *   dilation     the union over j is dilated by a (2r+1)^2 square on the
 *                grid_h x grid_w token grid (r = dilation, 0..8), neighbours
 *                outside the grid ignored.
 *   mask         out, u8 [N] 0/1.
 *   dirty_idx    out, int32 [N] capacity; the first D entries are the dirty
 *                tokens in ascending order.
 *   dirty_count  out, int32 [1] device: D.
 *   workspace    device scratch of rc_localize_workspace_size() bytes.
 * The comparison is taken in f32 with round-to-nearest subtraction and
 * division, so the result is bit-identical to a float32 evaluation of the
 * same definition.  Errors: RC_ERR_INVALID_ARG, RC_ERR_SHAPE
 * (N != grid_h * grid_w, N > 16384, M < 1). */
rc_status rc_localize_mask(const float* xattn, int S, int N, int M, int grid_h, int grid_w,
                           const int32_t* delta_ids_host, int n_delta, float threshold,
                           int dilation, uint8_t* mask, int32_t* dirty_idx,
                           int32_t* dirty_count, void* workspace, size_t workspace_bytes,
                           rc_stream stream);

/* Allocation-free variant of rc_localize_mask.  The paper has no counterpart
 * to this entry point; it exists for callers that cannot allocate device
 * memory where they need a mask: code running inside an inference server's
 * plugin hook that must not call the CUDA allocator, programs whose device
 * memory is wholly owned by another framework's pool, and latency-critical
 * loops that cannot afford cudaMalloc's implicit device-wide synchronisation.
 *
 * It computes exactly what rc_localize_mask computes (same arguments minus
 * the workspace, same bit-exact result) but takes its scratch from a fixed
 * array compiled into the library: RC_NOALLOC_SCRATCH_BYTES (about 1 MiB) of
 * device memory that every GPU which loads the library holds until the
 * process exits.  It calls no cudaMalloc, cudaFree or other allocating
 * routine.
 *   Limits: N <= RC_NOALLOC_MAX_TOKENS and n_delta <= RC_NOALLOC_MAX_DELTA;
 *   larger sizes return RC_ERR_SHAPE with a message naming the limit.
 *   Set-up: the first call on each device (with that device current) looks
 *   up the array's device address once and keeps it for the rest of the
 *   process; make that first call before any stream capture.  The kept
 *   address does not survive cudaDeviceReset (or any destruction of the
 *   device's primary context): do not call this entry point after one.
 *   Sharing: every call on a device uses the same scratch, which keeps the
 *   previous call's contents; no part of it needs to start at zero (each
 *   pass overwrites what the next pass reads).  Calls whose work overlaps on
 *   the GPU (for example issued on two unordered streams) race on the
 *   scratch and can return wrong masks: serialise them on one stream or
 *   order them with events. */
#define RC_NOALLOC_MAX_TOKENS 16384
#define RC_NOALLOC_MAX_DELTA 16
#define RC_NOALLOC_SCRATCH_BYTES 1073408
rc_status rc_localize_mask_noalloc(const float* xattn, int S, int N, int M, int grid_h,
                                   int grid_w, const int32_t* delta_ids_host, int n_delta,
                                   float threshold, int dilation, uint8_t* mask,
                                   int32_t* dirty_idx, int32_t* dirty_count, rc_stream stream);

/* ------------------------------------------------------------ block / step */

/* Region-level sparse forward of block `layer` at timestep slot `t` of
 * `session` (Section 3.3, Region-Level Sparse Attention; Section 3.4, Kernel
 * Fusing).
 *   hidden       f32 [N][hidden], in/out: rows dirty_idx[r] are the dirty
 *                tokens' block inputs and are overwritten with their block
 *                outputs; other rows are neither read nor written.
 *   dirty_idx    int32 device, distinct token indices in [0, N) (any order).
 *   D            number of dirty tokens, 0..N; with dirty_count non-null it
 *                is only an upper bound (-1 = N) and *dirty_count is used.
 *   mod6         f32 [6][hidden] device: this block's adaLN-single vector
 *                (table + timestep projection).
 * Effect on the cache slot (session, layer, t): K and V rows of the dirty
 * tokens are replaced by their fresh projections before the attention (the
 * dirty queries attend over all N keys: cached for clean tokens, fresh for
 * dirty ones); H rows of the dirty tokens are replaced by their block
 * outputs (bf16), so H holds the merged H^{l+1}.  Clean rows are untouched.
 * D = 0 is legal and changes nothing.  Errors: RC_ERR_INVALID_ARG,
 * RC_ERR_STATE (weights or text not set). */
rc_status rc_block_forward_region(rc_ctx* ctx, rc_cache* cache, int session, int layer, int t,
                                  float* hidden, const int32_t* dirty_idx, int D,
                                  const int32_t* dirty_count, const float* mod6,
                                  rc_stream stream);

/* One denoising step t of `session` following the reuse schedule
 * schedule_host[timesteps] (modes RC_MODE_*; Section 3.3, Eq. 2):
 *   DENSE   every token is embedded and pushed through all blocks; every
 *           cache row of (session, *, t) is overwritten.
 *   SPARSE  only the dirty tokens (dirty_idx / D / dirty_count as in
 *           rc_block_forward_region) are embedded and recomputed through all
 *           blocks; clean rows come from the cache.
 *   REUSE   no block runs; the final layer reads the cached H of the last
 *           block.
 * Then the final layer (LayerNorm, modulation by the timestep embedding,
 * linear to p*p*out_ch) gives eps (the first in_ch output channels) for all
 * tokens and the latent is updated in place by DDIM (eta = 0).
 *   latent  f32 [in_ch][grid_h*patch][grid_w*patch], in/out.
 * Errors: RC_ERR_INVALID_ARG, RC_ERR_STATE (weights, schedule or text not
 * set). */
rc_status rc_step(rc_ctx* ctx, rc_cache* cache, int session, float* latent, int t,
                  const uint8_t* schedule_host, const int32_t* dirty_idx, int D,
                  const int32_t* dirty_count, rc_stream stream);

/* One item of a batched step: one session's denoising step.
 *   session      cache session (an item per (session, t) at most per call)
 *   latent       device f32 [in_ch][grid_h*patch][grid_w*patch], in/out
 *   t            timestep index in [0, timesteps)
 *   mode         RC_MODE_DENSE / SPARSE / REUSE for this step
 *   dirty_idx, D, dirty_count   SPARSE only, as in rc_step */
typedef struct rc_batch_item {
  int session;
  float* latent;
  int t;
  int mode;
  const int32_t* dirty_idx;
  int D;
  const int32_t* dirty_count;
} rc_batch_item;

/* Batched serving (no counterpart in the paper, which serves one request at
 * a time): one denoising step for each of n_items sessions, each exactly as
 * rc_step would compute it (Section 3.3 region-level sparse attention per
 * item: an item's dirty queries attend over its own session's cached and
 * fresh keys / values at its own timestep, with its own text context).  The
 * dirty rows of all items are processed together, so every weight matrix is
 * read once per call.  items: host array; 1 <= n_items <= the context's
 * max_batch.  Errors: RC_ERR_INVALID_ARG (bad item, two items on the same
 * (session, t), n_items out of range), RC_ERR_STATE (weights, schedule or a
 * session's text not set). */
rc_status rc_step_batched(rc_ctx* ctx, rc_cache* cache, const rc_batch_item* items, int n_items,
                          rc_stream stream);

/* A DENSE step (as rc_step with mode DENSE) that also produces the
 * localisation scores of Section 3.2 for the next sparse steps: for each of
 * the n_delta (1..8) newly introduced or modified text tokens j in
 * delta_ids_host (host array, values in [0, text_len)), the cross-attention
 * probabilities of j, aggregated (averaged) over the heads and layers of
 * the step:  scores[i][j] = mean_{l,h} softmax_j'(q'_{l,h,i} k_{l,h,j'} /
 * sqrt(head_dim))[j], for every image token i.
 *   scores  device f32 [N][text_len] (caller-owned, 16-B aligned): zeroed,
 *           then the delta columns written; it is the [S = 1][N][M] score map
 *           rc_localize_mask takes.
 * Errors: as rc_step; RC_ERR_INVALID_ARG for bad ids or n_delta. */
rc_status rc_step_capture(rc_ctx* ctx, rc_cache* cache, int session, float* latent, int t,
                          const int32_t* delta_ids_host, int n_delta, float* scores,
                          rc_stream stream);

/* The localisation scores of Section 3.2 for a new editing turn, computed
 * from the cached states of the previous turn instead of a dense step, so
 * that a turn scheduled by Eq. 2 (REUSE steps, then SPARSE steps, no dense
 * step at all) can localise its edit before anything is recomputed.  Call
 * it after rc_set_text with the new prompt.  For each of the n_delta (1..8)
 * new or modified text tokens j in delta_ids_host (host array, values in
 * [0, text_len)):
 *   scores[i][j] = mean over blocks l and heads h of
 *                  softmax_j'(q'_{l,h,i} k_{l,h,j'} / sqrt(head_dim))[j],
 * where the text keys k are the session's current ones and the image
 * queries q' = H^l W_xq^T + b_xq use the hidden state entering block l as
 * the cache holds it at timestep slot t: for l >= 1 the cached output of
 * block l - 1 (bf16), for l = 0 the patch embedding of `latent` (f32
 * [in_ch][grid_h*patch][grid_w*patch], the latent of step t).  The cache is
 * only read.
 *   scores  device f32 [N][text_len] (caller-owned, 16-B aligned): zeroed,
 *           then the delta columns written; it is the [S = 1][N][M] score
 *           map rc_localize_mask takes.
 * Errors: RC_ERR_INVALID_ARG (bad session, t, ids or n_delta, a host-tier
 * cache), RC_ERR_STATE (weights or the session's text not set). */
rc_status rc_localize_scores(rc_ctx* ctx, rc_cache* cache, int session, int t,
                             const float* latent, const int32_t* delta_ids_host, int n_delta,
                             float* scores, rc_stream stream);

/* Semantic-aware adaptive reuse scheduling (Section 3.3), host-only.
 * rc_prompt_similarity: Eq. 1, s = cos(e(tau-), e(tau+)) of two token
 *   embeddings (host arrays of dim floats), accumulated in double.
 * rc_reuse_schedule: Eq. 2, T_reuse = T if s >= tau_s else floor(rho T), and
 *   the per-step modes of an edited region for rc_step: RC_MODE_REUSE for
 *   t < T_reuse, RC_MODE_SPARSE after (modes_out: host array of T).  The
 *   paper sets rho = 0.2.
 * Errors: RC_ERR_INVALID_ARG (null, dim or T <= 0, zero embedding, rho
 * outside [0, 1], NaN). */
rc_status rc_prompt_similarity(const float* e_minus, const float* e_plus, int dim, float* s_out);
rc_status rc_reuse_schedule(float s, float tau_s, float rho, int T, uint8_t* modes_out);

/* CUDA Graph of one rc_step (no counterpart in the paper; serving
 * plumbing): the step's ~290 kernel launches for fixed arguments are
 * recorded once and replayed with one launch call.  The arguments are those
 * of rc_step; the graph keeps the device pointers (latent, dirty_idx,
 * dirty_count, the cache slots of (session, t)) and reads and writes their
 * CONTENTS at each replay, so a new edit region only needs new dirty_idx /
 * dirty_count contents (use D = -1 with a device count whose bound is N).
 * Mode schedule_host[t] and the host bound D are fixed at creation.  The
 * graph reuses the context's scratch: replays of graphs of one context are
 * serialised on one stream, like its steps.  Creation enqueues nothing on
 * the caller's streams; when the per-timestep embedding tables are stale
 * (see rc_set_global_weights) it computes them first, on a private stream
 * that it waits for.  A replay reads those tables but keeps the DDIM
 * coefficients of the schedule at creation: create graphs again after
 * rc_set_schedule or rc_set_global_weights.
 * Errors: as rc_step; RC_ERR_INVALID_ARG for a host-tier cache or while a
 * timing probe is enabled; RC_ERR_CUDA when capture or instantiation fails. */
typedef struct rc_graph rc_graph;
rc_status rc_step_graph_create(rc_ctx* ctx, rc_cache* cache, int session, float* latent, int t,
                               const uint8_t* schedule_host, const int32_t* dirty_idx, int D,
                               const int32_t* dirty_count, rc_graph** out);
/* Replays the graph on `stream`. */
rc_status rc_graph_launch(rc_graph* graph, rc_stream stream);
void rc_graph_destroy(rc_graph* graph);

/* Cross-session serving scheduler (no counterpart in the paper, which serves
 * one request at a time): editing sessions join and leave between steps,
 * and every tick runs ONE rc_step_batched over up to max_items of the turns
 * in progress, each at its own timestep, so that one pass over the weights
 * serves them all.  A turn = the steps t = 0 .. timesteps-1 of one session,
 * in order, each computed exactly as rc_step would compute it.  When more
 * turns are running than a tick takes, the least recently stepped go first
 * (ties: admission order), so every turn advances in round robin.  Host
 * state only; drive a server from one host thread, and let no other call
 * step the sessions it is running.
 *   rc_server_create   max_items in [1, the context's max_batch] (1 for a
 *                      host-tier cache).
 *   rc_server_admit    starts a turn of `session` (not already running):
 *                      latent f32 [in_ch][grid_h*patch][grid_w*patch]
 *                      device, in/out; schedule_host[timesteps] modes
 *                      (copied); dirty_idx / D / dirty_count as in rc_step,
 *                      read at each SPARSE step (borrowed until the turn
 *                      ends).
 *   rc_server_tick     one batched step on `stream`; sessions_out (host,
 *                      max_items entries, may be null) receives the sessions
 *                      stepped, *n_out their number (0 when no turn is
 *                      running).  A turn whose last step ran leaves the
 *                      server.  On an error nothing advances.
 *   rc_server_state    *next_t = the next step of the session's running
 *                      turn, or -1 when it has none.
 *   rc_server_running  number of turns in progress.
 * Errors: RC_ERR_INVALID_ARG, and those of rc_step_batched. */
typedef struct rc_server rc_server;
rc_status rc_server_create(rc_ctx* ctx, rc_cache* cache, int max_items, rc_server** out);
void rc_server_destroy(rc_server* server);
rc_status rc_server_admit(rc_server* server, int session, float* latent,
                          const uint8_t* schedule_host, const int32_t* dirty_idx, int D,
                          const int32_t* dirty_count);
rc_status rc_server_tick(rc_server* server, rc_stream stream, int* sessions_out, int* n_out);
rc_status rc_server_state(const rc_server* server, int session, int* next_t);
int rc_server_running(const rc_server* server);

/* Full-recompute baseline: rc_step with mode DENSE. */
rc_status rc_step_dense(rc_ctx* ctx, rc_cache* cache, int session, float* latent, int t,
                        rc_stream stream);

/* ------------------------------------------------------------- auxiliary */

/* The tensor-core GEMM of the block on its own: y = x W^T + b.
 *   x bf16 [rows][k], W bf16 [n][k], b f32 [n] (may be null), y f32 [rows][n].
 *   k % 64 == 0, n % 64 == 0, rows >= 0.
 * Provided so the GEMM can be checked and timed in isolation. */
rc_status rc_linear(rc_ctx* ctx, const void* x, const void* W, const float* b, float* y,
                    int rows, int n, int k, rc_stream stream);

/* The dirty-query attention of the block on its own (Section 3.3,
 * Region-Level Sparse Attention): for each of the context's heads h,
 * O[r][h*dh..] = softmax(Q_r,h K_h^T / sqrt(dh)) V_h over the Nk keys.
 *   Q bf16 [Nq][ldq], K and V bf16 [Nk][ldkv] (head h in columns h*dh ..
 *   h*dh+dh-1), O bf16 [Nq][ldo].  ldq, ldkv, ldo multiples of 8, >= heads*dh;
 *   pointers 16-byte aligned; Nq, Nk >= 0.
 * Provided so the attention kernel can be checked and timed in isolation. */
rc_status rc_attention(rc_ctx* ctx, const void* Q, int ldq, const void* K, const void* V,
                       int ldkv, int Nq, int Nk, void* O, int ldo, rc_stream stream);

/* Waits for `stream`, then reports (and clears) the context's device error
 * word: RC_ERR_DEVICE_ASSERT if a kernel met a bad index or count,
 * RC_ERR_TIMEOUT if a bounded wait gave up, RC_ERR_CUDA on a CUDA error. */
rc_status rc_sync(rc_ctx* ctx, rc_stream stream);

/* Timing probe.  rc_probe_enable(ctx, which, capacity) makes the context
 * record a pair of CUDA events on the launching stream around each of the
 * next `capacity` launches of kernel class `which` (RC_PROBE_GEMM: every
 * tensor-core GEMM of a block, five, or six when the cross-query projection
 * runs as its own GEMM; RC_PROBE_ATTENTION: the self- and the
 * cross-attention launch of a block;
 * RC_PROBE_LN: both LayerNorm-modulation launches of a block);
 * which = RC_PROBE_OFF disables it.  rc_probe_read waits for the recorded
 * events and returns the summed device time (ms) and the number of launches
 * recorded, then rearms the ring.  rc_probe_read_each does the same but
 * writes each launch's device time (ms, launch order) to the host array
 * ms_out[0 .. capacity) (caller-owned; launches beyond capacity are counted
 * in *launches but not written).  Errors: RC_ERR_INVALID_ARG, RC_ERR_CUDA. */
#define RC_PROBE_OFF 0
#define RC_PROBE_GEMM 1
#define RC_PROBE_ATTENTION 2
#define RC_PROBE_LN 3
rc_status rc_probe_enable(rc_ctx* ctx, int which, int capacity);
rc_status rc_probe_read(rc_ctx* ctx, double* total_ms, int* launches);
rc_status rc_probe_read_each(rc_ctx* ctx, float* ms_out, int capacity, int* launches);

/* Self-test of the device-side failure path (no counterpart in the paper):
 * every kernel of this library that waits on another agent (an mbarrier, a
 * flag) gives up after a bounded time, records RC_ERR_TIMEOUT in the
 * context's error word and returns, so the context stays usable.  This
 * entry point runs that bounded wait on its own: one thread polls a
 * context-owned device flag for at most timeout_us (1 .. 10^6)
 * microseconds; with set_flag = 0 nothing raises the flag, the wait gives
 * up and the next rc_sync returns RC_ERR_TIMEOUT; with set_flag = 1 the
 * flag is raised first and the wait ends at once.  Nothing faults or traps.
 * Errors: RC_ERR_INVALID_ARG. */
rc_status rc_selftest_wait(rc_ctx* ctx, int timeout_us, int set_flag, rc_stream stream);

/* Number of kernels this library has launched in the calling process. */
uint64_t rc_launch_count(void);

const char* rc_status_string(rc_status s);
const char* rc_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* REGIONCACHE_H */
