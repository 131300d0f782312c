/*
 * rift.h -- C ABI of the GB300 (sm_103a) hot path of Rift: query-conditioned tile
 * pruning and elastic, per-tile token-budgeted prefill over a tiled scene.
 *
 * Calls, in the order the method runs them:
 *   rift_query_prep              Section 2.3 Stage 1: the query embedding t and the
 *                                background embeddings B_j that Eq. 1 compares against
 *   rift_score_tiles             Eq. 1 on every vision token and every tile, then the
 *                                kNN smoothing of Appendix B Step 2
 *   rift_select_budgeted_tokens  per-scene min-max and the tau threshold (Section 2.3
 *                                Stage 1, Appendix B Step 3), the budget argmax of Eq. 2
 *                                (Section 2.3 Stage 2), and each kept tile's top-b tokens
 *   rift_pack_ragged             one sequence per kept tile, [system | tokens | query],
 *                                packed back to back with varlen offsets
 *                                (rift_pack_ragged_at: a later query of a batch)
 *   rift_prefill_layers          the decoder prefill over the packed batch (Section 2.1)
 *
 * Conventions shared by every call
 *   - Every array argument is a DEVICE pointer owned by the caller, unless marked
 *     "host".  The library never allocates device memory: scratch comes from the
 *     caller's workspace `ws` (size from the matching *_workspace_bytes query; pass
 *     at least that many bytes, 256-byte aligned).  One exception: the library image
 *     holds a static device array of RIFT_NOALLOC_SCORE_SCRATCH_BYTES (64 MiB), the
 *     scratch of rift_score_tiles_noalloc, on every device that loads it.
 *   - Sizes are host ints.  Counts that only the device knows (n_kept, T) are written
 *     to device ints and can be read after rift_sync_status.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; 0 = the legacy default stream)
 *     and return RIFT_OK once the work is enqueued.  Argument errors that the host can
 *     see are returned at once and nothing is launched.  Errors that only the device can
 *     see (a non-finite score, a packed batch larger than its capacity, an id outside
 *     the vocabulary, a bounded wait that ran out) set a per-process device flag; the
 *     next rift_sync_status returns and clears it.
 *   - Nothing throws across this boundary; no call keeps a pointer after it returns.
 *   - Matrices are row-major.  bf16 is IEEE binary16-brain (1-8-7) stored in uint16.
 *   - Every fp32 value that decides an integer (a neighbour, a kept tile, a budget, a
 *     selected token) is computed in fp32 with the operation order documented below,
 *     and ties go to the lower index.
 */
#ifndef RIFT_H
#define RIFT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  RIFT_OK = 0,
  RIFT_ERR_INVALID = 1,     /* bad argument: null pointer, size out of range, misalignment */
  RIFT_ERR_CAPACITY = 2,    /* an output did not fit its capacity (e.g. T > max_T) */
  RIFT_ERR_NONFINITE = 3,   /* a NaN or Inf score reached a decision */
  RIFT_ERR_CUDA = 4,        /* a CUDA runtime call failed */
  RIFT_ERR_TIMEOUT = 5,     /* a bounded device-side wait gave up */
  RIFT_ERR_UNSUPPORTED = 6, /* a valid request the library does not implement */
  RIFT_ERR_BAD_ID = 7       /* a token or tile id outside its range */
} rift_status;

typedef enum { RIFT_F32 = 0, RIFT_BF16 = 1 } rift_dtype;

typedef void* rift_stream_t; /* cudaStream_t */

#define RIFT_MAX_BUDGETS 8
#define RIFT_MAX_NV 1024      /* vision tokens per tile */
#define RIFT_MAX_TILES 65536
#define RIFT_MAX_KNN 16

/* Stage-1 threshold and Stage-2 budget table (Section 2.3, Eq. 2).
 *   tau        keep tile i iff u_i >= tau, 0 <= tau <= 1 (Appendix B: tau = 0.37)
 *   n_c, C     candidate budgets, strictly ascending, each in [1, n_v]
 *              (the paper: {72, 144, 288, 432, 576})
 *   alpha_pos  profiled accuracy on tiles that contain the object, per c
 *   alpha_neg  profiled accuracy on tiles that do not, per c
 *   energy     profiled energy per c;  lambda  the accuracy-energy trade-off
 * U_i(c) = ((p_i * alpha_pos[c]) + ((1 - p_i) * alpha_neg[c])) - (lambda * energy[c]),
 * each operation a correctly rounded fp32 op; b_i = C[argmax_c U_i(c)], ties to the
 * lower index (the cheaper budget).
 *   ctx_num, ctx_den  the merge of Stage 2 (VisionZip's mechanism: keep the dominant tokens,
 *              merge the remainder): a budget b < n_v holds floor(ctx_num b / ctx_den)
 *              contextual tokens and b minus that many selected (dominant) tokens; ctx_num = 0
 *              turns the merge off (every budget token is selected).  0 <= ctx_num < ctx_den.
 *              VisionZip's split is 10 / 64. */
typedef struct {
  float tau;
  int n_c;
  int C[RIFT_MAX_BUDGETS];
  float alpha_pos[RIFT_MAX_BUDGETS];
  float alpha_neg[RIFT_MAX_BUDGETS];
  float energy[RIFT_MAX_BUDGETS];
  float lambda;
  int ctx_num, ctx_den;
} rift_policy;

/* A LLaMA/Vicuna-shaped decoder (Section 2.1; LLaVA-1.5-7B: 32 layers, d 4096, 32 heads
 * x 128, FFN 11008, eps 1e-6, rope_theta 1e4).  The per-layer fields are HOST arrays of
 * n_layers DEVICE pointers; projection weights are fp16 (the tensor-core operand type, and the
 * dtype of the LLaVA-1.5-7B checkpoint), norm gains bf16:
 *   w_qkv      [3d, d]   rows 0..d-1 = W_q, d..2d-1 = W_k, 2d..3d-1 = W_v (out x in)
 *   w_o        [d, d]
 *   w_gate_up  [2 ffn, d] W_gate and W_up interleaved in groups of 16 rows:
 *              rows 32g..32g+15 = W_gate rows 16g..16g+15, rows 32g+16..32g+31 = W_up
 *              rows 16g..16g+15 (ffn must be a multiple of 16)
 *   w_down     [d, ffn]
 *   g_attn, g_ffn [d]    RMSNorm gains;  g_final [d] (one device pointer)
 *   lm_head    [vocab, d] fp16, the untied output matrix (one device pointer), or NULL when no
 *              call asks for logits; vocab % 8 == 0 when it is given
 * Requirements: d % 64 == 0, head_dim in {64, 128}, n_heads * head_dim == d. */
typedef struct {
  int n_layers, d, n_heads, head_dim, ffn;
  float eps, rope_theta;
  const void* const* w_qkv;
  const void* const* w_o;
  const void* const* w_gate_up;
  const void* const* w_down;
  const void* const* g_attn;
  const void* const* g_ffn;
  const void* g_final;
  int vocab;
  const void* lm_head;
} rift_model;

/* Version of this ABI (bumped on any signature change). */
int rift_abi_version(void);

/* Human-readable name of a status code (static string, never NULL). */
const char* rift_status_string(rift_status s);

/* Waits for all work on `stream`, then returns and clears the device error flags set
 * by earlier calls (RIFT_OK if none).  If several flags are set, the most specific one
 * is returned (BAD_ID, NONFINITE, CAPACITY, TIMEOUT, in that order). */
rift_status rift_sync_status(rift_stream_t stream);

/* ---- a1. Query preparation (Section 2.3 Stage 1; Listing 1's E(phrase), E(terms)) ----
 * The paper embeds the query's object phrase and M background terms with RemoteCLIP.
 * Stand-in here: the decoder's own token embedding.
 *   embed       bf16 [vocab, d]
 *   phrase_ids  int32 [n_templates * n_phrase]: template k's ids at k*n_phrase
 *   bg_ids      int32 [M] (M may be 0; bg_ids may then be NULL)
 *   t           out fp32 [d]:   t = l2norm(mean_k l2norm(mean_q embed[phrase_ids[k][q]]))
 *   B           out fp32 [M,d]: B_j = l2norm(embed[bg_ids[j]]) (NULL allowed if M == 0)
 * Ids outside [0, vocab) set RIFT_ERR_BAD_ID. */
rift_status rift_query_prep(const void* embed, int vocab, int d,
                            const int* phrase_ids, int n_templates, int n_phrase,
                            const int* bg_ids, int M, float* t, float* B,
                            rift_stream_t stream);

/* ---- a2-a4. Relevance scores (Eq. 1) and kNN smoothing (Appendix B Step 2) ----
 *   X             [N, n_v, d] vision tokens, fp32 or bf16 (xdt)
 *   t, B          from rift_query_prep (B may be NULL if M == 0)
 *   knn_m         neighbours per tile; the call uses m = min(knn_m, N - 1), 0 <= knn_m <= 16
 *   token_scores  out fp32 [N, n_v]: r_ik = x_ik . w / ||x_ik||, w = t - (1/M) sum_j B_j
 *                 (Eq. 1 applied to each token)
 *   tile_s_raw    out fp32 [N]: s_i = V_i . w, V_i = P_i / ||P_i||, P_i = sum_k x_ik (Eq. 1)
 *   tile_s        out fp32 [N]: s~_i = (sum over {i} + NN(i) in ascending index of s_j)
 *                 / (m + 1), NN(i) = the m tiles j != i of largest V_i . V_j, ties to the lower
 *                 j (candidates found in fp32, ranked by their fp64-accumulated similarity)
 *   nbr           out int32 [N, m] (nullable): NN(i) in rank order
 * Limits: 1 <= N <= RIFT_MAX_TILES, 1 <= n_v <= RIFT_MAX_NV, 64 <= d <= 8192, d % 64 == 0,
 * 0 <= M <= 64; X 16-byte aligned. */
size_t rift_score_workspace_bytes(int N, int n_v, int d, int M);
rift_status rift_score_tiles(const void* X, rift_dtype xdt, int N, int n_v, int d,
                             const float* t, const float* B, int M, int knn_m,
                             float* token_scores, float* tile_s_raw, float* tile_s, int* nbr,
                             void* ws, size_t ws_bytes, rift_stream_t stream);

/* ---- rift_score_tiles without a workspace (no counterpart in the paper) ----
 * For callers that cannot allocate device memory at all -- e.g. an edge or flight program
 * whose device memory is planned once before launch, or a plug-in inside another runtime's
 * memory pool -- this variant of rift_score_tiles takes its scratch from a fixed array
 * compiled into the library (RIFT_NOALLOC_SCORE_SCRATCH_BYTES on every GPU that loads the
 * library, held until the process exits) and allocates nothing.  Arguments and outputs are
 * those of rift_score_tiles without ws/ws_bytes; results are the same.
 *   - A scene whose scratch (rift_score_workspace_bytes(N, n_v, d, M)) exceeds the array
 *     returns RIFT_ERR_CAPACITY and launches nothing (64 MiB holds N = 400 tiles at d = 4096).
 *   - Each call looks the array's device address up in the CUDA context current on the calling
 *     thread (each context has its own copy of the array).  A call made while its stream is being
 *     captured does not look it up but reuses the address an earlier call recorded for that
 *     context (RIFT_ERR_UNSUPPORTED if there was none): make the first call in each context
 *     before any stream capture.
 *   - All calls share the array and it keeps the last call's contents (nothing needs to start
 *     at zero).  Calls whose work overlaps on the GPU race on it: order them. */
#define RIFT_NOALLOC_SCORE_SCRATCH_BYTES (64u << 20)
rift_status rift_score_tiles_noalloc(const void* X, rift_dtype xdt, int N, int n_v, int d,
                                     const float* t, const float* B, int M, int knn_m,
                                     float* token_scores, float* tile_s_raw, float* tile_s, int* nbr,
                                     rift_stream_t stream);

/* ---- a5-a7. Prune, budget and select (Section 2.3; Appendix B Steps 3-4) ----
 *   token_scores, tile_s  from rift_score_tiles (tile_s = the smoothed scores)
 *   p          fp32 [N] (nullable): p_i, the probability that tile i holds the object;
 *              NULL uses p_i = u_i (stand-in for the paper's learned predictor)
 *   policy     host pointer, see rift_policy
 *   u          out fp32 [N]: (s~_i - min) / (max - min), or 1 for all if max == min
 *   kept       out int32 [N]: the kept tiles (u_i >= tau) in ascending order, first n_kept
 *   n_kept     out int32 [1]
 *   budgets    out int32 [N]: b_j for kept slot j (first n_kept entries)
 *   sel        out int32 [N * n_v]: kept slot j's selected token indices at sel_off[j],
 *              the s_j largest token scores (ties to the lower index), ascending, with
 *              s_j = b_j less its contextual tokens (s_j = b_j without the merge)
 *   sel_off    out int32 [N + 1]: exclusive prefix sum of the s_j; entries j > n_kept
 *              are set to the total
 * A NaN or Inf among the scores that are read sets RIFT_ERR_NONFINITE. */
size_t rift_select_workspace_bytes(int N, int n_v);
rift_status rift_select_budgeted_tokens(const float* token_scores, const float* tile_s,
                                        int N, int n_v, const float* p,
                                        const rift_policy* policy,
                                        float* u, int* kept, int* n_kept, int* budgets,
                                        int* sel, int* sel_off,
                                        void* ws, size_t ws_bytes, rift_stream_t stream);

/* ---- One scene sharded over several ranks (GPUs or hosts) ----
 * Every step of the method is per tile except two that need the whole scene: the kNN smoothing of
 * Appendix B Step 2 (each tile's m most similar tiles, anywhere in the scene) and the per-scene
 * min-max of Section 2.3 Stage 1 (Listing 1's u = (s - min) / (max - min)).  A scene split into
 * contiguous shards of tiles runs, on each rank:
 *   rift_score_shard                   Eq. 1 on the shard's tokens and tiles, and its tile
 *                                      embeddings V
 *   (exchange: every rank's V and tile_s_raw, gathered in tile order)
 *   rift_smooth_rows                   the smoothing of the shard's tiles against the whole scene
 *   rift_score_range                   (min, max) of the shard's smoothed scores
 *   (exchange: the scene's min of the mins and max of the maxes)
 *   rift_select_budgeted_tokens_ranged prune, budgets and top-b of the shard's tiles with the
 *                                      scene's range
 *   rift_pack_ragged                   the shard's kept tiles, as for one rank
 * The exchanges are the caller's (two collectives; the library makes no collective call).  With
 * the same inputs every score, neighbour, kept tile, budget and selected token equals what
 * rift_score_tiles and rift_select_budgeted_tokens compute on the whole scene on one rank (the
 * fp32 sums of a tile's scores and of a pair's similarity do not depend on the split).
 *
 *   rift_score_shard: X [N_local, n_v, d] the shard's tokens; t, B, M as for rift_score_tiles;
 *     token_scores out fp32 [N_local, n_v], tile_s_raw out fp32 [N_local] (Eq. 1, as
 *     rift_score_tiles), V out fp32 [N_local, d]: V_i = P_i / ||P_i||, P_i = sum_k x_ik.
 *     ws: rift_score_shard_workspace_bytes(N_local, n_v, d) bytes.
 *   rift_smooth_rows: V fp32 [N, d] and tile_s_raw fp32 [N] of the whole scene (16-byte aligned
 *     V); the rows row0 .. row0 + n_rows - 1 are smoothed: tile_s out fp32 [n_rows] and nbr out
 *     int32 [n_rows, m] (nullable) for those rows, m = min(knn_m, N - 1), exactly as
 *     rift_score_tiles' tile_s and nbr.  ws: rift_smooth_workspace_bytes(N, n_rows, d) bytes.
 *   rift_score_range: range out fp32 [2] = (min, max) of tile_s [n]; a NaN or Inf sets
 *     RIFT_ERR_NONFINITE.
 *   rift_select_budgeted_tokens_ranged: rift_select_budgeted_tokens for N tiles of a larger scene,
 *     with u_i = (s~_i - s_range[0]) / (s_range[1] - s_range[0]) (device fp32 [2], the scene's
 *     min and max; u = 1 for every tile if they are equal).  kept holds shard-local tile
 *     indices.  A non-finite range or score sets RIFT_ERR_NONFINITE. */
size_t rift_score_shard_workspace_bytes(int N_local, int n_v, int d);
rift_status rift_score_shard(const void* X, rift_dtype xdt, int N_local, int n_v, int d,
                             const float* t, const float* B, int M, float* token_scores,
                             float* tile_s_raw, float* V, void* ws, size_t ws_bytes,
                             rift_stream_t stream);
size_t rift_smooth_workspace_bytes(int N, int n_rows, int d);
rift_status rift_smooth_rows(const float* V, const float* tile_s_raw, int N, int d, int row0,
                             int n_rows, int knn_m, float* tile_s, int* nbr, void* ws,
                             size_t ws_bytes, rift_stream_t stream);
rift_status rift_score_range(const float* tile_s, int n, float* range, rift_stream_t stream);
rift_status rift_select_budgeted_tokens_ranged(const float* token_scores, const float* tile_s,
                                               int N, int n_v, const float* s_range,
                                               const float* p, const rift_policy* policy,
                                               float* u, int* kept, int* n_kept, int* budgets,
                                               int* sel, int* sel_off, rift_stream_t stream);

/* ---- Predictor features (Section 2.3, Stage 2: the features of the paper's p_i predictor,
 * computed for the listed tiles, e.g. the kept ones, whose p_i the budget rule uses) ----
 *   X, xdt, N, n_v, d   the scene; t, B, M   as for rift_score_tiles (Eq. 1's query and
 *              background embeddings); token_scores  from rift_score_tiles
 *   tiles      int32 [*n_tiles] tile indices (device), or NULL for every tile (slot j = tile j)
 *   features   out fp32 [N, RIFT_N_FEATURES]: slot j = (s_TL, s_TR, s_BL, s_BR, r_max, r_mean,
 *              r_std): Eq. 1 of each quadrant's pooled embedding (quadrants of the g x g token grid,
 *              n_v = g^2 with g even, tokens in row-major grid order; top-left, top-right,
 *              bottom-left, bottom-right), then the max, mean and population standard deviation
 *              of the tile's token scores
 *   V          out fp32 [N, d] (nullable): slot j's tile embedding, l2norm of its pooled tokens
 *   ws         rift_features_workspace_bytes(N, d) bytes
 * n_v not an even square returns RIFT_ERR_UNSUPPORTED. */
#define RIFT_N_FEATURES 7
size_t rift_features_workspace_bytes(int N, int d);
rift_status rift_tile_features(const void* X, rift_dtype xdt, int N, int n_v, int d, const float* t,
                               const float* B, int M, const float* token_scores, const int* tiles,
                               const int* n_tiles, float* features, float* V, void* ws,
                               size_t ws_bytes, rift_stream_t stream);

/* ---- a7b. Merge of the unselected tokens (Section 2.3, Stage 2: VisionZip's mechanism keeps
 * the dominant tokens and merges the remainder) ----
 * For kept slot j with m_j = budgets[j] - (sel_off[j+1] - sel_off[j]) contextual tokens (see
 * rift_policy ctx_num): the R_j tokens of the tile that were not selected, in ascending index,
 * give the targets rest[q floor(R_j / m_j)], q < m_j; every other remaining token joins the target
 * with the largest cosine similarity to it (ties to the lower target; decided at ~fp64 accuracy),
 * and contextual token q is the mean of its group, target included (fp32 sums in ascending token
 * index, stored as bf16).
 *   X, xdt, N, n_v, d   the scene (as rift_score_tiles); kept, n_kept, budgets, sel, sel_off
 *              from rift_select_budgeted_tokens
 *   ctx        out bf16 [max_ctx, d]: slot j's contextual tokens at rows ctx_off[j] ..
 *   ctx_off    out int32 [N + 1]: exclusive prefix sum of the m_j; entries j > n_kept are the
 *              total (all zero when the merge is off)
 *   ctx_target out int32 [max_ctx]: the target token index of each contextual token
 *   ws         rift_merge_workspace_bytes(N, n_v) bytes
 * More than max_ctx contextual tokens set RIFT_ERR_CAPACITY (the excess is not written). */
size_t rift_merge_workspace_bytes(int N, int n_v);
rift_status rift_merge_contextual(const void* X, rift_dtype xdt, int N, int n_v, int d,
                                  const int* kept, const int* n_kept, const int* budgets,
                                  const int* sel, const int* sel_off, void* ctx, int max_ctx,
                                  int* ctx_off, int* ctx_target, void* ws, size_t ws_bytes,
                                  rift_stream_t stream);

/* ---- a8. Ragged packing (the per-tile VLM prompt of Appendix B Step 5) ----
 *   X, xdt, N, n_v, d     as for rift_score_tiles (fp32 tokens are rounded to bf16)
 *   kept, n_kept, sel, sel_off   from rift_select_budgeted_tokens
 *   sys_ids    int32 [S] system-prompt ids;  query_ids int32 [Q] query ids
 *   embed      bf16 [vocab, d]
 *   ctx, ctx_off  contextual tokens and offsets from rift_merge_contextual, or both NULL
 *   packed     out bf16 [max_T, d]: sequence j = [embed[sys_ids] | X[kept[j], sel_j] |
 *              ctx rows ctx_off[j] .. ctx_off[j+1] | embed[query_ids]], sequences back to back
 *              in kept order
 *   cu_seqlens out int32 [N + 1]: cu_seqlens[j] = j (S + Q) + sel_off[j] + ctx_off[j]; entries
 *              j > n_kept are set to T
 *   positions  out int32 [max_T]: position of each packed row in its sequence (0..L_j-1)
 *   T          out int32 [1]: total packed rows
 * T > max_T sets RIFT_ERR_CAPACITY (rows beyond max_T are not written). */
rift_status rift_pack_ragged(const void* X, rift_dtype xdt, int N, int n_v, int d,
                             const int* kept, const int* n_kept,
                             const int* sel, const int* sel_off,
                             const int* sys_ids, int S, const int* query_ids, int Q,
                             const void* embed, int vocab, const void* ctx, const int* ctx_off,
                             void* packed, int max_T, int* cu_seqlens, int* positions, int* T,
                             rift_stream_t stream);

/* ---- a8 for a batch of scene queries (several queries in one prefill) ----
 * The paper answers one scene query at a time; a server batches several.  Packing them into
 * one batch is rift_pack_ragged once per query, each time with packed, positions and
 * cu_seqlens pointing at the query's part of the batch buffers (after the rows and sequences
 * of the queries before it) and row_base = the rows before it, so that the batch's
 * cu_seqlens holds absolute row offsets:
 *   cu_seqlens[j] = row_base + (the rift_pack_ragged value); T out = this query's rows alone;
 *   max_T = the rows left in the batch buffer.  row_base = 0 is rift_pack_ragged.
 * The sequences stay independent (no attention across them), so each query's final hidden
 * states are those of its own prefill, row for row.
 * row_base < 0 returns RIFT_ERR_INVALID. */
rift_status rift_pack_ragged_at(const void* X, rift_dtype xdt, int N, int n_v, int d,
                                const int* kept, const int* n_kept,
                                const int* sel, const int* sel_off,
                                const int* sys_ids, int S, const int* query_ids, int Q,
                                const void* embed, int vocab, const void* ctx, const int* ctx_off,
                                void* packed, int max_T, int* cu_seqlens, int* positions, int* T,
                                int row_base, rift_stream_t stream);

/* ---- a9. Decoder prefill (Section 2.1) ----
 *   hidden     bf16 [max_T, d]: in, the packed batch; out, the final hidden states (after the
 *              final RMSNorm) of its first T rows.  The residual stream is kept in fp32 in the
 *              workspace.
 *   T          int32 [1] DEVICE: the packed rows, as rift_pack_ragged writes it; read by the
 *              kernels, so the call can be enqueued right after the packing with no host read-back.
 *              NULL: max_T is the row count.
 *   max_T      host: the rows that hidden, positions and kv_out hold (a count above it is clamped
 *              to it; rift_pack_ragged has then already raised RIFT_ERR_CAPACITY)
 *   cu_seqlens int32 [max_seqs + 1], positions int32 [max_T] from rift_pack_ragged
 *   n_seq      int32 [1] DEVICE: the packed sequences (rift_select_budgeted_tokens' n_kept);
 *              NULL: max_seqs is the count.  Above max_seqs sets RIFT_ERR_CAPACITY (the first
 *              max_seqs are prefilled); so does a sequence that ends past max_T (it and the ones
 *              after it are left out).
 *   max_seqs   host: an upper bound on the sequence count (sizes the workspace and the logits)
 *   max_len    an upper bound on every sequence length (host int)
 * Each layer: h += W_o Attn(RoPE(q), RoPE(k), v) with x = RMSNorm(h) g_attn, causal within
 * each sequence only; h += W_down(SiLU(W_gate x) * (W_up x)) with x = RMSNorm(h) g_ffn.
 * GEMM and attention operands are fp16 (normalised activations, q/k/v, softmax weights,
 * attention output, SwiGLU output), accumulation fp32, residual stream fp32.  The launches are
 * sized for the capacities and stop at the device counts.
 * Optional outputs (NULL = not written):
 *   kv_out      fp16 [n_layers][2][max_T][d]: per layer the keys after RoPE ([l][0]) and the values
 *               ([l][1]) of every packed row, heads contiguous: the KV cache the prefill builds
 *               (Section 2.1), as rift_decode_step reads it.  16-byte aligned.
 *   last_logits fp32 [max_seqs, vocab]: logits of each sequence's last row,
 *               (RMSNorm(h_last) g_final) lm_head^T; needs m->lm_head.  16-byte aligned. */
size_t rift_prefill_workspace_bytes(const rift_model* m, int max_T, int max_seqs, int max_len);
rift_status rift_prefill_layers(const rift_model* m, void* hidden, const int* T, int max_T,
                                const int* cu_seqlens, const int* n_seq, int max_seqs, int max_len,
                                const int* positions, void* kv_out, float* last_logits,
                                void* ws, size_t ws_bytes, rift_stream_t stream);

/* ---- Prefill over a shared system prompt (an extension of Section 2.1's prefill, not in the paper:
 * the S system-prompt rows open every per-tile sequence at positions 0..S-1, so their hidden
 * states and cache are the same in every sequence) ----
 * The prompt is prefilled once and every sequence's remaining rows (its b_i vision tokens and
 * the query; pack them with S = 0) are prefilled over the prompt's cache.  Results equal
 * rift_prefill_layers on the full sequences (row for row, up to the fp32 summation order).
 *   sys_ids     int32 [S] (device), embed bf16 [vocab, d]
 *   prefix_hidden out bf16 [S, d]: the prompt's final hidden states
 *   prefix_kv   out fp16 [n_layers][2][S][d]: the prompt's cache (the layout of kv_out)
 *   hidden      bf16 [max_T, d] in/out: the suffix rows (packed with S = 0), then their final
 *               hidden states; T (device, nullable), max_T, cu_seqlens [max_seqs + 1], n_seq (device,
 *               nullable), max_seqs and positions [max_T] (0-based) over them, as for
 *               rift_prefill_layers
 *   max_len     an upper bound on S + every suffix length
 *   last_logits out fp32 [max_seqs, vocab] (nullable; needs m->lm_head): each sequence's last row
 *   ws          rift_prefill_shared_prefix_workspace_bytes(m, max_T, max_seqs, max_len, S) bytes */
size_t rift_prefill_shared_prefix_workspace_bytes(const rift_model* m, int max_T, int max_seqs, int max_len,
                                                  int S);
rift_status rift_prefill_shared_prefix(const rift_model* m, const int* sys_ids, int S, const void* embed,
                                       int vocab, void* prefix_hidden, void* prefix_kv, void* hidden,
                                       const int* T, int max_T, const int* cu_seqlens, const int* n_seq,
                                       int max_seqs, int max_len, const int* positions, float* last_logits,
                                       void* ws, size_t ws_bytes, rift_stream_t stream);

/* ---- Decode step after the prefill (Section 2.1: decoding extends the prefilled KV cache one
 * token at a time) ----
 * One new token per sequence: sequence i's token token_ids[i] (an id into embed [vocab_embed, d]
 * bf16) at position L_i = cu_seqlens[i+1] - cu_seqlens[i], attending to that sequence's cached
 * rows and to itself, through every layer and the final RMSNorm.
 *   kv_cache   fp16 [n_layers][2][T][d] as written by rift_prefill_layers (kv_out) for the
 *              same cu_seqlens; T is the row capacity it was written with (that call's max_T)
 *   max_len    an upper bound on every L_i + 1 (host int, at most 32768)
 *   hidden_out bf16 [n_seq, d] final hidden states of the new tokens, or NULL
 *   kv_new     fp16 [n_layers][2][n_seq][d] the new tokens' keys (after RoPE) and values, or NULL
 *   logits     fp32 [n_seq, vocab] (needs m->lm_head), or NULL
 * An id outside [0, vocab_embed) sets RIFT_ERR_BAD_ID (its row is computed from a zero
 * embedding); L_i + 1 > max_len sets RIFT_ERR_CAPACITY or RIFT_ERR_BAD_ID. */
size_t rift_decode_workspace_bytes(const rift_model* m, int n_seq, int max_len);
rift_status rift_decode_step(const rift_model* m, const void* kv_cache, int T, const int* cu_seqlens,
                             int n_seq, int max_len, const int* token_ids, const void* embed,
                             int vocab_embed, void* hidden_out, void* kv_new, float* logits,
                             void* ws, size_t ws_bytes, rift_stream_t stream);

/* ---- The linear layer of a9 on its own (the GEMM every prefill layer runs four times) ----
 * out = A W^T with A fp16 [M, K], W fp16 [N, K] (both row-major, K contiguous), products
 * accumulated in fp32 on the tensor cores, then:
 *   RIFT_EPI_STORE_F16   out fp16 [M, N] = A W^T
 *   RIFT_EPI_RESID_F32   out fp32 [M, N] += A W^T      (the residual adds after W_o and W_down)
 *   RIFT_EPI_SWIGLU      W holds gate and up rows interleaved in groups of 16 (as w_gate_up);
 *                        out fp16 [M, N/2] = SiLU(x W_gate^T) * (x W_up^T), N % 32 == 0
 * K % 8 == 0 and N % 8 == 0; A, W, out 16-byte aligned.  M == 0 is a no-op. */
#define RIFT_EPI_STORE_F16 0
#define RIFT_EPI_RESID_F32 1
#define RIFT_EPI_SWIGLU 2
rift_status rift_linear(const void* A, const void* W, int M, int N, int K, int epilogue, void* out,
                        rift_stream_t stream);

/* ---- The attention of a9 on its own (varlen, causal within each packed sequence) ----
 *   qkv   fp16 [T, 3 n_heads head_dim]: per row q | k | v, each with heads contiguous, RoPE
 *         already applied to q and k (as the prefill's QKV step leaves it)
 *   cu_seqlens int32 [n_seq + 1]; out fp16 [T, n_heads head_dim] = softmax(q k^T / sqrt(head_dim)
 *   + causal mask) v per sequence and head, softmax in fp32 with fp16 weights, fp32 accumulation
 *   ws    rift_attention_workspace_bytes(T, n_seq) bytes (the q-block schedule)
 * head_dim in {64, 128}. */
size_t rift_attention_workspace_bytes(int max_T, int max_seqs);
rift_status rift_attention_varlen(const void* qkv, int T, const int* cu_seqlens, int n_seq, int n_heads,
                                  int head_dim, void* out, void* ws, size_t ws_bytes, rift_stream_t stream);

/* ---- Instrumentation for benchmarks (does not change any result) ----
 * Kernel classes timed by the profiler: */
#define RIFT_PROF_GEMM 0      /* the prefill GEMMs (QKV, O, gate/up, down) */
#define RIFT_PROF_ATTN 1      /* varlen causal attention (with its q-block schedule) */
#define RIFT_PROF_NORM 2      /* RMSNorm kernels */
#define RIFT_PROF_ROPE 3      /* RoPE table and rotation */
#define RIFT_PROF_SCORE 4     /* query prep, token/tile scores, kNN */
#define RIFT_PROF_SELECT 5    /* prune, budgets, top-b */
#define RIFT_PROF_PACK 6      /* ragged packing */
#define RIFT_PROF_CLASSES 7
/* ---- Diagnostics ----
 * Enqueues a kernel whose pipeline wait can never complete (an mbarrier no one arrives at),
 * through the same bounded wait as the library's kernels: after ~4 s it gives up, and the next
 * rift_sync_status returns RIFT_ERR_TIMEOUT with the context still usable.  A check of the
 * failure path, not of any result. */
rift_status rift_check_wait_timeout(rift_stream_t stream);

/* rift_profile_enable(1) starts recording a pair of CUDA events on the launch stream around
 * every kernel launch of the classes above (0 stops).  rift_profile_read waits for the recorded
 * events, writes per-class totals (ms[c] in milliseconds, launches[c]) for n_classes classes and
 * clears the record.  Returns RIFT_ERR_CUDA if an event query fails. */
void rift_profile_enable(int on);
rift_status rift_profile_read(double* ms, long long* launches, int n_classes);
/* Number of kernels this library has launched since it was loaded (always counted). */
long long rift_launch_count(void);

#ifdef __cplusplus
}
#endif
#endif /* RIFT_H */
