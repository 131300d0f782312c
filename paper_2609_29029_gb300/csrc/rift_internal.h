// Internal launcher declarations shared by the translation units of the Rift library.
#pragma once

#include "rift_common.cuh"

namespace rift {

// Benchmark instrumentation: events around launches of a class (when enabled) and a launch
// counter.  prof_begin/prof_end bracket the launches; n is the number of kernels inside.
void prof_begin(int cls, cudaStream_t st);
void prof_end(int cls, cudaStream_t st, int n);

// Per-translation-unit device error flags (read and cleared by rift_sync_status).
unsigned int read_clear_err_score();
unsigned int read_clear_err_select();
unsigned int read_clear_err_pack();
unsigned int read_clear_err_prefill();
unsigned int read_clear_err_gemm();

// ---- score.cu ----
// The token pass over N tiles (Eq. 1 per token, pooled sums): w and the partial pooled sums.
struct ShardLayout {
  int chunk_tokens, n_chunks;
  size_t w_off, cnt_off, ppart_off, total;
};
ShardLayout shard_layout(int N, int n_v, int d);
// The kNN smoothing of n_rows rows against all N tiles (Appendix B Step 2).
struct SmoothLayout {
  size_t top_off, split_off, gram_off, splitk_off, splitk_bytes, total;
};
SmoothLayout smooth_layout(int N, int n_rows, int d);
// rift_score_tiles: V [N, d], then the token pass's scratch, which the smoothing of all N rows
// reuses once V is formed.
struct ScoreLayout {
  ShardLayout T;
  SmoothLayout S;
  size_t V_off, tokens_off, smooth_off, total;
};
ScoreLayout score_layout(int N, int n_v, int d, int M);
// The host-side argument checks shared by the scoring entry points (rift_score_tiles and
// rift_score_tiles_noalloc): RIFT_OK, or the status the call returns without launching.
rift_status score_args_check(const void* X, rift_dtype xdt, int N, int n_v, int d, const float* t, const float* B,
                             int M, int knn_m, const float* token_scores, const float* tile_s_raw,
                             const float* tile_s);
int launch_query_prep(const void* embed, int vocab, int d, const int* phrase_ids, int n_tmpl,
                      int n_phrase, const int* bg_ids, int M, float* t, float* B, cudaStream_t st);
// Returns the number of kernels launched, or -1 if a launch could not be set up.
int launch_score(const void* X, rift_dtype xdt, int N, int n_v, int d, const float* t, const float* B,
                 int M, int m, float* token_scores, float* s_raw, float* s_tilde, int* nbr, char* ws,
                 cudaStream_t st);
// a2, a3 on N tiles: token scores, tile scores and the tile embeddings V [N, d] (ws: shard_layout).
// S16 (nullable): also write the whole scene's Gram operand (the layout of launch_smooth's split
// rows, [hi | lo] per tile), so that launch_smooth can skip its split.
int launch_score_tokens(const void* X, rift_dtype xdt, int N, int n_v, int d, const float* t, const float* B,
                        int M, float* token_scores, float* s_raw, float* V, char* ws, cudaStream_t st,
                        uint16_t* S16 = nullptr);
// a4 for tiles row0 .. row0 + n_rows - 1 of a scene of N tiles (V [N, d], s_raw [N]); s_tilde and
// nbr are indexed by the local row (ws: smooth_layout).
// split_done: the split operands in ws were written by launch_score_tokens (whole scene).
int launch_smooth(const float* V, const float* s_raw, int N, int d, int row0, int n_rows, int m, float* s_tilde,
                  int* nbr, char* ws, cudaStream_t st, bool split_done = false);
// range = (min, max) of n scores.
void launch_score_range(const float* s, int n, float* range, cudaStream_t st);

// ---- select.cu ----
// s_range (nullable): the scene's (min, max) of tile_s, when the N tiles are a shard of it.
void launch_select(const float* token_scores, const float* tile_s, int N, int n_v, const float* p,
                   const rift_policy& pol, float* u, int* kept, int* n_kept, int* budgets, int* sel,
                   int* sel_off, cudaStream_t st, const float* s_range = nullptr);

// ---- features.cu ----
struct FeaturesLayout {
  size_t w_off, qsum_off, total;
};
FeaturesLayout features_layout(int N, int d);
int launch_features(const void* X, rift_dtype xdt, int N, int n_v, int d, int g, const float* t, const float* B, int M,
                    const float* token_scores, const int* tiles, const int* n_tiles, float* features, float* V,
                    char* ws, cudaStream_t st);

// ---- merge.cu ----
struct MergeLayout {
  size_t rest_off, assign_off, tnorm_off, memb_off, gstart_off, pos_off, tinv_off, cand_off, total;
};
#define RIFT_MERGE_MAX_D 8192
MergeLayout merge_layout(int N, int n_v);
unsigned int read_clear_err_merge();
// Returns the number of kernels launched, or -1 if a launch could not be set up.
int launch_merge(const void* X, rift_dtype xdt, int N, int n_v, int d, const int* kept, const int* n_kept,
                 const int* budgets, const int* sel, const int* sel_off, uint16_t* ctx, int max_ctx, int* ctx_off,
                 int* ctx_target, char* ws, cudaStream_t st);

// ---- pack.cu ----
void launch_pack(const void* X, rift_dtype xdt, int N, int n_v, int d, const int* kept,
                 const int* n_kept, const int* sel, const int* sel_off, const int* sys_ids, int S,
                 const int* query_ids, int Q, const void* embed, int vocab, const void* ctx, const int* ctx_off,
                 void* packed, int max_T, int* cu_seqlens, int* positions, int* T, int row_base,
                 cudaStream_t st);

// ---- prefill (prefill.cu, gemm.cu, attention.cu) ----
struct PrefillLayout {
  size_t h32_off, xn_off, qkv_off, attn_off, act_off, rope_off, sched_off, last32_off, last16_off, total;
  int max_qblocks;
};
PrefillLayout prefill_layout(const rift_model& m, int max_T, int max_seqs, int max_len);
// T, n_seq: the row and sequence capacities (host); T_dev, n_seq_dev (nullable): the device
// counts the launches read, clamped to the capacities (without them, T and n_seq are the counts).
// The kv_out layout [n_layers][2][T][d] uses the capacity T as its row stride.
// prefix_kv (optional): fp16 [n_layers][2][S_pre][d] cache of a prefix shared by every sequence
// (each sequence's rows attend to it first; their positions are positions[] + S_pre).
int launch_prefill(const rift_model& m, void* hidden, int T, const int* T_dev, const int* cu_seqlens, int n_seq,
                   const int* n_seq_dev, int max_len, const int* positions, void* kv_out, float* last_logits,
                   char* ws, cudaStream_t st, const void* prefix_kv = nullptr, int S_pre = 0);
struct SharedPrefixLayout {
  size_t prefill_bytes, cu_off, pos_off, total;
};
SharedPrefixLayout shared_prefix_layout(const rift_model& m, int max_T, int max_seqs, int max_len, int S);
int launch_prefill_shared_prefix(const rift_model& m, const int* sys_ids, int S, const void* embed, int vocab,
                                 void* prefix_hidden, void* prefix_kv, void* hidden, int T, const int* T_dev,
                                 const int* cu_seqlens, int n_seq, const int* n_seq_dev, int max_len,
                                 const int* positions, float* last_logits, char* ws, cudaStream_t st);
struct DecodeLayout {
  size_t h32_off, x0_off, xn_off, qkv_off, attn_off, act_off, rope_off, pos_off, dpart_off, split_off, split_bytes,
      total;
};
DecodeLayout decode_layout(const rift_model& m, int n_seq, int max_len);
int launch_decode(const rift_model& m, const void* kv_cache, int T, const int* cu_seqlens, int n_seq, int max_len,
                  const int* token_ids, const void* embed, int vocab_embed, void* hidden_out, void* kv_new,
                  float* logits, char* ws, cudaStream_t st);

// GEMM: C[M, N] = A[M, K] . B[N, K]^T (fp16 operands, fp32 accumulation) + epilogue.
enum GemmEpilogue {
  EPI_STORE_BF16 = 0,  // C fp16 [M, N] (name kept from the ABI's numbering)
  EPI_RESID_F32 = 1,   // R fp32 [M, N] += acc
  EPI_SWIGLU = 2,      // N = 2F interleaved in 16-column groups; C fp16 [M, F] = silu(g) * u
  EPI_QKV_ROPE = 3,    // C fp16 [M, N]; columns < rope_cols get rotate-half RoPE at positions[row]
  EPI_STORE_F32 = 4,   // C fp32 [M, N] = acc * out_scale
  EPI_STORE_F32_T = 5  // C fp32 [N, M] = acc (transposed; the swapped few-row products)
};
struct EpiParams {
  const int* positions = nullptr;  // [M] position of each row (EPI_QKV_ROPE)
  const float2* rope = nullptr;    // [max_len, head_dim/2] (cos, sin)
  int rope_cols = 0;               // q and k columns: 2 d
  int head_dim = 0;
  int max_len = 0;
  int pos_offset = 0;              // added to positions[row] (rows that follow a shared prefix)
  float out_scale = 1.f;           // EPI_STORE_F32
  // EPI_RESID_F32 with split scratch: also norm_out fp16 [M, N] = RMSNorm(C) norm_gain (bf16 [N])
  const void* norm_gain = nullptr;
  uint16_t* norm_out = nullptr;
  float norm_eps = 0.f;
  // Device row count (nullable): the product covers rows min(M, *m_dev); M is then the capacity
  // the operands and the output are sized for.  Not used with split-K.
  const int* m_dev = nullptr;
  // EPI_STORE_F32 of a symmetric product (A = B's first M rows, M <= N <= M + 7: a Gram matrix):
  // only the tiles on and above the diagonal are computed, each off-diagonal one stored twice
  // (as itself and transposed).  Honoured on the SM-pair path; the other paths compute every tile.
  int symmetric = 0;
  // K-block remap of the two operands (the kNN's split-operand Gram): with kmap_d > 0 each operand
  // row is stored as [hi | lo], kmap_d K-blocks each (K = 3 kmap_d blocks of 64), and read as
  // kmap_a / kmap_b: 1 = [hi | hi | lo], 2 = [hi | lo | hi] along K (0 = as stored).
  int kmap_d = 0;
  int kmap_a = 0, kmap_b = 0;
};
// split_ws (optional): scratch for split-K partial products; with it, products whose tiles leave
// most SMs idle run as (tile, K-slice) units plus a reduction kernel.
// pdl: launch as a programmatic dependent of the previous kernel in the stream (decode step).
int launch_gemm(const void* A, const void* B, int M, int N, int K, int epi, void* C,
                cudaStream_t st, const EpiParams& ep = EpiParams(), void* split_ws = nullptr,
                size_t split_ws_bytes = 0, bool pdl = false);
// b_const: B does not depend on earlier kernels (constant weights), so a programmatic dependent
// launch may request its first tiles before waiting for the kernel before it.
int launch_gemm_tc(const void* A, const void* B, int M, int N, int K, int epi, void* C, const EpiParams& ep,
                   cudaStream_t st, void* split_ws = nullptr, size_t split_ws_bytes = 0, bool pdl = false,
                   bool b_const = true);
int launch_wait_timeout_check(cudaStream_t st);
// Merge screening on the tensor cores (bf16 tokens): per kept slot and 128-token block, the two
// best merge targets (by x.t / ||t||) of every unselected non-target token.  targets: bf16
// [max_ctx, d] target rows; tinv [max_ctx] = 1 / ||t||; pos [N, n_v] = position of each token
// among the slot's unselected ones (-1 if selected); cand [N, n_v] out, indexed by that position.
int launch_merge_screen(const uint16_t* X, int N, int n_v, int d, const int* kept, const int* n_kept,
                        const int* sel_off, const int* ctx_off, int max_ctx, const uint16_t* targets,
                        const float* tinv, const int* pos, int2* cand, cudaStream_t st);

// Varlen causal attention (attention_tc.cu): q-block schedule built once per prefill from
// cu_seqlens, then one launch per layer.  qkv fp16 [T, 3 d], out fp16 [T, d].
int attention_max_qblocks(int max_T, int max_seqs);
// The schedule holds n_sched_max + 1 entries (the last: the count in use).  n_seq_dev (nullable):
// a device sequence count clamped to n_seq; sequences ending past row_cap rows are dropped.
void launch_attention_schedule(const int* cu_seqlens, int n_seq, const int* n_seq_dev, int row_cap, int4* sched,
                               int n_sched_max, cudaStream_t st);
// prefix_k, prefix_v (optional): fp16 [S_pre, d] keys (after RoPE) and values of a prefix that every
// sequence attends to before its own rows.
int launch_attention(const void* qkv, int T, const int* cu_seqlens, int n_seq, int n_heads, int head_dim,
                     const int4* sched, int n_sched_max, void* out, cudaStream_t st, const void* prefix_k = nullptr,
                     const void* prefix_v = nullptr, int S_pre = 0);
unsigned int read_clear_err_attn();

}  // namespace rift
