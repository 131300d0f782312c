// The C ABI of include/rift.h: argument validation, workspace carving and launches on the
// caller's stream.  Nothing here allocates device memory.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <mutex>
#include <vector>

#include "rift_internal.h"

using namespace rift;

namespace {

constexpr size_t WS_ALIGN = 256;

bool ws_ok(const void* ws, size_t have, size_t need) {
  if (need == 0) return true;
  return ws != nullptr && have >= need && (reinterpret_cast<uintptr_t>(ws) % WS_ALIGN) == 0;
}

bool dims_ok(int N, int n_v, int d) {
  return N >= 1 && N <= RIFT_MAX_TILES && n_v >= 1 && n_v <= RIFT_MAX_NV && d >= 64 && d <= 8192 &&
         d % 64 == 0;
}

struct ProfRec {
  int cls, n;
  cudaEvent_t a, b;
};
std::mutex g_prof_mu;
bool g_prof_on = false;
std::vector<cudaEvent_t> g_pool;
std::vector<ProfRec> g_recs;
cudaEvent_t g_open[RIFT_PROF_CLASSES] = {};
std::atomic<long long> g_launches{0};

cudaEvent_t pool_get() {
  if (!g_pool.empty()) {
    cudaEvent_t e = g_pool.back();
    g_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

}  // namespace

namespace rift {

unsigned long long current_context_id() {
  static PFN_cuCtxGetCurrent_v4000 get_current = nullptr;
  static PFN_cuCtxGetId_v12000 get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(p);
  });
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS)
    return 0;
  return id;
}

void prof_begin(int cls, cudaStream_t st) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (!g_prof_on) return;
  cudaEvent_t e = pool_get();
  if (e && cudaEventRecord(e, st) == cudaSuccess) g_open[cls] = e;
}

void prof_end(int cls, cudaStream_t st, int n) {
  g_launches += n;
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (!g_prof_on || !g_open[cls]) return;
  cudaEvent_t e = pool_get();
  if (e && cudaEventRecord(e, st) == cudaSuccess) g_recs.push_back({cls, n, g_open[cls], e});
  g_open[cls] = nullptr;
}

rift_status score_args_check(const void* X, rift_dtype xdt, int N, int n_v, int d, const float* t, const float* B,
                             int M, int knn_m, const float* token_scores, const float* tile_s_raw,
                             const float* tile_s) {
  if (!dims_ok(N, n_v, d) || !X || !t || !token_scores || !tile_s_raw || !tile_s) return RIFT_ERR_INVALID;
  if (xdt != RIFT_F32 && xdt != RIFT_BF16) return RIFT_ERR_INVALID;
  if (xdt == RIFT_F32 && d > 4096) return RIFT_ERR_UNSUPPORTED;
  if (M < 0 || M > 64 || (M > 0 && !B) || knn_m < 0 || knn_m > RIFT_MAX_KNN) return RIFT_ERR_INVALID;
  if (!aligned16(X)) return RIFT_ERR_INVALID;
  return RIFT_OK;
}

}  // namespace rift

extern "C" {

void rift_profile_enable(int on) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  g_prof_on = on != 0;
}

rift_status rift_profile_read(double* ms, long long* launches, int n_classes) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  rift_status st = RIFT_OK;
  for (int c = 0; c < n_classes; ++c) {
    if (ms) ms[c] = 0.0;
    if (launches) launches[c] = 0;
  }
  for (const ProfRec& r : g_recs) {
    float t = 0.f;
    if (cudaEventSynchronize(r.b) != cudaSuccess || cudaEventElapsedTime(&t, r.a, r.b) != cudaSuccess) st = RIFT_ERR_CUDA;
    if (r.cls < n_classes) {
      if (ms) ms[r.cls] += t;
      if (launches) launches[r.cls] += r.n;
    }
    g_pool.push_back(r.a);
    g_pool.push_back(r.b);
  }
  g_recs.clear();
  return st;
}

long long rift_launch_count(void) { return g_launches.load(); }

int rift_abi_version(void) { return 5; }

const char* rift_status_string(rift_status s) {
  switch (s) {
    case RIFT_OK: return "ok";
    case RIFT_ERR_INVALID: return "invalid argument";
    case RIFT_ERR_CAPACITY: return "output capacity exceeded";
    case RIFT_ERR_NONFINITE: return "non-finite score";
    case RIFT_ERR_CUDA: return "CUDA runtime error";
    case RIFT_ERR_TIMEOUT: return "device wait timed out";
    case RIFT_ERR_UNSUPPORTED: return "unsupported";
    case RIFT_ERR_BAD_ID: return "id out of range";
  }
  return "unknown status";
}

rift_status rift_sync_status(rift_stream_t stream) {
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return RIFT_ERR_CUDA;
  unsigned int f = read_clear_err_score() | read_clear_err_select() | read_clear_err_pack() |
                   read_clear_err_prefill() | read_clear_err_gemm() | read_clear_err_attn() | read_clear_err_merge();
  if (cudaGetLastError() != cudaSuccess) return RIFT_ERR_CUDA;
  if (f & RIFT_EBIT_BADID) return RIFT_ERR_BAD_ID;
  if (f & RIFT_EBIT_NONFINITE) return RIFT_ERR_NONFINITE;
  if (f & RIFT_EBIT_CAPACITY) return RIFT_ERR_CAPACITY;
  if (f & RIFT_EBIT_TIMEOUT) return RIFT_ERR_TIMEOUT;
  return RIFT_OK;
}

rift_status rift_query_prep(const void* embed, int vocab, int d, const int* phrase_ids, int n_templates,
                            int n_phrase, const int* bg_ids, int M, float* t, float* B,
                            rift_stream_t stream) {
  if (!embed || !phrase_ids || !t || vocab < 1 || d < 64 || d > 8192 || d % 64 != 0 || n_templates < 1 ||
      n_phrase < 1 || M < 0 || M > 64 || (M > 0 && (!bg_ids || !B)))
    return RIFT_ERR_INVALID;
  prof_begin(RIFT_PROF_SCORE, static_cast<cudaStream_t>(stream));
  const int nk = launch_query_prep(embed, vocab, d, phrase_ids, n_templates, n_phrase, bg_ids, M, t, B,
                                   static_cast<cudaStream_t>(stream));
  prof_end(RIFT_PROF_SCORE, static_cast<cudaStream_t>(stream), nk);
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

size_t rift_score_workspace_bytes(int N, int n_v, int d, int M) {
  if (!dims_ok(N, n_v, d)) return 0;
  return score_layout(N, n_v, d, M).total;
}

rift_status rift_score_tiles(const void* X, rift_dtype xdt, int N, int n_v, int d, const float* t,
                             const float* B, int M, int knn_m, float* token_scores, float* tile_s_raw,
                             float* tile_s, int* nbr, void* ws, size_t ws_bytes, rift_stream_t stream) {
  const rift_status chk = score_args_check(X, xdt, N, n_v, d, t, B, M, knn_m, token_scores, tile_s_raw, tile_s);
  if (chk != RIFT_OK) return chk;
  const size_t need = rift_score_workspace_bytes(N, n_v, d, M);
  if (!ws_ok(ws, ws_bytes, need)) return RIFT_ERR_INVALID;
  const int m = std::min(knn_m, N - 1);
  prof_begin(RIFT_PROF_SCORE, static_cast<cudaStream_t>(stream));
  const int nk = launch_score(X, xdt, N, n_v, d, t, B, M, m, token_scores, tile_s_raw, tile_s, nbr,
                              static_cast<char*>(ws), static_cast<cudaStream_t>(stream));
  prof_end(RIFT_PROF_SCORE, static_cast<cudaStream_t>(stream), nk < 0 ? 0 : nk);
  if (nk < 0) return RIFT_ERR_CUDA;
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

size_t rift_select_workspace_bytes(int N, int n_v) {
  (void)N;
  (void)n_v;
  return 0;
}

static rift_status select_args_check(const float* token_scores, const float* tile_s, int N, int n_v,
                                     const rift_policy* policy, const float* u, const int* kept, const int* n_kept,
                                     const int* budgets, const int* sel, const int* sel_off) {
  if (!token_scores || !tile_s || !policy || !u || !kept || !n_kept || !budgets || !sel || !sel_off)
    return RIFT_ERR_INVALID;
  if (N < 1 || N > RIFT_MAX_TILES || n_v < 1 || n_v > RIFT_MAX_NV) return RIFT_ERR_INVALID;
  const rift_policy& pol = *policy;
  if (!(pol.tau >= 0.f && pol.tau <= 1.f)) return RIFT_ERR_INVALID;
  if (pol.n_c < 1 || pol.n_c > RIFT_MAX_BUDGETS) return RIFT_ERR_INVALID;
  for (int c = 0; c < pol.n_c; ++c) {
    if (pol.C[c] < 1 || pol.C[c] > n_v) return RIFT_ERR_INVALID;
    if (c > 0 && pol.C[c] <= pol.C[c - 1]) return RIFT_ERR_INVALID;
    if (!std::isfinite(pol.alpha_pos[c]) || !std::isfinite(pol.alpha_neg[c]) || !std::isfinite(pol.energy[c]))
      return RIFT_ERR_INVALID;
  }
  if (!std::isfinite(pol.lambda)) return RIFT_ERR_INVALID;
  if (pol.ctx_num < 0 || pol.ctx_den < 1 || pol.ctx_num >= pol.ctx_den) return RIFT_ERR_INVALID;
  return RIFT_OK;
}

rift_status rift_select_budgeted_tokens(const float* token_scores, const float* tile_s, int N, int n_v,
                                        const float* p, const rift_policy* policy, float* u, int* kept,
                                        int* n_kept, int* budgets, int* sel, int* sel_off, void* ws,
                                        size_t ws_bytes, rift_stream_t stream) {
  (void)ws;
  (void)ws_bytes;
  const rift_status chk =
      select_args_check(token_scores, tile_s, N, n_v, policy, u, kept, n_kept, budgets, sel, sel_off);
  if (chk != RIFT_OK) return chk;
  prof_begin(RIFT_PROF_SELECT, static_cast<cudaStream_t>(stream));
  launch_select(token_scores, tile_s, N, n_v, p, *policy, u, kept, n_kept, budgets, sel, sel_off,
                static_cast<cudaStream_t>(stream));
  prof_end(RIFT_PROF_SELECT, static_cast<cudaStream_t>(stream), 2);
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

// ---- one scene sharded over several ranks (a shard of its tiles per rank) ----

size_t rift_score_shard_workspace_bytes(int N_local, int n_v, int d) {
  if (!dims_ok(N_local, n_v, d)) return 0;
  return shard_layout(N_local, n_v, d).total;
}

rift_status rift_score_shard(const void* X, rift_dtype xdt, int N_local, int n_v, int d, const float* t,
                             const float* B, int M, float* token_scores, float* tile_s_raw, float* V, void* ws,
                             size_t ws_bytes, rift_stream_t stream) {
  if (!V) return RIFT_ERR_INVALID;
  const rift_status chk = score_args_check(X, xdt, N_local, n_v, d, t, B, M, 0, token_scores, tile_s_raw, V);
  if (chk != RIFT_OK) return chk;
  if (!ws_ok(ws, ws_bytes, rift_score_shard_workspace_bytes(N_local, n_v, d))) return RIFT_ERR_INVALID;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  prof_begin(RIFT_PROF_SCORE, st);
  const int nk = launch_score_tokens(X, xdt, N_local, n_v, d, t, B, M, token_scores, tile_s_raw, V,
                                     static_cast<char*>(ws), st);
  prof_end(RIFT_PROF_SCORE, st, nk);
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

size_t rift_smooth_workspace_bytes(int N, int n_rows, int d) {
  if (N < 1 || N > RIFT_MAX_TILES || n_rows < 1 || n_rows > N || d < 64 || d > 8192 || d % 64 != 0) return 0;
  return smooth_layout(N, n_rows, d).total;
}

rift_status rift_smooth_rows(const float* V, const float* tile_s_raw, int N, int d, int row0, int n_rows, int knn_m,
                             float* tile_s, int* nbr, void* ws, size_t ws_bytes, rift_stream_t stream) {
  if (!V || !tile_s_raw || !tile_s || N < 1 || N > RIFT_MAX_TILES || d < 64 || d > 8192 || d % 64 != 0)
    return RIFT_ERR_INVALID;
  if (row0 < 0 || n_rows < 1 || row0 + n_rows > N || knn_m < 0 || knn_m > RIFT_MAX_KNN) return RIFT_ERR_INVALID;
  if (!aligned16(V)) return RIFT_ERR_INVALID;
  if (!ws_ok(ws, ws_bytes, rift_smooth_workspace_bytes(N, n_rows, d))) return RIFT_ERR_INVALID;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int m = std::min(knn_m, N - 1);
  prof_begin(RIFT_PROF_SCORE, st);
  const int nk = launch_smooth(V, tile_s_raw, N, d, row0, n_rows, m, tile_s, nbr, static_cast<char*>(ws), st);
  prof_end(RIFT_PROF_SCORE, st, nk < 0 ? 0 : nk);
  if (nk < 0) return RIFT_ERR_CUDA;
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

rift_status rift_score_range(const float* tile_s, int n, float* range, rift_stream_t stream) {
  if (!tile_s || !range || n < 1 || n > RIFT_MAX_TILES) return RIFT_ERR_INVALID;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  prof_begin(RIFT_PROF_SELECT, st);
  launch_score_range(tile_s, n, range, st);
  prof_end(RIFT_PROF_SELECT, st, 1);
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

rift_status rift_select_budgeted_tokens_ranged(const float* token_scores, const float* tile_s, int N, int n_v,
                                               const float* s_range, const float* p, const rift_policy* policy,
                                               float* u, int* kept, int* n_kept, int* budgets, int* sel,
                                               int* sel_off, rift_stream_t stream) {
  if (!s_range) return RIFT_ERR_INVALID;
  const rift_status chk =
      select_args_check(token_scores, tile_s, N, n_v, policy, u, kept, n_kept, budgets, sel, sel_off);
  if (chk != RIFT_OK) return chk;
  prof_begin(RIFT_PROF_SELECT, static_cast<cudaStream_t>(stream));
  launch_select(token_scores, tile_s, N, n_v, p, *policy, u, kept, n_kept, budgets, sel, sel_off,
                static_cast<cudaStream_t>(stream), s_range);
  prof_end(RIFT_PROF_SELECT, static_cast<cudaStream_t>(stream), 2);
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

rift_status rift_pack_ragged(const void* X, rift_dtype xdt, int N, int n_v, int d, const int* kept,
                             const int* n_kept, const int* sel, const int* sel_off, const int* sys_ids, int S,
                             const int* query_ids, int Q, const void* embed, int vocab, const void* ctx,
                             const int* ctx_off, void* packed, int max_T, int* cu_seqlens, int* positions, int* T,
                             rift_stream_t stream) {
  return rift_pack_ragged_at(X, xdt, N, n_v, d, kept, n_kept, sel, sel_off, sys_ids, S, query_ids, Q, embed, vocab,
                             ctx, ctx_off, packed, max_T, cu_seqlens, positions, T, 0, stream);
}

rift_status rift_pack_ragged_at(const void* X, rift_dtype xdt, int N, int n_v, int d, const int* kept,
                                const int* n_kept, const int* sel, const int* sel_off, const int* sys_ids, int S,
                                const int* query_ids, int Q, const void* embed, int vocab, const void* ctx,
                                const int* ctx_off, void* packed, int max_T, int* cu_seqlens, int* positions,
                                int* T, int row_base, rift_stream_t stream) {
  if (!dims_ok(N, n_v, d) || !X || !kept || !n_kept || !sel || !sel_off || !embed || !packed || !cu_seqlens ||
      !positions || !T || row_base < 0)
    return RIFT_ERR_INVALID;
  if (xdt != RIFT_F32 && xdt != RIFT_BF16) return RIFT_ERR_INVALID;
  if (S < 0 || Q < 0 || (S > 0 && !sys_ids) || (Q > 0 && !query_ids) || vocab < 1 || max_T < 0)
    return RIFT_ERR_INVALID;
  if (!aligned16(X) || !aligned16(embed) || !aligned16(packed)) return RIFT_ERR_INVALID;
  if ((ctx == nullptr) != (ctx_off == nullptr) || (ctx && !aligned16(ctx))) return RIFT_ERR_INVALID;
  prof_begin(RIFT_PROF_PACK, static_cast<cudaStream_t>(stream));
  launch_pack(X, xdt, N, n_v, d, kept, n_kept, sel, sel_off, sys_ids, S, query_ids, Q, embed, vocab, ctx, ctx_off,
              packed, max_T, cu_seqlens, positions, T, row_base, static_cast<cudaStream_t>(stream));
  prof_end(RIFT_PROF_PACK, static_cast<cudaStream_t>(stream), 2);
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

size_t rift_features_workspace_bytes(int N, int d) {
  if (N < 1 || N > RIFT_MAX_TILES || d < 64 || d > 8192 || d % 64 != 0) return 0;
  return features_layout(N, d).total;
}

rift_status rift_tile_features(const void* X, rift_dtype xdt, int N, int n_v, int d, const float* t, const float* B,
                               int M, const float* token_scores, const int* tiles, const int* n_tiles,
                               float* features, float* V, void* ws, size_t ws_bytes, rift_stream_t stream) {
  if (!dims_ok(N, n_v, d) || !X || !t || !token_scores || !features) return RIFT_ERR_INVALID;
  if (xdt != RIFT_F32 && xdt != RIFT_BF16) return RIFT_ERR_INVALID;
  if (M < 0 || M > 64 || (M > 0 && !B) || (tiles == nullptr) != (n_tiles == nullptr)) return RIFT_ERR_INVALID;
  if (!aligned16(X) || !aligned16(features) || (V && !aligned16(V))) return RIFT_ERR_INVALID;
  if (!ws_ok(ws, ws_bytes, features_layout(N, d).total)) return RIFT_ERR_INVALID;
  int g = 0;
  while ((g + 1) * (g + 1) <= n_v) ++g;
  if (g * g != n_v || g % 2 != 0) return RIFT_ERR_UNSUPPORTED;
  prof_begin(RIFT_PROF_SCORE, static_cast<cudaStream_t>(stream));
  const int nk = launch_features(X, xdt, N, n_v, d, g, t, B, M, token_scores, tiles, n_tiles, features, V,
                                 static_cast<char*>(ws), static_cast<cudaStream_t>(stream));
  prof_end(RIFT_PROF_SCORE, static_cast<cudaStream_t>(stream), nk);
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

size_t rift_merge_workspace_bytes(int N, int n_v) {
  if (N < 1 || N > RIFT_MAX_TILES || n_v < 1 || n_v > RIFT_MAX_NV) return 0;
  return merge_layout(N, n_v).total;
}

rift_status rift_merge_contextual(const void* X, rift_dtype xdt, int N, int n_v, int d, const int* kept,
                                  const int* n_kept, const int* budgets, const int* sel, const int* sel_off, void* ctx,
                                  int max_ctx, int* ctx_off, int* ctx_target, void* ws, size_t ws_bytes,
                                  rift_stream_t stream) {
  if (!dims_ok(N, n_v, d) || !X || !kept || !n_kept || !budgets || !sel || !sel_off || !ctx_off || !ctx_target ||
      max_ctx < 0 || (max_ctx > 0 && !ctx))
    return RIFT_ERR_INVALID;
  if (xdt != RIFT_F32 && xdt != RIFT_BF16) return RIFT_ERR_INVALID;
  if (!aligned16(X) || (ctx && !aligned16(ctx))) return RIFT_ERR_INVALID;
  if (!ws_ok(ws, ws_bytes, merge_layout(N, n_v).total)) return RIFT_ERR_INVALID;
  prof_begin(RIFT_PROF_SELECT, static_cast<cudaStream_t>(stream));
  const int nk = launch_merge(X, xdt, N, n_v, d, kept, n_kept, budgets, sel, sel_off, static_cast<uint16_t*>(ctx),
                              max_ctx, ctx_off, ctx_target, static_cast<char*>(ws), static_cast<cudaStream_t>(stream));
  if (nk < 0) return RIFT_ERR_CUDA;
  prof_end(RIFT_PROF_SELECT, static_cast<cudaStream_t>(stream), nk);
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

static bool model_ok(const rift_model* m) {
  if (!m) return false;
  if (m->n_layers < 1 || m->d < 64 || m->d > 8192 || m->d % 64 != 0) return false;
  if (m->head_dim != 64 && m->head_dim != 128) return false;
  if (m->n_heads < 1 || m->n_heads * m->head_dim != m->d) return false;
  if (m->ffn < 16 || m->ffn % 16 != 0) return false;
  if (!(m->eps > 0.f) || !(m->rope_theta > 0.f)) return false;
  if (!m->w_qkv || !m->w_o || !m->w_gate_up || !m->w_down || !m->g_attn || !m->g_ffn || !m->g_final)
    return false;
  for (int l = 0; l < m->n_layers; ++l) {
    const void* p[6] = {m->w_qkv[l], m->w_o[l], m->w_gate_up[l], m->w_down[l], m->g_attn[l], m->g_ffn[l]};
    for (const void* q : p)
      if (!q || !aligned16(q)) return false;
  }
  return aligned16(m->g_final);
}

rift_status rift_check_wait_timeout(rift_stream_t stream) {
  launch_wait_timeout_check(static_cast<cudaStream_t>(stream));
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

size_t rift_prefill_workspace_bytes(const rift_model* m, int max_T, int max_seqs, int max_len) {
  if (!model_ok(m) || max_T < 0 || max_seqs < 0 || max_len < 1) return 0;
  return prefill_layout(*m, max_T, max_seqs, max_len).total;
}

static bool lm_head_ok(const rift_model* m) {
  return m->lm_head && aligned16(m->lm_head) && m->vocab >= 8 && m->vocab % 8 == 0;
}

rift_status rift_prefill_layers(const rift_model* m, void* hidden, const int* T, int max_T, const int* cu_seqlens,
                                const int* n_seq, int max_seqs, int max_len, const int* positions, void* kv_out,
                                float* last_logits, void* ws, size_t ws_bytes, rift_stream_t stream) {
  if (!model_ok(m) || !hidden || !cu_seqlens || !positions || max_T < 0 || max_seqs < 0 || max_len < 1)
    return RIFT_ERR_INVALID;
  if (max_T > 0 && max_seqs < 1) return RIFT_ERR_INVALID;
  if (!aligned16(hidden) || (kv_out && !aligned16(kv_out)) || (last_logits && !aligned16(last_logits)))
    return RIFT_ERR_INVALID;
  if (last_logits && !lm_head_ok(m)) return RIFT_ERR_INVALID;
  const size_t need = prefill_layout(*m, max_T, max_seqs, max_len).total;
  if (!ws_ok(ws, ws_bytes, need)) return RIFT_ERR_INVALID;
  if (launch_prefill(*m, hidden, max_T, T, cu_seqlens, max_seqs, n_seq, max_len, positions, kv_out, last_logits,
                     static_cast<char*>(ws), static_cast<cudaStream_t>(stream)))
    return RIFT_ERR_INVALID;
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

size_t rift_prefill_shared_prefix_workspace_bytes(const rift_model* m, int max_T, int max_seqs, int max_len, int S) {
  if (!model_ok(m) || max_T < 0 || max_seqs < 0 || max_len < 1 || S < 1 || S > max_len) return 0;
  return shared_prefix_layout(*m, max_T, max_seqs, max_len, S).total;
}

rift_status rift_prefill_shared_prefix(const rift_model* m, const int* sys_ids, int S, const void* embed, int vocab,
                                       void* prefix_hidden, void* prefix_kv, void* hidden, const int* T, int max_T,
                                       const int* cu_seqlens, const int* n_seq, int max_seqs, int max_len,
                                       const int* positions, float* last_logits, void* ws, size_t ws_bytes,
                                       rift_stream_t stream) {
  if (!model_ok(m) || !sys_ids || !embed || !prefix_hidden || !prefix_kv || S < 1 || vocab < 1 || max_T < 0 ||
      max_seqs < 0 || max_len < 1 || S > max_len)
    return RIFT_ERR_INVALID;
  if (max_T > 0 && (!hidden || !cu_seqlens || !positions || max_seqs < 1)) return RIFT_ERR_INVALID;
  if (!aligned16(embed) || !aligned16(prefix_hidden) || !aligned16(prefix_kv) || (hidden && !aligned16(hidden)) ||
      (last_logits && !aligned16(last_logits)))
    return RIFT_ERR_INVALID;
  if (last_logits && !lm_head_ok(m)) return RIFT_ERR_INVALID;
  if (!ws_ok(ws, ws_bytes, shared_prefix_layout(*m, max_T, max_seqs, max_len, S).total)) return RIFT_ERR_INVALID;
  if (launch_prefill_shared_prefix(*m, sys_ids, S, embed, vocab, prefix_hidden, prefix_kv, hidden, max_T, T,
                                   cu_seqlens, max_seqs, n_seq, max_len, positions, last_logits,
                                   static_cast<char*>(ws), static_cast<cudaStream_t>(stream)))
    return RIFT_ERR_INVALID;
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

size_t rift_decode_workspace_bytes(const rift_model* m, int n_seq, int max_len) {
  if (!model_ok(m) || n_seq < 0 || max_len < 1 || max_len > 32768) return 0;
  return decode_layout(*m, n_seq, max_len).total;
}

rift_status rift_decode_step(const rift_model* m, const void* kv_cache, int T, const int* cu_seqlens, int n_seq,
                             int max_len, const int* token_ids, const void* embed, int vocab_embed,
                             void* hidden_out, void* kv_new, float* logits, void* ws, size_t ws_bytes,
                             rift_stream_t stream) {
  if (!model_ok(m) || !kv_cache || !cu_seqlens || !token_ids || !embed || T < 0 || n_seq < 0 || max_len < 1 ||
      max_len > 32768 || vocab_embed < 1)
    return RIFT_ERR_INVALID;
  if (!aligned16(kv_cache) || !aligned16(embed) || (hidden_out && !aligned16(hidden_out)) ||
      (kv_new && !aligned16(kv_new)) || (logits && !aligned16(logits)))
    return RIFT_ERR_INVALID;
  if (logits && !lm_head_ok(m)) return RIFT_ERR_INVALID;
  const size_t need = decode_layout(*m, n_seq, max_len).total;
  if (!ws_ok(ws, ws_bytes, need)) return RIFT_ERR_INVALID;
  if (launch_decode(*m, kv_cache, T, cu_seqlens, n_seq, max_len, token_ids, embed, vocab_embed, hidden_out, kv_new,
                    logits, static_cast<char*>(ws), static_cast<cudaStream_t>(stream)))
    return RIFT_ERR_INVALID;
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

rift_status rift_linear(const void* A, const void* W, int M, int N, int K, int epilogue, void* out,
                        rift_stream_t stream) {
  if (!A || !W || !out || M < 0 || N < 1 || K < 1) return RIFT_ERR_INVALID;
  if (epilogue < RIFT_EPI_STORE_F16 || epilogue > RIFT_EPI_SWIGLU) return RIFT_ERR_INVALID;
  if (K % 8 != 0 || N % 8 != 0 || (epilogue == RIFT_EPI_SWIGLU && N % 32 != 0)) return RIFT_ERR_INVALID;
  if (!aligned16(A) || !aligned16(W) || !aligned16(out)) return RIFT_ERR_INVALID;
  if (M == 0) return RIFT_OK;
  if (launch_gemm(A, W, M, N, K, epilogue, out, static_cast<cudaStream_t>(stream))) return RIFT_ERR_CUDA;
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

size_t rift_attention_workspace_bytes(int max_T, int max_seqs) {
  if (max_T <= 0 || max_seqs < 0) return 0;  // no rows: nothing to schedule
  return (size_t)(attention_max_qblocks(max_T, max_seqs) + 1) * sizeof(int4);
}

rift_status rift_attention_varlen(const void* qkv, int T, const int* cu_seqlens, int n_seq, int n_heads,
                                  int head_dim, void* out, void* ws, size_t ws_bytes, rift_stream_t stream) {
  if (!qkv || !cu_seqlens || !out || T < 0 || n_seq < 0 || n_heads < 1) return RIFT_ERR_INVALID;
  if (head_dim != 64 && head_dim != 128) return RIFT_ERR_INVALID;
  if (T > 0 && n_seq < 1) return RIFT_ERR_INVALID;
  if (!aligned16(qkv) || !aligned16(out)) return RIFT_ERR_INVALID;
  const size_t need = rift_attention_workspace_bytes(T, n_seq);
  if (!ws_ok(ws, ws_bytes, need)) return RIFT_ERR_INVALID;
  if (T == 0) return RIFT_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int4* sched = static_cast<int4*>(ws);
  const int n_max = attention_max_qblocks(T, n_seq);
  prof_begin(RIFT_PROF_ATTN, st);
  launch_attention_schedule(cu_seqlens, n_seq, nullptr, T, sched, n_max, st);
  if (launch_attention(qkv, T, cu_seqlens, n_seq, n_heads, head_dim, sched, n_max, out, st)) return RIFT_ERR_CUDA;
  prof_end(RIFT_PROF_ATTN, st, 2);
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}

}  // extern "C"
