// rift_score_tiles_noalloc: the relevance scoring of rift_score_tiles for callers that cannot
// allocate device memory.
//
// Some hosts of this library have no allocator to give it: a flight or edge program whose device
// memory is laid out once before the mission starts and never grows, or a plug-in running inside
// another runtime's memory pool with no way to obtain a workspace of its own.  For them this
// entry point takes its scratch (partial pooled sums, tile embeddings, kNN candidates) from a
// fixed array compiled into the library instead of from a caller-provided workspace.
//
// The array is a file-scope __device__ variable: every GPU that loads the library holds
// RIFT_NOALLOC_SCORE_SCRATCH_BYTES of it until the process exits.  Host code cannot use the
// array's name as a device address (on the host it names a stand-in object), so the first call
// on each device looks the address up with cudaGetSymbolAddress while that device is current and
// caches it.  That first call should therefore come before any stream capture.
//
// All calls share the one array, and it keeps whatever the last call left in it.  Nothing needs
// clearing: every scratch element a call reads is written earlier by the same call.  Two calls
// whose work overlaps on the GPU (different streams, or different host threads) race on the
// array; callers must order them.
#include <mutex>

#include "rift_internal.h"

namespace {

static __device__ __align__(256) unsigned char g_score_scratch[RIFT_NOALLOC_SCORE_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_score_scratch on the current device, looked up once per device.
rift_status scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return RIFT_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return RIFT_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_score_scratch) != cudaSuccess || !p) return RIFT_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return RIFT_OK;
}

}  // namespace

extern "C" rift_status rift_score_tiles_noalloc(const void* X, rift_dtype xdt, int N, int n_v, int d,
                                                const float* t, const float* B, int M, int knn_m,
                                                float* token_scores, float* tile_s_raw, float* tile_s,
                                                int* nbr, rift_stream_t stream) {
  if (N < 1 || N > RIFT_MAX_TILES || n_v < 1 || n_v > RIFT_MAX_NV || d < 64 || d > 8192 || d % 64 != 0)
    return RIFT_ERR_INVALID;
  if (!X || !t || !token_scores || !tile_s_raw || !tile_s) return RIFT_ERR_INVALID;
  if (xdt != RIFT_F32 && xdt != RIFT_BF16) return RIFT_ERR_INVALID;
  if (xdt == RIFT_F32 && d > 4096) return RIFT_ERR_UNSUPPORTED;
  if (M < 0 || M > 64 || (M > 0 && !B) || knn_m < 0 || knn_m > RIFT_MAX_KNN) return RIFT_ERR_INVALID;
  if (!rift::aligned16(X)) return RIFT_ERR_INVALID;
  const size_t need = rift::score_layout(N, n_v, d, M).total;
  if (need > RIFT_NOALLOC_SCORE_SCRATCH_BYTES) return RIFT_ERR_CAPACITY;  // scene too large for the array
  void* ws = nullptr;
  const rift_status st = scratch_address(&ws);
  if (st != RIFT_OK) return st;
  const int m = knn_m < N - 1 ? knn_m : N - 1;
  rift::prof_begin(RIFT_PROF_SCORE, static_cast<cudaStream_t>(stream));
  const int nk = rift::launch_score(X, xdt, N, n_v, d, t, B, M, m, token_scores, tile_s_raw, tile_s, nbr,
                                    static_cast<char*>(ws), static_cast<cudaStream_t>(stream));
  rift::prof_end(RIFT_PROF_SCORE, static_cast<cudaStream_t>(stream), nk < 0 ? 0 : nk);
  if (nk < 0) return RIFT_ERR_CUDA;
  RIFT_LAUNCH_CHECK();
  return RIFT_OK;
}
