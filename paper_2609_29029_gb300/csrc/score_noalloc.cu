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
// array's name as a device address (on the host it names a stand-in object), so each call looks
// the address up with cudaGetSymbolAddress in the CUDA context current on the calling thread.  The
// address belongs to that context: a context rebuilt after cudaDeviceReset, or another context on
// the same device (a driver-API host), has its own copy of the array at another address, so an
// address is never reused across contexts.  The one exception is a call made while its stream is
// being captured, where the lookup (which may load the module) is not made: it takes the address
// recorded for the current context by an earlier call, so the first call in each context should
// come before any stream capture.
//
// All calls share the one array, and it keeps whatever the last call left in it.  Nothing needs
// clearing: every scratch element a call reads is written earlier by the same call.  Two calls
// whose work overlaps on the GPU (different streams, or different host threads) race on the
// array; callers must order them.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "rift_internal.h"

namespace {

static __device__ __align__(256) unsigned char g_score_scratch[RIFT_NOALLOC_SCORE_SCRATCH_BYTES];

// The addresses recorded by uncaptured calls, one per context id (a small table: a process rarely
// has more than one context per device).
constexpr int kMaxContexts = 64;
std::mutex g_mu;
unsigned long long g_ctx_id[kMaxContexts] = {};
void* g_ctx_ptr[kMaxContexts] = {};
int g_n_ctx = 0;

// Device address of g_score_scratch in the current context.
rift_status scratch_address(cudaStream_t stream, void** out) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(stream, &cs) != cudaSuccess) return RIFT_ERR_CUDA;
  const unsigned long long id = rift::current_context_id();
  std::lock_guard<std::mutex> lk(g_mu);
  int slot = -1;
  for (int i = 0; i < g_n_ctx; ++i)
    if (id != 0 && g_ctx_id[i] == id) slot = i;
  if (cs != cudaStreamCaptureStatusNone) {  // no lookup under capture: the recorded address or nothing
    if (slot < 0) return RIFT_ERR_UNSUPPORTED;
    *out = g_ctx_ptr[slot];
    return RIFT_OK;
  }
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_score_scratch) != cudaSuccess || !p) return RIFT_ERR_CUDA;
  if (id != 0) {
    if (slot < 0 && g_n_ctx < kMaxContexts) slot = g_n_ctx++;
    if (slot >= 0) {
      g_ctx_id[slot] = id;
      g_ctx_ptr[slot] = p;
    }
  }
  *out = p;
  return RIFT_OK;
}

}  // namespace

extern "C" rift_status rift_score_tiles_noalloc(const void* X, rift_dtype xdt, int N, int n_v, int d,
                                                const float* t, const float* B, int M, int knn_m,
                                                float* token_scores, float* tile_s_raw, float* tile_s,
                                                int* nbr, rift_stream_t stream) {
  const rift_status chk =
      rift::score_args_check(X, xdt, N, n_v, d, t, B, M, knn_m, token_scores, tile_s_raw, tile_s);
  if (chk != RIFT_OK) return chk;
  const size_t need = rift::score_layout(N, n_v, d, M).total;
  if (need > RIFT_NOALLOC_SCORE_SCRATCH_BYTES) return RIFT_ERR_CAPACITY;  // scene too large for the array
  void* ws = nullptr;
  const rift_status st = scratch_address(static_cast<cudaStream_t>(stream), &ws);
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
