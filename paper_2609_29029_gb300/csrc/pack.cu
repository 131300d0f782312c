// Ragged packing on sm_103a: one sequence per kept tile, [system | selected tokens | query],
// back to back, with cu_seqlens and per-row positions.
//
// Each packed row is an 8 KB (d = 4096, bf16) copy.  A CTA owns 32 rows of one sequence; a
// warp moves one row with 16-byte loads and stores.  The system and query rows come from the
// embedding table and stay in L2 across sequences; the vision rows stream from X once.
#include "rift_internal.h"

namespace rift {

__device__ unsigned int g_err_pack;

unsigned int read_clear_err_pack() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_err_pack, sizeof(v));
  cudaMemcpyToSymbol(g_err_pack, &z, sizeof(z));
  return v;
}

constexpr int PK_ROWS = 32;
constexpr int PK_THREADS = 256;

// cu_seqlens[j] = min(j, n) (S + Q) + sel_off[min(j, n)], T = cu_seqlens[n].
__global__ void seqlens_kernel(const int* __restrict__ n_kept, const int* __restrict__ sel_off, int N,
                               int S, int Q, int max_T, int* __restrict__ cu, int* __restrict__ T) {
  const int n = *n_kept;
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j <= N; j += gridDim.x * blockDim.x) {
    const int jj = min(j, n);
    const int v = jj * (S + Q) + sel_off[jj];
    cu[j] = v;
    if (j == N) {
      *T = v;
      if (v > max_T) atomicOr(&g_err_pack, RIFT_EBIT_CAPACITY);
    }
  }
}

template <typename XT>
__global__ void __launch_bounds__(PK_THREADS) pack_kernel(
    const XT* __restrict__ X, int N, int n_v, int d, const int* __restrict__ kept,
    const int* __restrict__ n_kept, const int* __restrict__ sel, const int* __restrict__ sel_off,
    const int* __restrict__ sys_ids, int S, const int* __restrict__ query_ids, int Q,
    const uint16_t* __restrict__ embed, int vocab, uint16_t* __restrict__ packed, int max_T,
    int* __restrict__ positions) {
  const int j = blockIdx.x;
  if (j >= *n_kept) return;
  const int so = sel_off[j];
  const int b = sel_off[j + 1] - so;
  const int L = S + b + Q;
  const int base = j * (S + Q) + so;
  const int tile = kept[j];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int r_end = min(L, (blockIdx.y + 1) * PK_ROWS);
  for (int r = blockIdx.y * PK_ROWS + wid; r < r_end; r += PK_THREADS / 32) {
    const int dst = base + r;
    if (dst >= max_T) {
      if (lane == 0) atomicOr(&g_err_pack, RIFT_EBIT_CAPACITY);
      continue;
    }
    uint4* out = reinterpret_cast<uint4*>(packed + (size_t)dst * d);
    const int nv8 = d / 8;
    if (r < S || r >= S + b) {
      const int id = (r < S) ? sys_ids[r] : query_ids[r - S - b];
      if (id < 0 || id >= vocab) {
        if (lane == 0) atomicOr(&g_err_pack, RIFT_EBIT_BADID);
        continue;
      }
      const uint4* src = reinterpret_cast<const uint4*>(embed + (size_t)id * d);
      for (int q = lane; q < nv8; q += 32) out[q] = src[q];
    } else {
      const int k = sel[so + r - S];
      if (k < 0 || k >= n_v || tile < 0 || tile >= N) {
        if (lane == 0) atomicOr(&g_err_pack, RIFT_EBIT_BADID);
        continue;
      }
      const XT* row = X + ((size_t)tile * n_v + k) * d;
      if constexpr (sizeof(XT) == 2) {
        const uint4* src = reinterpret_cast<const uint4*>(row);
        for (int q = lane; q < nv8; q += 32) out[q] = __ldcs(src + q);
      } else {
        const float4* src = reinterpret_cast<const float4*>(row);
        for (int q = lane; q < nv8; q += 32) {
          float4 a = __ldcs(src + 2 * q), c = __ldcs(src + 2 * q + 1);
          out[q] = make_uint4(pack_bf16x2(a.x, a.y), pack_bf16x2(a.z, a.w), pack_bf16x2(c.x, c.y),
                              pack_bf16x2(c.z, c.w));
        }
      }
    }
    if (lane == 0) positions[dst] = r;
  }
}

void launch_pack(const void* X, rift_dtype xdt, int N, int n_v, int d, const int* kept,
                 const int* n_kept, const int* sel, const int* sel_off, const int* sys_ids, int S,
                 const int* query_ids, int Q, const void* embed, int vocab, void* packed, int max_T,
                 int* cu_seqlens, int* positions, int* T, cudaStream_t st) {
  seqlens_kernel<<<(N + 1 + 255) / 256, 256, 0, st>>>(n_kept, sel_off, N, S, Q, max_T, cu_seqlens, T);
  const int max_L = S + n_v + Q;
  dim3 grid(N, (max_L + PK_ROWS - 1) / PK_ROWS);
  if (xdt == RIFT_BF16)
    pack_kernel<uint16_t><<<grid, PK_THREADS, 0, st>>>(
        static_cast<const uint16_t*>(X), N, n_v, d, kept, n_kept, sel, sel_off, sys_ids, S, query_ids, Q,
        static_cast<const uint16_t*>(embed), vocab, static_cast<uint16_t*>(packed), max_T, positions);
  else
    pack_kernel<float><<<grid, PK_THREADS, 0, st>>>(
        static_cast<const float*>(X), N, n_v, d, kept, n_kept, sel, sel_off, sys_ids, S, query_ids, Q,
        static_cast<const uint16_t*>(embed), vocab, static_cast<uint16_t*>(packed), max_T, positions);
}

}  // namespace rift
