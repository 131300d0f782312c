// Stage 1 of Rift on sm_103a: query preparation, Eq. 1 relevance of every vision token and
// every tile, and the kNN smoothing of Appendix B Step 2.
//
// HBM-bound part: token_score_kernel makes the one pass over X [N, n_v, d].  Per token it
// forms x.w and ||x||^2 (fp32), giving r = x.w / ||x|| with w = t - (1/M) sum_j B_j (Eq. 1
// with the background mean folded into one vector), and it adds the token into the tile's
// pooled sum P_i.  Several CTAs share a tile; each writes its partial P to the workspace and
// tile_finalize_kernel adds them in a fixed order.
#include <algorithm>

#include "rift_internal.h"

namespace rift {

__device__ unsigned int g_err_score;

unsigned int read_clear_err_score() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_err_score, sizeof(v));
  cudaMemcpyToSymbol(g_err_score, &z, sizeof(z));
  return v;
}

// ------------------------------------------------------------------------------------------
// a1: t = l2norm(mean_k l2norm(e_k)), e_k = mean of template k's embedding rows; B_j =
// l2norm(embed[bg_j]).  One CTA; dynamic shared memory holds 2 d floats.
// ------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) query_prep_kernel(const uint16_t* __restrict__ embed,
                                                         int vocab, int d,
                                                         const int* __restrict__ phrase_ids,
                                                         int n_tmpl, int n_phrase,
                                                         const int* __restrict__ bg_ids, int M,
                                                         float* __restrict__ t,
                                                         float* __restrict__ B) {
  extern __shared__ float qp_sm[];
  float* e = qp_sm;
  float* acc = qp_sm + d;
  __shared__ float red[32];
  for (int c = threadIdx.x; c < d; c += blockDim.x) acc[c] = 0.f;
  for (int k = 0; k < n_tmpl; ++k) {
    float ss = 0.f;
    for (int c = threadIdx.x; c < d; c += blockDim.x) {
      float s = 0.f;
      for (int q = 0; q < n_phrase; ++q) {
        int id = phrase_ids[k * n_phrase + q];
        if (id < 0 || id >= vocab) {
          atomicOr(&g_err_score, RIFT_EBIT_BADID);
          continue;
        }
        s += bf16_bits_to_float(embed[(size_t)id * d + c]);
      }
      s = s / (float)n_phrase;
      e[c] = s;
      ss += s * s;
    }
    float inv = 1.f / sqrtf(block_sum(ss, red));
    for (int c = threadIdx.x; c < d; c += blockDim.x) acc[c] += e[c] * inv;
    __syncthreads();
  }
  float ss = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) ss += acc[c] * acc[c];
  float inv = 1.f / sqrtf(block_sum(ss, red));
  for (int c = threadIdx.x; c < d; c += blockDim.x) t[c] = acc[c] * inv;
  for (int j = 0; j < M; ++j) {
    int id = bg_ids[j];
    bool ok = id >= 0 && id < vocab;
    if (!ok && threadIdx.x == 0) atomicOr(&g_err_score, RIFT_EBIT_BADID);
    float s2 = 0.f;
    for (int c = threadIdx.x; c < d; c += blockDim.x) {
      float v = ok ? bf16_bits_to_float(embed[(size_t)id * d + c]) : 0.f;
      e[c] = v;
      s2 += v * v;
    }
    float tot = block_sum(s2, red);
    float iv = tot > 0.f ? 1.f / sqrtf(tot) : 0.f;
    for (int c = threadIdx.x; c < d; c += blockDim.x) B[(size_t)j * d + c] = e[c] * iv;
    __syncthreads();
  }
}

// One caption template: rows are plain means / copies, so every column is independent.  One
// thread per column writes the unnormalised query row into t and the background rows into B;
// normalize_rows_kernel then scales each row to unit length (one CTA per row).
__global__ void query_rows_kernel(const uint16_t* __restrict__ embed, int vocab, int d,
                                  const int* __restrict__ phrase_ids, int n_phrase,
                                  const int* __restrict__ bg_ids, int M, float* __restrict__ t,
                                  float* __restrict__ B) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= d) return;
  float s = 0.f;
  for (int q = 0; q < n_phrase; ++q) {
    const int id = phrase_ids[q];
    if (id < 0 || id >= vocab) {
      atomicOr(&g_err_score, RIFT_EBIT_BADID);
      continue;
    }
    s += bf16_bits_to_float(embed[(size_t)id * d + c]);
  }
  t[c] = s / (float)n_phrase;
  for (int j = 0; j < M; ++j) {
    const int id = bg_ids[j];
    const bool ok = id >= 0 && id < vocab;
    if (!ok && c == 0) atomicOr(&g_err_score, RIFT_EBIT_BADID);
    B[(size_t)j * d + c] = ok ? bf16_bits_to_float(embed[(size_t)id * d + c]) : 0.f;
  }
}

// Row r of {t, B_0, ..., B_{M-1}} divided by its length (zero rows stay zero).
__global__ void __launch_bounds__(256) normalize_rows_kernel(float* __restrict__ t, float* __restrict__ B, int d) {
  __shared__ float red[32];
  float* row = blockIdx.x == 0 ? t : B + (size_t)(blockIdx.x - 1) * d;
  float ss = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) ss += row[c] * row[c];
  const float tot = block_sum(ss, red);
  const float inv = tot > 0.f ? 1.f / sqrtf(tot) : 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) row[c] *= inv;
}

// w = t - (1/M) sum_j B_j  (M = 0: w = t)
__global__ void fold_w_kernel(const float* __restrict__ t, const float* __restrict__ B, int M,
                              int d, float* __restrict__ w) {
  int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= d) return;
  float s = 0.f;
  for (int j = 0; j < M; ++j) s += B[(size_t)j * d + c];
  w[c] = M > 0 ? t[c] - s / (float)M : t[c];
}

// ------------------------------------------------------------------------------------------
// a2: token scores + partial pooled sums.  256 threads; thread t owns the 16-byte vectors
// t, t + 256, ... of a token row (NVEC of them).  Tokens go in groups of 8: every thread
// loads its vectors of all 8 tokens first (8 * NVEC 16-byte loads in flight), then the 16
// partial sums (x.w and x.x of each token) are reduced across the CTA.
// ------------------------------------------------------------------------------------------
constexpr int SC_THREADS = 256;
constexpr int SC_GROUP = 8;

template <typename XT>
struct VecTraits;
template <>
struct VecTraits<uint16_t> {  // bf16: 8 per 16-byte vector
  static constexpr int W = 8;
  __device__ static void unpack(const uint4& v, float* f) { unpack_bf16x8(v, f); }
};
template <>
struct VecTraits<float> {  // fp32: 4 per 16-byte vector
  static constexpr int W = 4;
  __device__ static void unpack(const uint4& v, float* f) {
    f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
  }
};

// Reduce 16 values across a warp with 16 shuffles; afterwards lanes 2q and 2q+1 both hold
// the warp total of value q.
__device__ __forceinline__ float warp_reduce16(float (&v)[16]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int s = 16, n = 16; s >= 2; s >>= 1, n >>= 1) {
    const bool up = (lane & s) != 0;
#pragma unroll
    for (int k = 0; k < n / 2; ++k) {
      float a = v[k], b = v[k + n / 2];
      float send = up ? a : b;
      float keep = up ? b : a;
      v[k] = keep + __shfl_xor_sync(0xffffffffu, send, s);
    }
  }
  return v[0] + __shfl_xor_sync(0xffffffffu, v[0], 1);
}

template <typename XT, int NVEC>
__global__ void __launch_bounds__(SC_THREADS, 2)
    token_score_kernel(const XT* __restrict__ X, int n_v, int d, int chunk_tokens, int n_chunks,
                       const float* __restrict__ w, float* __restrict__ token_scores,
                       float* __restrict__ Ppart) {
  using VT = VecTraits<XT>;
  constexpr int VW = VT::W;
  constexpr int GROUP = (NVEC <= 2) ? SC_GROUP : SC_GROUP / 2;  // raw loads: GROUP*NVEC*4 regs
  __shared__ float red[SC_THREADS / 32][16];
  __shared__ float tot[16];
  const int tile = blockIdx.x / n_chunks;
  const int chunk = blockIdx.x - tile * n_chunks;
  const int k0 = chunk * chunk_tokens;
  const int k1 = min(n_v, k0 + chunk_tokens);
  const int nvec = d / VW;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;

  float wv[NVEC][VW], P[NVEC][VW];
#pragma unroll
  for (int j = 0; j < NVEC; ++j) {
    int v = threadIdx.x + j * SC_THREADS;
#pragma unroll
    for (int e = 0; e < VW; ++e) {
      wv[j][e] = (v < nvec) ? w[v * VW + e] : 0.f;
      P[j][e] = 0.f;
    }
  }
  const XT* base = X + ((size_t)tile * n_v) * d;
  for (int g0 = k0; g0 < k1; g0 += GROUP) {
    uint4 raw[GROUP][NVEC];
#pragma unroll
    for (int g = 0; g < GROUP; ++g) {
#pragma unroll
      for (int j = 0; j < NVEC; ++j) {
        int v = threadIdx.x + j * SC_THREADS;
        if (g0 + g < k1 && v < nvec)
          raw[g][j] = __ldcs(reinterpret_cast<const uint4*>(base + (size_t)(g0 + g) * d + v * VW));
        else
          raw[g][j] = make_uint4(0u, 0u, 0u, 0u);
      }
    }
    float part[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) part[q] = 0.f;
#pragma unroll
    for (int g = 0; g < GROUP; ++g) {
      float dt = 0.f, ss = 0.f;
#pragma unroll
      for (int j = 0; j < NVEC; ++j) {
        float xv[VW];
        VT::unpack(raw[g][j], xv);
#pragma unroll
        for (int e = 0; e < VW; ++e) {
          dt = fmaf(xv[e], wv[j][e], dt);
          ss = fmaf(xv[e], xv[e], ss);
          P[j][e] += xv[e];
        }
      }
      part[g] = dt;
      part[8 + g] = ss;
    }
    float r = warp_reduce16(part);
    if ((lane & 1) == 0) red[wid][lane >> 1] = r;
    __syncthreads();
    if (threadIdx.x < 16) {
      float s = 0.f;
#pragma unroll
      for (int q = 0; q < SC_THREADS / 32; ++q) s += red[q][threadIdx.x];
      tot[threadIdx.x] = s;
    }
    __syncthreads();
    if (threadIdx.x < GROUP && g0 + threadIdx.x < k1) {
      token_scores[(size_t)tile * n_v + g0 + threadIdx.x] =
          tot[threadIdx.x] / sqrtf(tot[8 + threadIdx.x]);
    }
  }
  float* out = Ppart + (size_t)blockIdx.x * d;
#pragma unroll
  for (int j = 0; j < NVEC; ++j) {
    int v = threadIdx.x + j * SC_THREADS;
    if (v < nvec) {
#pragma unroll
      for (int e = 0; e < VW; e += 4)
        *reinterpret_cast<float4*>(out + v * VW + e) = make_float4(P[j][e], P[j][e + 1], P[j][e + 2], P[j][e + 3]);
    }
  }
}

// a3: P_i = sum of the tile's partials (fixed order), V_i = P_i / ||P_i||, s_i = V_i . w.
__global__ void __launch_bounds__(256) tile_finalize_kernel(const float* __restrict__ Ppart,
                                                            int n_chunks, int d,
                                                            const float* __restrict__ w,
                                                            float* __restrict__ V,
                                                            float* __restrict__ s_raw) {
  extern __shared__ float tf_sm[];
  __shared__ float red[32];
  const int i = blockIdx.x;
  float ss = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    float p = 0.f;
    for (int q = 0; q < n_chunks; ++q) p += Ppart[((size_t)i * n_chunks + q) * d + c];
    tf_sm[c] = p;
    ss += p * p;
  }
  float inv = 1.f / sqrtf(block_sum(ss, red));
  float dt = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    float v = tf_sm[c] * inv;
    V[(size_t)i * d + c] = v;
    dt += v * w[c];
  }
  dt = block_sum(dt, red);
  if (threadIdx.x == 0) s_raw[i] = dt;
}

// ------------------------------------------------------------------------------------------
// a4: G = V V^T in 64 x 64 blocks (fp32, k ascending, 32-term chunks).  Small scenes split K
// across CTAs and knn_row_topc_kernel picks each row's top-C from the summed slices; large ones
// keep a top-C list per block and knn_merge_kernel merges a row's lists.  Then
// knn_rescore_smooth_kernel recomputes the C candidates to ~fp64 accuracy, keeps the top m and
// smooths.
// ------------------------------------------------------------------------------------------
constexpr int KB = 64;   // rows (i) and columns (j) per block
constexpr int KNN_SPARE = 10;  // fp32 candidates kept beyond m for the fp64 rescoring
constexpr int KK = 32;   // d-chunk

// (g, j) beats (g2, j2): larger similarity first, then the lower index.
__device__ __forceinline__ bool knn_better(float g, int j, float g2, int j2) {
  return g > g2 || (g == g2 && j < j2);
}

// grid (column blocks, row blocks, K slices).  With one slice the kernel also extracts each
// row's top-C of the block (m here is C); with several it writes its partial similarities to
// Gpart[slice][i][j] for knn_row_topc_kernel.
__global__ void __launch_bounds__(256) knn_block_kernel(const float* __restrict__ V, int N, int d,
                                                        int m, float* __restrict__ cand_g,
                                                        int* __restrict__ cand_j,
                                                        float* __restrict__ Gpart) {
  __shared__ float As[KK][KB + 4];
  __shared__ float Bs[KK][KB + 4];
  __shared__ float Gs[KB][KB + 1];
  const int i0 = blockIdx.y * KB, j0 = blockIdx.x * KB;
  const int tid = threadIdx.x, ti = tid >> 4, tj = tid & 15;
  const int kslice = d / gridDim.z;
  const int kbeg = blockIdx.z * kslice, kend = kbeg + kslice;
  float acc[4][4] = {};
  for (int k0 = kbeg; k0 < kend; k0 += KK) {
    // 64 rows x 32 floats per operand = 512 float4; two per thread.
    for (int q = tid; q < KB * KK / 4; q += 256) {
      int row = q >> 3, c4 = (q & 7) * 4;
      float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b = a;
      if (i0 + row < N) a = *reinterpret_cast<const float4*>(V + (size_t)(i0 + row) * d + k0 + c4);
      if (j0 + row < N) b = *reinterpret_cast<const float4*>(V + (size_t)(j0 + row) * d + k0 + c4);
      As[c4 + 0][row] = a.x; As[c4 + 1][row] = a.y; As[c4 + 2][row] = a.z; As[c4 + 3][row] = a.w;
      Bs[c4 + 0][row] = b.x; Bs[c4 + 1][row] = b.y; Bs[c4 + 2][row] = b.z; Bs[c4 + 3][row] = b.w;
    }
    __syncthreads();
    // Each 32-term chunk is summed on its own and then added to the total: for nearly parallel
    // tiles the running sum approaches 1, and chunking cuts its rounding error about sixfold.
    float part[4][4] = {};
#pragma unroll 8
    for (int k = 0; k < KK; ++k) {
      float4 a = *reinterpret_cast<const float4*>(&As[k][ti * 4]);
      float4 b = *reinterpret_cast<const float4*>(&Bs[k][tj * 4]);
      float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) part[r][c] = fmaf(av[r], bv[c], part[r][c]);
    }
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[r][c] += part[r][c];
    __syncthreads();
  }
  if (gridDim.z > 1) {
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int i = i0 + ti * 4 + r, j = j0 + tj * 4 + c;
        if (i < N && j < N) Gpart[((size_t)blockIdx.z * N + i) * N + j] = acc[r][c];
      }
    return;
  }
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int c = 0; c < 4; ++c) Gs[ti * 4 + r][tj * 4 + c] = acc[r][c];
  __syncthreads();
  if (tid < KB && i0 + tid < N) {
    const int i = i0 + tid;
    float bg[RIFT_MAX_KNN];
    int bj[RIFT_MAX_KNN];
    for (int r = 0; r < m; ++r) { bg[r] = -INFINITY; bj[r] = 0x7fffffff; }
    for (int c = 0; c < KB; ++c) {
      const int j = j0 + c;
      if (j >= N || j == i) continue;
      float g = Gs[tid][c];
      if (!(g == g)) { atomicOr(&g_err_score, RIFT_EBIT_NONFINITE); continue; }
      if (!knn_better(g, j, bg[m - 1], bj[m - 1])) continue;
      int p = m - 1;
      while (p > 0 && knn_better(g, j, bg[p - 1], bj[p - 1])) { bg[p] = bg[p - 1]; bj[p] = bj[p - 1]; --p; }
      bg[p] = g; bj[p] = j;
    }
    const size_t o = ((size_t)i * gridDim.x + blockIdx.x) * m;
    for (int r = 0; r < m; ++r) { cand_g[o + r] = bg[r]; cand_j[o + r] = bj[r]; }
  }
}

// After a split-K Gram pass (N <= 1024): one warp per row sums the slices in slice order for
// every column and extracts the row's top-C directly (C rounds of a warp-wide argmax, larger
// similarity first, then the lower index).
constexpr int RT_WARPS = 4;
__global__ void __launch_bounds__(32 * RT_WARPS) knn_row_topc_kernel(const float* __restrict__ Gpart, int n_split,
                                                                      int N, int C, int* __restrict__ top_j) {
  __shared__ float gs[RT_WARPS][1024];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * RT_WARPS + w;
  if (i >= N) return;
  float* g = gs[w];
  for (int j = lane; j < N; j += 32) {
    float v = 0.f;
    for (int z = 0; z < n_split; ++z) v += Gpart[((size_t)z * N + i) * N + j];
    if (!(v == v)) { atomicOr(&g_err_score, RIFT_EBIT_NONFINITE); v = -INFINITY; }
    g[j] = (j == i) ? -INFINITY : v;
  }
  __syncwarp();
  for (int r = 0; r < C; ++r) {
    float bv = -INFINITY;
    int bj = 0x7fffffff;
    for (int j = lane; j < N; j += 32)
      if (knn_better(g[j], j, bv, bj)) { bv = g[j]; bj = j; }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
      const int oj = __shfl_xor_sync(0xffffffffu, bj, o);
      if (knn_better(ov, oj, bv, bj)) { bv = ov; bj = oj; }
    }
    if (lane == 0) top_j[(size_t)i * C + r] = (bv == -INFINITY) ? 0x7fffffff : bj;
    if (bj >= 0 && bj < N && (bj & 31) == lane) g[bj] = -INFINITY;
    __syncwarp();
  }
}

// Large scenes (N > 1024): the Gram matrix on the tensor cores.  Each fp32 row of V (scaled
// by 2^10, so that the low parts stay normal in fp16) is split into hi = fp16(v) and
// lo = fp16(v - hi); A = [hi | hi | lo] and B = [hi | lo | hi] along K, so one fp16 GEMM with
// K = 3 d gives hi.hi + hi.lo + lo.hi, i.e. V V^T to ~2^-22 relative (lo.lo is below that).
constexpr float KNN_SPLIT_SCALE = 1024.f;
// Rows N .. Np - 1 of B (the padding of the Gram matrix's column count to a multiple of 8) are zero.
__global__ void knn_split_kernel(const float* __restrict__ V, int N, int Np, int d, uint16_t* __restrict__ A,
                                 uint16_t* __restrict__ B) {
  const size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (size_t)Np * d) return;
  const size_t i = idx / d;
  const int k = (int)(idx % d);
  if (i >= (size_t)N) {
    uint16_t* b = B + i * 3 * d;
    b[k] = 0; b[d + k] = 0; b[2 * d + k] = 0;
    return;
  }
  const float v = V[idx] * KNN_SPLIT_SCALE;
  const __half hi = __float2half_rn(v);
  const __half lo = __float2half_rn(v - __half2float(hi));
  const uint16_t h = *reinterpret_cast<const uint16_t*>(&hi), l = *reinterpret_cast<const uint16_t*>(&lo);
  uint16_t* a = A + i * 3 * d;
  uint16_t* b = B + i * 3 * d;
  a[k] = h; a[d + k] = h; a[2 * d + k] = l;
  b[k] = h; b[d + k] = l; b[2 * d + k] = h;
}

// One warp per row of the materialised Gram matrix: each lane keeps a sorted top-C of its
// columns, then C rounds of a warp-wide argmax (larger similarity, then lower index) merge them.
__global__ void knn_gram_topc_kernel(const float* __restrict__ G, int N, int ld, int C, int* __restrict__ top_j) {
  const int lane = threadIdx.x & 31;
  const int i = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (i >= N) return;
  float bg[RIFT_MAX_KNN];
  int bj[RIFT_MAX_KNN];
  for (int r = 0; r < C; ++r) { bg[r] = -INFINITY; bj[r] = 0x7fffffff; }
  const float* row = G + (size_t)i * ld;
  for (int j = lane; j < N; j += 32) {
    if (j == i) continue;
    const float g = row[j];
    if (!(g == g)) { atomicOr(&g_err_score, RIFT_EBIT_NONFINITE); continue; }
    if (!knn_better(g, j, bg[C - 1], bj[C - 1])) continue;
    int p = C - 1;
    while (p > 0 && knn_better(g, j, bg[p - 1], bj[p - 1])) { bg[p] = bg[p - 1]; bj[p] = bj[p - 1]; --p; }
    bg[p] = g; bj[p] = j;
  }
  int head = 0;
  for (int r = 0; r < C; ++r) {
    float cg = head < C ? bg[head] : -INFINITY;
    int cj = head < C ? bj[head] : 0x7fffffff;
    int cl = lane;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float og = __shfl_xor_sync(0xffffffffu, cg, o);
      const int oj = __shfl_xor_sync(0xffffffffu, cj, o);
      const int ol = __shfl_xor_sync(0xffffffffu, cl, o);
      if (knn_better(og, oj, cg, cj)) { cg = og; cj = oj; cl = ol; }
    }
    if (cl == lane) ++head;
    if (lane == 0) top_j[(size_t)i * C + r] = (cg == -INFINITY) ? 0x7fffffff : cj;
  }
}

// One thread per tile: merge the blocks' candidate lists into the row's top-C by fp32
// similarity (C = m + a few spares).
__global__ void knn_merge_kernel(const float* __restrict__ cand_g, const int* __restrict__ cand_j, int n_lists,
                                 int N, int C, int* __restrict__ top_j) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= N) return;
  float bg[RIFT_MAX_KNN];
  int bj[RIFT_MAX_KNN];
  for (int r = 0; r < C; ++r) { bg[r] = -INFINITY; bj[r] = 0x7fffffff; }
  for (int l = 0; l < n_lists; ++l) {
    const size_t o = ((size_t)i * n_lists + l) * C;
    for (int r = 0; r < C; ++r) {
      float g = cand_g[o + r];
      int j = cand_j[o + r];
      if (!knn_better(g, j, bg[C - 1], bj[C - 1])) break;  // lists are sorted
      int p = C - 1;
      while (p > 0 && knn_better(g, j, bg[p - 1], bj[p - 1])) { bg[p] = bg[p - 1]; bj[p] = bj[p - 1]; --p; }
      bg[p] = g; bj[p] = j;
    }
  }
  for (int r = 0; r < C; ++r) top_j[(size_t)i * C + r] = bj[r];
}

// One CTA per tile, one warp per candidate: recompute the C candidates' similarities to ~fp64
// accuracy (the fp32 pass errs by ~sqrt(d) ulp for nearly parallel tiles, and fp32 cannot even
// separate similarities closer to 1 than 6e-8), keep the m best by those values (ties to the
// lower index), then s~_i = (sum over the ascending set {i} + NN(i) of s_raw) / (m + 1) with
// correctly rounded fp32 adds and divide.
__global__ void __launch_bounds__(32 * RIFT_MAX_KNN) knn_rescore_smooth_kernel(
    const float* __restrict__ V, int d, const int* __restrict__ top_j, int N, int C, int m,
    const float* __restrict__ s_raw, float* __restrict__ s_tilde, int* __restrict__ nbr) {
  __shared__ double g64[RIFT_MAX_KNN];
  __shared__ int jj[RIFT_MAX_KNN];
  const int i = blockIdx.x;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (w < C) {
    const int j = top_j[(size_t)i * C + w];
    // Each lane keeps its partial sum as an unevaluated pair hi + lo of floats: the product of
    // two floats is split exactly with an FMA (Dekker's TwoProduct as rewritten by Ogita, Rump
    // and Oishi) and added with Knuth's TwoSum, so the lane sum is good to ~2^-44 relative.
    float hi = 0.f, lo = 0.f;
    if (j >= 0 && j < N) {
      const float4* vi = reinterpret_cast<const float4*>(V + (size_t)i * d);
      const float4* vj = reinterpret_cast<const float4*>(V + (size_t)j * d);
      for (int k = lane; k < d / 4; k += 32) {
        const float4 a4 = vi[k], b4 = vj[k];
        const float av[4] = {a4.x, a4.y, a4.z, a4.w}, bv[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float p = __fmul_rn(av[e], bv[e]);
          const float pe = fmaf(av[e], bv[e], -p);
          const float s = __fadd_rn(hi, p);
          const float bb = __fsub_rn(s, hi);
          const float er = __fadd_rn(__fsub_rn(hi, __fsub_rn(s, bb)), __fsub_rn(p, bb));
          hi = s;
          lo = __fadd_rn(lo, __fadd_rn(er, pe));
        }
      }
    }
    double acc = (double)hi + (double)lo;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) {
      g64[w] = (j >= 0 && j < N) ? acc : -INFINITY;
      jj[w] = j;
    }
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  double gl[RIFT_MAX_KNN];
  int jl[RIFT_MAX_KNN];
  for (int a = 0; a < C; ++a) {  // insertion into (g desc, j asc) order
    double g = g64[a];
    int j = jj[a], b = a;
    while (b > 0 && (g > gl[b - 1] || (g == gl[b - 1] && j < jl[b - 1]))) { gl[b] = gl[b - 1]; jl[b] = jl[b - 1]; --b; }
    gl[b] = g; jl[b] = j;
  }
  if (nbr)
    for (int r = 0; r < m; ++r) nbr[(size_t)i * m + r] = jl[r];
  int mem[RIFT_MAX_KNN + 1];
  int n = 0;
  for (int r = 0; r < m; ++r) {
    if (jl[r] >= 0 && jl[r] < N) {
      mem[n++] = jl[r];
    } else {  // fewer than m finite similarities (a NaN row): reported, never indexed
      atomicOr(&g_err_score, RIFT_EBIT_NONFINITE);
    }
  }
  mem[n++] = i;
  for (int a = 1; a < n; ++a) {
    int v = mem[a], b = a;
    while (b > 0 && mem[b - 1] > v) { mem[b] = mem[b - 1]; --b; }
    mem[b] = v;
  }
  float acc = 0.f;
  for (int a = 0; a < n; ++a) acc = __fadd_rn(acc, s_raw[mem[a]]);
  s_tilde[i] = __fdiv_rn(acc, (float)(m + 1));
}

// ------------------------------------------------------------------------------------------
// Launchers
// ------------------------------------------------------------------------------------------
int launch_query_prep(const void* embed, int vocab, int d, const int* phrase_ids, int n_tmpl,
                      int n_phrase, const int* bg_ids, int M, float* t, float* B, cudaStream_t st) {
  if (n_tmpl == 1) {
    query_rows_kernel<<<(d + 255) / 256, 256, 0, st>>>(static_cast<const uint16_t*>(embed), vocab, d, phrase_ids,
                                                       n_phrase, bg_ids, M, t, B);
    normalize_rows_kernel<<<1 + M, 256, 0, st>>>(t, B, d);
    return 2;
  }
  // two fp32 rows of d in shared memory: 64 KB at the widest d (8192), past the 48 KB default
  static std::atomic<unsigned long long> smem_raised{0};
  if (raise_smem_limit(smem_raised, query_prep_kernel, (int)(2 * 8192 * sizeof(float))) != cudaSuccess)
    return 0;  // the launch check of the caller reports the failure
  query_prep_kernel<<<1, 256, 2 * d * sizeof(float), st>>>(
      static_cast<const uint16_t*>(embed), vocab, d, phrase_ids, n_tmpl, n_phrase, bg_ids, M, t, B);
  return 1;
}

ScoreLayout score_layout(int N, int n_v, int d, int M) {
  ScoreLayout L{};
  L.chunk_tokens = 96;  // 6 CTAs per 576-token tile
  L.n_chunks = (n_v + L.chunk_tokens - 1) / L.chunk_tokens;
  L.n_jblk = (N + KB - 1) / KB;
  size_t off = 0;
  auto take = [&](size_t bytes) { size_t o = off; off += (bytes + 255) & ~size_t(255); return o; };
  L.w_off = take(sizeof(float) * d);
  L.ppart_off = take(sizeof(float) * (size_t)N * L.n_chunks * d);
  L.V_off = take(sizeof(float) * (size_t)N * d);
  L.cand_g_off = take(sizeof(float) * (size_t)N * L.n_jblk * RIFT_MAX_KNN);
  L.cand_j_off = take(sizeof(int) * (size_t)N * L.n_jblk * RIFT_MAX_KNN);
  L.top_off = take(sizeof(int) * (size_t)N * RIFT_MAX_KNN);
  // K slices of the Gram pass: enough CTAs for small scenes; each slice a whole number of
  // 32-column chunks of d.
  int split = N <= 512 ? 8 : (N <= 1024 ? 4 : 1);
  while (split > 1 && (d / KK) % split != 0) split >>= 1;
  L.n_split = split;
  L.gpart_off = take(L.n_split > 1 ? sizeof(float) * (size_t)L.n_split * N * N : 0);
  L.tensor_gram = N > 1024;
  const size_t Np = ((size_t)N + 7) & ~size_t(7);
  L.split_a_off = take(L.tensor_gram ? sizeof(uint16_t) * (size_t)N * 3 * d : 0);
  L.split_b_off = take(L.tensor_gram ? sizeof(uint16_t) * Np * 3 * d : 0);
  L.gram_off = take(L.tensor_gram ? sizeof(float) * (size_t)N * Np : 0);
  L.total = off;
  (void)M;
  return L;
}

template <typename XT, int NVEC>
static void launch_tokens(const void* X, int N, int n_v, int d, const ScoreLayout& L, const float* w,
                          float* token_scores, float* Ppart, cudaStream_t st) {
  token_score_kernel<XT, NVEC><<<N * L.n_chunks, SC_THREADS, 0, st>>>(
      static_cast<const XT*>(X), n_v, d, L.chunk_tokens, L.n_chunks, w, token_scores, Ppart);
}

int launch_score(const void* X, rift_dtype xdt, int N, int n_v, int d, const float* t, const float* B,
                 int M, int m, float* token_scores, float* s_raw, float* s_tilde, int* nbr, char* ws,
                 cudaStream_t st) {
  ScoreLayout L = score_layout(N, n_v, d, M);
  float* w = reinterpret_cast<float*>(ws + L.w_off);
  float* Ppart = reinterpret_cast<float*>(ws + L.ppart_off);
  float* V = reinterpret_cast<float*>(ws + L.V_off);
  float* cg = reinterpret_cast<float*>(ws + L.cand_g_off);
  int* cj = reinterpret_cast<int*>(ws + L.cand_j_off);
  fold_w_kernel<<<(d + 255) / 256, 256, 0, st>>>(t, B, M, d, w);
  const int vw = (xdt == RIFT_BF16) ? 8 : 4;
  const int nvec_per_thread = (d / vw + SC_THREADS - 1) / SC_THREADS;
  if (xdt == RIFT_BF16) {
    if (nvec_per_thread <= 1) launch_tokens<uint16_t, 1>(X, N, n_v, d, L, w, token_scores, Ppart, st);
    else if (nvec_per_thread <= 2) launch_tokens<uint16_t, 2>(X, N, n_v, d, L, w, token_scores, Ppart, st);
    else launch_tokens<uint16_t, 4>(X, N, n_v, d, L, w, token_scores, Ppart, st);
  } else {
    if (nvec_per_thread <= 1) launch_tokens<float, 1>(X, N, n_v, d, L, w, token_scores, Ppart, st);
    else if (nvec_per_thread <= 2) launch_tokens<float, 2>(X, N, n_v, d, L, w, token_scores, Ppart, st);
    else launch_tokens<float, 4>(X, N, n_v, d, L, w, token_scores, Ppart, st);
  }
  tile_finalize_kernel<<<N, 256, d * sizeof(float), st>>>(Ppart, L.n_chunks, d, w, V, s_raw);
  int* topj = reinterpret_cast<int*>(ws + L.top_off);
  // candidates per row: m plus spares for the fp64 rescoring, at most the N - 1 other tiles
  const int C = m > 0 ? std::min(std::min(m + KNN_SPARE, RIFT_MAX_KNN), N - 1) : 0;
  int launched = 4;
  if (m > 0 && L.tensor_gram) {
    uint16_t* A16 = reinterpret_cast<uint16_t*>(ws + L.split_a_off);
    uint16_t* B16 = reinterpret_cast<uint16_t*>(ws + L.split_b_off);
    float* G = reinterpret_cast<float*>(ws + L.gram_off);
    const int Np = (N + 7) & ~7;
    const size_t n = (size_t)Np * d;
    knn_split_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(V, N, Np, d, A16, B16);
    EpiParams ep;
    ep.out_scale = 1.f / (KNN_SPLIT_SCALE * KNN_SPLIT_SCALE);
    if (launch_gemm_tc(A16, B16, N, Np, 3 * d, EPI_STORE_F32, G, ep, st)) return -1;
    knn_gram_topc_kernel<<<(N + 3) / 4, 128, 0, st>>>(G, N, Np, C, topj);
    launched += 3;
  } else if (m > 0) {
    float* gpart = reinterpret_cast<float*>(ws + L.gpart_off);
    dim3 grid(L.n_jblk, L.n_jblk, L.n_split);
    knn_block_kernel<<<grid, 256, 0, st>>>(V, N, d, C, cg, cj, gpart);
    if (L.n_split > 1)
      knn_row_topc_kernel<<<(N + RT_WARPS - 1) / RT_WARPS, 32 * RT_WARPS, 0, st>>>(gpart, L.n_split, N, C, topj);
    else
      knn_merge_kernel<<<(N + 127) / 128, 128, 0, st>>>(cg, cj, L.n_jblk, N, C, topj);
    launched += 2;
  }
  knn_rescore_smooth_kernel<<<N, 32 * RIFT_MAX_KNN, 0, st>>>(V, d, topj, N, C, m, s_raw, s_tilde, nbr);
  return launched;  // kernels launched
}

}  // namespace rift
