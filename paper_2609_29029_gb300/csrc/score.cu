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
// a4: G = V V^T in 64 x 64 blocks (fp32, k ascending), each block's per-row top-C written as a
// candidate list; knn_merge_kernel merges a row's lists; knn_rescore_smooth_kernel recomputes
// the C candidates in fp64, keeps the top m and smooths.
// ------------------------------------------------------------------------------------------
constexpr int KB = 64;   // rows (i) and columns (j) per block
constexpr int KNN_SPARE = 10;  // fp32 candidates kept beyond m for the fp64 rescoring
constexpr int KK = 32;   // d-chunk

// (g, j) beats (g2, j2): larger similarity first, then the lower index.
__device__ __forceinline__ bool knn_better(float g, int j, float g2, int j2) {
  return g > g2 || (g == g2 && j < j2);
}

__global__ void __launch_bounds__(256) knn_block_kernel(const float* __restrict__ V, int N, int d,
                                                        int m, float* __restrict__ cand_g,
                                                        int* __restrict__ cand_j) {
  // m here is the candidate count C kept per row and block
  __shared__ float As[KK][KB + 4];
  __shared__ float Bs[KK][KB + 4];
  __shared__ float Gs[KB][KB + 1];
  const int i0 = blockIdx.y * KB, j0 = blockIdx.x * KB;
  const int tid = threadIdx.x, ti = tid >> 4, tj = tid & 15;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < d; k0 += KK) {
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

// One warp per tile: recompute the C candidates' similarities with fp64 accumulation (the
// fp32 pass errs by ~sqrt(d) ulp for nearly parallel tiles, and fp32 cannot even separate
// similarities closer to 1 than 6e-8), keep the m best by the fp64 values (ties to the lower
// index), then s~_i = (sum over the ascending set {i} + NN(i) of s_raw) / (m + 1) with correctly
// rounded fp32 adds and divide.
__global__ void knn_rescore_smooth_kernel(const float* __restrict__ V, int d, const int* __restrict__ top_j, int N,
                                          int C, int m, const float* __restrict__ s_raw,
                                          float* __restrict__ s_tilde, int* __restrict__ nbr) {
  const int lane = threadIdx.x & 31;
  const int i = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (i >= N) return;
  double g64[RIFT_MAX_KNN];
  int jj[RIFT_MAX_KNN];
  const float* vi = V + (size_t)i * d;
  for (int r = 0; r < C; ++r) {
    const int j = top_j[(size_t)i * C + r];
    jj[r] = j;
    double acc = 0.0;
    if (j >= 0 && j < N) {
      const float* vj = V + (size_t)j * d;
      for (int k = lane; k < d; k += 32) acc = fma((double)vi[k], (double)vj[k], acc);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    g64[r] = (j >= 0 && j < N) ? acc : -INFINITY;
  }
  if (lane != 0) return;
  // top-m of the rescored candidates by (g64 desc, j asc)
  for (int a = 1; a < C; ++a) {
    double g = g64[a];
    int j = jj[a], b = a;
    while (b > 0 && (g > g64[b - 1] || (g == g64[b - 1] && j < jj[b - 1]))) {
      g64[b] = g64[b - 1]; jj[b] = jj[b - 1]; --b;
    }
    g64[b] = g; jj[b] = j;
  }
  if (nbr)
    for (int r = 0; r < m; ++r) nbr[(size_t)i * m + r] = jj[r];
  int mem[RIFT_MAX_KNN + 1];
  int n = 0;
  for (int r = 0; r < m; ++r) {
    if (jj[r] >= 0 && jj[r] < N) {
      mem[n++] = jj[r];
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
void launch_query_prep(const void* embed, int vocab, int d, const int* phrase_ids, int n_tmpl,
                       int n_phrase, const int* bg_ids, int M, float* t, float* B, cudaStream_t st) {
  query_prep_kernel<<<1, 256, 2 * d * sizeof(float), st>>>(
      static_cast<const uint16_t*>(embed), vocab, d, phrase_ids, n_tmpl, n_phrase, bg_ids, M, t, B);
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
  if (m > 0) {
    dim3 grid(L.n_jblk, L.n_jblk);
    knn_block_kernel<<<grid, 256, 0, st>>>(V, N, d, C, cg, cj);
    knn_merge_kernel<<<(N + 127) / 128, 128, 0, st>>>(cg, cj, L.n_jblk, N, C, topj);
    launched += 2;
  }
  knn_rescore_smooth_kernel<<<(N + 7) / 8, 256, 0, st>>>(V, d, topj, N, C, m, s_raw, s_tilde, nbr);
  return launched;  // kernels launched
}

}  // namespace rift
