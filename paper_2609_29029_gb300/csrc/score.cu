// Stage 1 of Rift on sm_103a: query preparation, Eq. 1 relevance of every vision token and
// every tile, and the kNN smoothing of Appendix B Step 2.
//
// HBM-bound part: token_score_kernel makes the one pass over X [N, n_v, d].  Per token it
// forms x.w and ||x||^2 (fp32), giving r = x.w / ||x|| with w = t - (1/M) sum_j B_j (Eq. 1
// with the background mean folded into one vector), and it adds the token into the tile's
// pooled sum P_i.  Several CTAs share a tile; each writes its partial P to the workspace, and
// the one that writes the tile's last partial adds them in a fixed order and finalises the tile.
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

// One caption template: CTA 0 forms t = l2norm(mean_q embed[phrase_ids[q]]), CTA 1 + j forms
// B_j = l2norm(embed[bg_ids[j]]); a thread owns 4 columns (VPT groups of them at d > 4096) and
// issues the loads of all its rows before summing them, so a CTA waits on one round of loads.
constexpr int QR_THREADS = 1024;
__global__ void __launch_bounds__(QR_THREADS) query_rows_kernel(const uint16_t* __restrict__ embed, int vocab, int d,
                                                                const int* __restrict__ phrase_ids, int n_phrase,
                                                                const int* __restrict__ bg_ids, int M,
                                                                float* __restrict__ t, float* __restrict__ B) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[32];
  const bool is_t = blockIdx.x == 0;
  float* out = is_t ? t : B + (size_t)(blockIdx.x - 1) * d;
  const int n_ids = is_t ? n_phrase : 1;
  const int* ids = is_t ? phrase_ids : bg_ids + (blockIdx.x - 1);
  const int nv = d / 4;
  float4 acc[2];
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const int c = threadIdx.x + k * QR_THREADS;
    acc[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (c >= nv) continue;
    for (int q0 = 0; q0 < n_ids; q0 += 8) {
      uint2 raw[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {  // up to eight rows' loads in flight
        const int q = q0 + u;
        const int id = q < n_ids ? ids[q] : -1;
        const bool ok = id >= 0 && id < vocab;
        if (q < n_ids && !ok && c == 0) atomicOr(&g_err_score, RIFT_EBIT_BADID);
        raw[u] = ok ? reinterpret_cast<const uint2*>(embed + (size_t)id * d)[c] : make_uint2(0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {  // ascending q, as the sum of the ids' rows is defined
        if (q0 + u >= n_ids) break;
        acc[k].x += __uint_as_float(raw[u].x << 16);
        acc[k].y += __uint_as_float(raw[u].x & 0xffff0000u);
        acc[k].z += __uint_as_float(raw[u].y << 16);
        acc[k].w += __uint_as_float(raw[u].y & 0xffff0000u);
      }
    }
    if (is_t) {
      const float inv_n = 1.f / (float)n_phrase;
      acc[k] = make_float4(acc[k].x * inv_n, acc[k].y * inv_n, acc[k].z * inv_n, acc[k].w * inv_n);
    }
    ss += acc[k].x * acc[k].x + acc[k].y * acc[k].y + acc[k].z * acc[k].z + acc[k].w * acc[k].w;
  }
  const float tot = block_sum(ss, red);
  const float inv = tot > 0.f ? 1.f / sqrtf(tot) : 0.f;
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const int c = threadIdx.x + k * QR_THREADS;
    if (c < nv)
      reinterpret_cast<float4*>(out)[c] = make_float4(acc[k].x * inv, acc[k].y * inv, acc[k].z * inv, acc[k].w * inv);
  }
}

// w = t - (1/M) sum_j B_j  (M = 0: w = t).  Also zeroes the token pass's per-tile arrival
// counters cnt[0 .. N) (every finalising CTA leaves its counter zeroed again).
__global__ void fold_w_kernel(const float* __restrict__ t, const float* __restrict__ B, int M,
                              int d, float* __restrict__ w, unsigned int* __restrict__ cnt, int N) {
  pdl_trigger();
  pdl_wait();
  int c = blockIdx.x * blockDim.x + threadIdx.x;
  for (int k = c; k < N; k += gridDim.x * blockDim.x) cnt[k] = 0u;
  if (c >= d) return;
  float s = 0.f;
  for (int j = 0; j < M; ++j) s += B[(size_t)j * d + c];
  w[c] = M > 0 ? t[c] - s / (float)M : t[c];
}

// The fp16 hi/lo split of the Gram operands (see knn_split_kernel): rows of V scaled by 2^10 so
// that the low parts stay normal in fp16.
constexpr float KNN_SPLIT_SCALE = 1024.f;

// a3 for tile i, by one CTA of any size (MAXC >= the float4 columns a thread holds): P_i = sum of
// the tile's n_chunks partials (in chunk order), V_i = P_i / ||P_i||, s_i = V_i . w.  A thread
// takes the float4 columns threadIdx.x + k blockDim.x, so that its partial loads all issue
// together; the partials are read through L2 (other CTAs wrote them).  With S16 (the whole scene's
// Gram operand, Np rows) it also writes tile i's split row, as knn_split_kernel would from V, and
// its share of the zero padding rows.
template <int MAXC>
__device__ __forceinline__ void finalize_tile(int i, const float* __restrict__ Ppart, int n_chunks, int d,
                                              const float* __restrict__ w, float* __restrict__ V,
                                              float* __restrict__ s_raw, uint16_t* __restrict__ S16, int N, int Np,
                                              float* red) {
  const int nv = d / 4;
  float4 p[MAXC];
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < MAXC; ++k) {
    const int c = threadIdx.x + k * blockDim.x;
    p[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (c < nv) {
      const float4* src = reinterpret_cast<const float4*>(Ppart + (size_t)i * n_chunks * d) + c;
      for (int q = 0; q < n_chunks; ++q) {
        const float4 v = __ldcg(src + (size_t)q * nv);
        p[k].x += v.x;
        p[k].y += v.y;
        p[k].z += v.z;
        p[k].w += v.w;
      }
      ss += p[k].x * p[k].x + p[k].y * p[k].y + p[k].z * p[k].z + p[k].w * p[k].w;
    }
  }
  const float inv = 1.f / sqrtf(block_sum(ss, red));
  float dt = 0.f;
#pragma unroll
  for (int k = 0; k < MAXC; ++k) {
    const int c = threadIdx.x + k * blockDim.x;
    if (c < nv) {
      const float4 v = make_float4(p[k].x * inv, p[k].y * inv, p[k].z * inv, p[k].w * inv);
      reinterpret_cast<float4*>(V + (size_t)i * d)[c] = v;
      if (S16) {
        const float a[4] = {v.x * KNN_SPLIT_SCALE, v.y * KNN_SPLIT_SCALE, v.z * KNN_SPLIT_SCALE,
                            v.w * KNN_SPLIT_SCALE};
        uint32_t h[2], l[2];
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          const __half h0 = __float2half_rn(a[2 * q]), h1 = __float2half_rn(a[2 * q + 1]);
          h[q] = pack_half2(__half2float(h0), __half2float(h1));
          l[q] = pack_half2(a[2 * q] - __half2float(h0), a[2 * q + 1] - __half2float(h1));
        }
        uint2* row = reinterpret_cast<uint2*>(S16 + (size_t)i * 2 * d) + c;  // [hi | lo]
        row[0] = make_uint2(h[0], h[1]);
        row[d / 4] = make_uint2(l[0], l[1]);
      }
      const float4 wc = reinterpret_cast<const float4*>(w)[c];
      dt += v.x * wc.x + v.y * wc.y + v.z * wc.z + v.w * wc.w;
    }
  }
  dt = block_sum(dt, red);
  if (threadIdx.x == 0) s_raw[i] = dt;
  if (S16)  // the padding rows N .. Np - 1 are zero: tile i takes rows N + i, N + i + N, ...
    for (int r = N + i; r < Np; r += N)
      for (int c = threadIdx.x; c < 2 * d / 8; c += blockDim.x)
        reinterpret_cast<uint4*>(S16 + (size_t)r * 2 * d)[c] = make_uint4(0, 0, 0, 0);
}

// a3 after the token pass (scenes below the in-pass size): one CTA per tile of the token pass's
// width, SC_THREADS, so that the finalisation's sums (and V, bit for bit) are the same whichever
// kernel runs it and whatever the scene's or shard's size; each thread has four float4 columns of
// loads in flight (d = 4096).
__global__ void __launch_bounds__(256) tile_finalize_kernel(const float* __restrict__ Ppart, int n_chunks, int d,
                                                           const float* __restrict__ w, float* __restrict__ V,
                                                           float* __restrict__ s_raw, uint16_t* __restrict__ S16,
                                                           int N, int Np) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[32];
  finalize_tile<8192 / 4 / 256>(blockIdx.x, Ppart, n_chunks, d, w, V, s_raw, S16, N, Np, red);
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
                       float* __restrict__ Ppart, unsigned int* __restrict__ cnt, float* __restrict__ V,
                       float* __restrict__ s_raw, uint16_t* __restrict__ S16, int N, int Np) {
  pdl_trigger();
  pdl_wait();
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
  // With cnt (large scenes), the CTA that stores the tile's last partial finalises the tile (the
  // classic last-block reduction: every thread's stores are fenced before the count; the
  // finalising CTA fences before it reads the other partials), so no finalisation kernel follows
  // the pass.  Without it, tile_finalize_kernel does the same after the pass.
  if (!cnt) return;
  __shared__ unsigned int last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const bool l = atomicAdd(cnt + tile, 1u) == (unsigned)n_chunks - 1u;
    if (l) atomicExch(cnt + tile, 0u);
    last = l;
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  finalize_tile<(8192 / 4 + SC_THREADS - 1) / SC_THREADS>(tile, Ppart, n_chunks, d, w, V, s_raw, S16, N, Np,
                                                          &red[0][0]);
}

// ------------------------------------------------------------------------------------------
// a4: each row's C candidate neighbours from an approximate Gram matrix G = V V^T on the tensor
// cores, then knn_rescore_smooth_kernel recomputes the C candidates to ~fp64 accuracy, keeps the
// top m and smooths.
// ------------------------------------------------------------------------------------------
constexpr int KNN_SPARE = 10;  // candidates kept beyond m for the fp64 rescoring

// (g, j) beats (g2, j2): larger similarity first, then the lower index.
__device__ __forceinline__ bool knn_better(float g, int j, float g2, int j2) {
  return g > g2 || (g == g2 && j < j2);
}

// The Gram matrix on the tensor cores.  Each fp32 row of V (scaled by 2^10, so that the low parts
// stay normal in fp16) is split into hi = fp16(v) and lo = fp16(v - hi), stored once as the row
// [hi | lo] of S (2 d fp16).  The product reads S twice through a K-block remap: A = [hi | hi | lo]
// and B = [hi | lo | hi] along K, so one fp16 GEMM with K = 3 d gives hi.hi + hi.lo + lo.hi, i.e.
// V V^T to ~2^-22 relative (lo.lo is below that).  S holds every tile; A is its rows row0 ..
// row1 - 1.  Rows N .. Np - 1 of S (the padding of the Gram matrix's column count to a multiple of
// 8) are zero.  A thread handles 8 consecutive elements of a row (two float4 loads, a 16-byte
// store into each half of the row).
__global__ void knn_split_kernel(const float* __restrict__ V, int N, int Np, int d, uint16_t* __restrict__ S) {
  pdl_trigger();
  pdl_wait();
  const int n8 = d / 8;
  const size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (size_t)Np * n8) return;
  const size_t i = idx / n8;
  const int k = (int)(idx % n8) * 8;
  uint4* row = reinterpret_cast<uint4*>(S + i * 2 * d + k);
  if (i >= (size_t)N) {
    const uint4 z = make_uint4(0, 0, 0, 0);
    row[0] = z;
    row[d / 8] = z;
    return;
  }
  const float4 v0 = reinterpret_cast<const float4*>(V + i * d + k)[0];
  const float4 v1 = reinterpret_cast<const float4*>(V + i * d + k)[1];
  const float v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
  uint32_t h[4], l[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float a0 = v[2 * q] * KNN_SPLIT_SCALE, a1 = v[2 * q + 1] * KNN_SPLIT_SCALE;
    const __half h0 = __float2half_rn(a0), h1 = __float2half_rn(a1);
    h[q] = pack_half2(__half2float(h0), __half2float(h1));
    l[q] = pack_half2(a0 - __half2float(h0), a1 - __half2float(h1));
  }
  row[0] = make_uint4(h[0], h[1], h[2], h[3]);
  row[d / 8] = make_uint4(l[0], l[1], l[2], l[3]);
}

// One warp per row of the materialised Gram matrix: the row's 16 best columns (larger
// similarity, then lower index) are kept sorted across lanes 0..15, one entry per lane.  The row
// is read 32 columns at a time; a ballot picks the columns that beat the current 16th entry, and
// each of them (in ascending column order) is inserted at the position the entries above it
// give, the entries below moving down a lane.  Row il of G is tile row0 + il.
__global__ void knn_gram_topc_kernel(const float* __restrict__ G, int N, int ld, int row0, int n_rows, int C,
                                     int* __restrict__ top_j) {
  pdl_trigger();
  pdl_wait();
  constexpr int K = RIFT_MAX_KNN;  // list length (C <= K)
  const int lane = threadIdx.x & 31;
  const int il = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (il >= n_rows) return;
  const int i = row0 + il;
  float lg = -INFINITY;  // this lane's entry (lanes >= K stay empty)
  int lj = 0x7fffffff;
  float tg = -INFINITY;  // the 16th entry: what a column must beat
  int tj = 0x7fffffff;
  const float* row = G + (size_t)il * ld;
  bool bad = false;
  // 16 loads in flight per lane (512 columns per step): a step is bounded by the loads' latency,
  // not by the insertions, so fewer and wider steps finish a row sooner
  constexpr int NL = 16;
  for (int j0 = 0; j0 < N; j0 += 32 * NL) {
    float gv[NL];
#pragma unroll
    for (int q = 0; q < NL; ++q) {
      const int j = j0 + 32 * q + lane;
      gv[q] = j < N ? row[j] : -INFINITY;
    }
#pragma unroll
    for (int q = 0; q < NL; ++q) {
      const int j = j0 + 32 * q + lane;
      float g = gv[q];
      if (!(g == g)) {
        bad = true;
        g = -INFINITY;
      }
      if (j >= N || j == i) g = -INFINITY;
      unsigned mask = __ballot_sync(0xffffffffu, g != -INFINITY && knn_better(g, j, tg, tj));
      while (mask) {
        const int src = __ffs(mask) - 1;
        mask &= mask - 1;
        const float cg = __shfl_sync(0xffffffffu, g, src);
        const int cj = __shfl_sync(0xffffffffu, j, src);
        if (!knn_better(cg, cj, tg, tj)) continue;  // the threshold rose meanwhile (uniform)
        const int pos = __popc(__ballot_sync(0xffffffffu, lane < K && knn_better(lg, lj, cg, cj)));
        const float ug = __shfl_up_sync(0xffffffffu, lg, 1);
        const int uj = __shfl_up_sync(0xffffffffu, lj, 1);
        if (lane > pos && lane < K) {
          lg = ug;
          lj = uj;
        }
        if (lane == pos) {
          lg = cg;
          lj = cj;
        }
        tg = __shfl_sync(0xffffffffu, lg, K - 1);
        tj = __shfl_sync(0xffffffffu, lj, K - 1);
      }
    }
  }
  if (__any_sync(0xffffffffu, bad) && lane == 0) atomicOr(&g_err_score, RIFT_EBIT_NONFINITE);
  if (lane < C) top_j[(size_t)il * C + lane] = (lg == -INFINITY) ? 0x7fffffff : lj;
}

// One CTA per tile, one warp per candidate: recompute the C candidates' similarities to ~fp64
// accuracy (the fp32 pass errs by ~sqrt(d) ulp for nearly parallel tiles, and fp32 cannot even
// separate similarities closer to 1 than 6e-8), keep the m best by those values (ties to the
// lower index), then s~_i = (sum over the ascending set {i} + NN(i) of s_raw) / (m + 1) with
// correctly rounded fp32 adds and divide.
// CTA il smooths tile i = row0 + il and writes s_tilde[il], nbr[il].
__global__ void __launch_bounds__(32 * RIFT_MAX_KNN) knn_rescore_smooth_kernel(
    const float* __restrict__ V, int d, const int* __restrict__ top_j, int N, int row0, int C, int m,
    const float* __restrict__ s_raw, float* __restrict__ s_tilde, int* __restrict__ nbr) {
  pdl_trigger();
  pdl_wait();
  __shared__ double g64[RIFT_MAX_KNN];
  __shared__ int jj[RIFT_MAX_KNN];
  const int il = blockIdx.x, i = row0 + il;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (w < C) {
    const int j = top_j[(size_t)il * C + w];
    // Each lane keeps its partial sum as an unevaluated pair hi + lo of floats: the product of
    // two floats is split exactly with an FMA (Dekker's TwoProduct as rewritten by Ogita, Rump
    // and Oishi) and added with Knuth's TwoSum, so the lane sum is good to ~2^-44 relative.
    // V_i is read by all the CTA's warps (L1 serves all but the first).  The kernel moves 16 rows
    // of V per tile from L2: its time follows those bytes, not the length of this chain (four
    // independent chains with loads ahead measured slower, at fewer resident CTAs).
    float hi = 0.f, lo = 0.f;
    if (j >= 0 && j < N) {
      const float4* vi = reinterpret_cast<const float4*>(V + (size_t)i * d);
      const float4* vj = reinterpret_cast<const float4*>(V + (size_t)j * d);
#pragma unroll 4
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
    for (int r = 0; r < m; ++r) nbr[(size_t)il * m + r] = jl[r];
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
  s_tilde[il] = __fdiv_rn(acc, (float)(m + 1));
}

// ------------------------------------------------------------------------------------------
// Launchers
// ------------------------------------------------------------------------------------------
int launch_query_prep(const void* embed, int vocab, int d, const int* phrase_ids, int n_tmpl,
                      int n_phrase, const int* bg_ids, int M, float* t, float* B, cudaStream_t st) {
  if (n_tmpl == 1) {
    launch_ex(query_rows_kernel, dim3(1 + M), dim3(std::min(QR_THREADS, (d / 4 + 31) / 32 * 32)), 0, st, true,
              static_cast<const uint16_t*>(embed), vocab, d, phrase_ids, n_phrase, bg_ids, M, t, B);
    return 1;
  }
  // two fp32 rows of d in shared memory: 64 KB at the widest d (8192), past the 48 KB default
  static std::atomic<unsigned long long> smem_raised{0};
  if (raise_smem_limit(smem_raised, query_prep_kernel, (int)(2 * 8192 * sizeof(float))) != cudaSuccess)
    return 0;  // the launch check of the caller reports the failure
  query_prep_kernel<<<1, 256, 2 * d * sizeof(float), st>>>(
      static_cast<const uint16_t*>(embed), vocab, d, phrase_ids, n_tmpl, n_phrase, bg_ids, M, t, B);
  return 1;
}

// Scratch of the kNN smoothing of rows row0 .. row0 + n_rows - 1 against all N tiles: the split
// rows of every tile, the Gram rows, split-K partials when the product has fewer tiles than SMs (at most 16
// slices within 16 MB), the candidate lists.
SmoothLayout smooth_layout(int N, int n_rows, int d) {
  SmoothLayout L{};
  size_t off = 0;
  auto take = [&](size_t bytes) { size_t o = off; off += (bytes + 255) & ~size_t(255); return o; };
  const size_t Np = ((size_t)N + 7) & ~size_t(7);
  L.top_off = take(sizeof(int) * (size_t)n_rows * RIFT_MAX_KNN);
  L.gram_off = take(sizeof(float) * (size_t)n_rows * Np);
  const size_t slice = sizeof(float) * (size_t)n_rows * Np;
  size_t part = ((size_t)16 << 20) / slice;
  part = part > 16 ? 16 : part;
  L.splitk_bytes = part >= 2 ? part * slice : 0;
  L.splitk_off = take(L.splitk_bytes);
  L.split_off = take(sizeof(uint16_t) * Np * 2 * d);  // the split rows last
  L.total = off;
  return L;
}

// Scratch of the token pass over N tiles: w, the per-tile arrival counters and the partial pooled
// sums.
ShardLayout shard_layout(int N, int n_v, int d) {
  ShardLayout L{};
  L.chunk_tokens = 192;  // 3 CTAs per 576-token tile
  L.n_chunks = (n_v + L.chunk_tokens - 1) / L.chunk_tokens;
  size_t off = 0;
  auto take = [&](size_t bytes) { size_t o = off; off += (bytes + 255) & ~size_t(255); return o; };
  L.w_off = take(sizeof(float) * d);
  L.cnt_off = take(sizeof(unsigned int) * (size_t)N);
  L.ppart_off = take(sizeof(float) * (size_t)N * L.n_chunks * d);
  L.total = off;
  return L;
}

ScoreLayout score_layout(int N, int n_v, int d, int M) {
  (void)M;
  ScoreLayout L{};
  L.T = shard_layout(N, n_v, d);
  L.S = smooth_layout(N, N, d);
  // V first; after it the token pass's scratch (w, counters, partial pooled sums).  The
  // smoothing's scratch reuses the token scratch once the pass is over (the smoothing runs after it
  // on the stream), except for its split rows, which the pass's finalising CTAs write while other
  // tiles' partial sums are still in use: they start past the token scratch.
  L.V_off = 0;
  L.tokens_off = (sizeof(float) * (size_t)N * d + 255) & ~size_t(255);
  L.smooth_off = L.tokens_off + (L.T.total > L.S.split_off ? L.T.total - L.S.split_off : 0);
  L.total = L.smooth_off + L.S.total;
  return L;
}

template <typename XT, int NVEC>
static void launch_tokens(const void* X, int N, int n_v, int d, const ShardLayout& L, const float* w,
                          float* token_scores, float* Ppart, unsigned int* cnt, float* V, float* s_raw,
                          uint16_t* S16, cudaStream_t st) {
  launch_ex(token_score_kernel<XT, NVEC>, dim3(N * L.n_chunks), dim3(SC_THREADS), 0, st, true,
            static_cast<const XT*>(X), n_v, d, L.chunk_tokens, L.n_chunks, (const float*)w, token_scores, Ppart,
            cnt, V, s_raw, S16, N, (N + 7) & ~7);
}

int launch_score_tokens(const void* X, rift_dtype xdt, int N, int n_v, int d, const float* t, const float* B,
                        int M, float* token_scores, float* s_raw, float* V, char* ws, cudaStream_t st,
                        uint16_t* S16) {
  const ShardLayout L = shard_layout(N, n_v, d);
  float* w = reinterpret_cast<float*>(ws + L.w_off);
  float* Ppart = reinterpret_cast<float*>(ws + L.ppart_off);
  // Large scenes finalise each tile inside the pass (no second read of the partial sums from
  // HBM); below kFinalizeInPassTiles a separate kernel is faster (the pass is too short to hide
  // the finalising CTAs' extra work: 0.458 against 0.441 ms per query at 400 tiles, 6.11 against
  // 6.14 at 6400).
  constexpr int kFinalizeInPassTiles = 3200;
  const bool in_pass = N >= kFinalizeInPassTiles;
  unsigned int* cnt = in_pass ? reinterpret_cast<unsigned int*>(ws + L.cnt_off) : nullptr;
  launch_ex(fold_w_kernel, dim3((d + 255) / 256), dim3(256), 0, st, true, t, B, M, d, w, cnt, cnt ? N : 0);
  const int vw = (xdt == RIFT_BF16) ? 8 : 4;
  const int nvec_per_thread = (d / vw + SC_THREADS - 1) / SC_THREADS;
  auto go = [&](auto xt, auto nvec) {
    using XT = decltype(xt);
    launch_tokens<XT, decltype(nvec)::value>(X, N, n_v, d, L, w, token_scores, Ppart, cnt, V, s_raw, S16, st);
  };
  using I1 = std::integral_constant<int, 1>;
  using I2 = std::integral_constant<int, 2>;
  using I4 = std::integral_constant<int, 4>;
  if (xdt == RIFT_BF16) {
    if (nvec_per_thread <= 1) go(uint16_t{}, I1{});
    else if (nvec_per_thread <= 2) go(uint16_t{}, I2{});
    else go(uint16_t{}, I4{});
  } else {
    if (nvec_per_thread <= 1) go(float{}, I1{});
    else if (nvec_per_thread <= 2) go(float{}, I2{});
    else go(float{}, I4{});
  }
  if (in_pass) return 2;
  static_assert(SC_THREADS == 256, "the separate finalisation has the token pass's width");
  launch_ex(tile_finalize_kernel, dim3(N), dim3(SC_THREADS), 0, st, true, (const float*)Ppart, L.n_chunks, d,
            (const float*)w, V, s_raw, S16, N, (N + 7) & ~7);
  return 3;
}

int launch_smooth(const float* V, const float* s_raw, int N, int d, int row0, int n_rows, int m, float* s_tilde,
                  int* nbr, char* ws, cudaStream_t st, bool split_done) {
  const SmoothLayout L = smooth_layout(N, n_rows, d);
  int* topj = reinterpret_cast<int*>(ws + L.top_off);
  // candidates per row: m plus spares for the fp64 rescoring, at most the N - 1 other tiles
  const int C = m > 0 ? std::min(std::min(m + KNN_SPARE, RIFT_MAX_KNN), N - 1) : 0;
  int launched = 1;
  if (m > 0) {
    uint16_t* S16 = reinterpret_cast<uint16_t*>(ws + L.split_off);
    float* G = reinterpret_cast<float*>(ws + L.gram_off);
    const int Np = (N + 7) & ~7;
    const size_t n = (size_t)Np * (d / 8);
    if (!split_done)
      launch_ex(knn_split_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, st, true, V, N, Np, d, S16);
    EpiParams ep;
    ep.out_scale = 1.f / (KNN_SPLIT_SCALE * KNN_SPLIT_SCALE);
    // A = rows row0 .. row0 + n_rows - 1 of S read as [hi | hi | lo], B = all of S as [hi | lo | hi]
    ep.kmap_d = d / 64;
    ep.kmap_a = 1;
    ep.kmap_b = 2;
    // the whole scene's rows: G is symmetric (A holds the same rows as B, in the permuted parts
    // [hi | hi | lo] against [hi | lo | hi], whose product is symmetric up to the order of its sums)
    ep.symmetric = (row0 == 0 && n_rows == N) ? 1 : 0;
    // split-K partials for products with fewer tiles than SMs (a scene up to ~2000 tiles)
    void* part = L.splitk_bytes ? static_cast<void*>(ws + L.splitk_off) : nullptr;
    // S is written by an earlier kernel of the chain, not a constant operand
    if (launch_gemm_tc(S16 + (size_t)row0 * 2 * d, S16, n_rows, Np, 3 * d, EPI_STORE_F32, G, ep, st, part,
                       L.splitk_bytes, true, false))
      return -1;
    launch_ex(knn_gram_topc_kernel, dim3((n_rows + 3) / 4), dim3(128), 0, st, true, (const float*)G, N, Np, row0,
              n_rows, C, topj);
    launched += split_done ? 3 : 4;
  }
  launch_ex(knn_rescore_smooth_kernel, dim3(n_rows), dim3(32 * RIFT_MAX_KNN), 0, st, true, V, d,
            (const int*)topj, N, row0, C, m, s_raw, s_tilde, nbr);
  return launched;
}

int launch_score(const void* X, rift_dtype xdt, int N, int n_v, int d, const float* t, const float* B,
                 int M, int m, float* token_scores, float* s_raw, float* s_tilde, int* nbr, char* ws,
                 cudaStream_t st) {
  const ScoreLayout L = score_layout(N, n_v, d, M);
  float* V = reinterpret_cast<float*>(ws + L.V_off);
  // with neighbours to find, the token pass's finalisation also writes the Gram's split rows
  uint16_t* S16 = m > 0 ? reinterpret_cast<uint16_t*>(ws + L.smooth_off + L.S.split_off) : nullptr;
  const int a = launch_score_tokens(X, xdt, N, n_v, d, t, B, M, token_scores, s_raw, V, ws + L.tokens_off, st, S16);
  const int b = launch_smooth(V, s_raw, N, d, 0, N, m, s_tilde, nbr, ws + L.smooth_off, st, m > 0);
  return b < 0 ? -1 : a + b;
}

// (min, max) of n fp32 scores into range[0], range[1]; a NaN among them sets RIFT_EBIT_NONFINITE
// (min and max then skip it, as fminf / fmaxf do).  One CTA.
__global__ void __launch_bounds__(1024) score_range_kernel(const float* __restrict__ s, int n,
                                                           float* __restrict__ range) {
  pdl_trigger();
  pdl_wait();
  __shared__ float rmin[32], rmax[32];
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  float lo = INFINITY, hi = -INFINITY;
  bool bad = false;
  for (int i = tid; i < n; i += blockDim.x) {
    const float v = s[i];
    if (!isfinite(v)) bad = true;
    lo = fminf(lo, v);
    hi = fmaxf(hi, v);
  }
  if (bad) atomicOr(&g_err_score, RIFT_EBIT_NONFINITE);
  lo = warp_min(lo);
  hi = warp_max(hi);
  if (lane == 0) { rmin[wid] = lo; rmax[wid] = hi; }
  __syncthreads();
  if (tid < 32) {
    lo = warp_min(tid < (int)(blockDim.x >> 5) ? rmin[tid] : INFINITY);
    hi = warp_max(tid < (int)(blockDim.x >> 5) ? rmax[tid] : -INFINITY);
    if (tid == 0) { range[0] = lo; range[1] = hi; }
  }
}

void launch_score_range(const float* s, int n, float* range, cudaStream_t st) {
  launch_ex(score_range_kernel, dim3(1), dim3(1024), 0, st, true, s, n, range);
}

}  // namespace rift
