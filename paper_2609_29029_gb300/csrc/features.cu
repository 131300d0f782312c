// The per-tile features of the p_i predictor (Section 2.3, Stage 2: the tile embedding, its
// Stage-1 relevance, the vision-token scores and the relevance of its four quadrants) for a list of
// tiles, on sm_103a.
//
//   features_fold_kernel   w = t - (1/M) sum_j B_j (Eq. 1's background mean folded into one vector)
//   quad_sum_kernel        per (listed tile, quadrant, 2048 columns): the sum of the quadrant's
//                          g/2 x g/2 tokens (fp32, 16-byte loads, token rows in grid order)
//   features_final_kernel  per listed tile: each quadrant's Eq. 1 score l2norm(sum) . w, the tile
//                          embedding l2norm(sum of the four), and max / mean / population std of
//                          the tile's token scores (two passes)
#include "rift_internal.h"

namespace rift {

namespace ft {

constexpr int QT = 256;        // threads of the quadrant sum
constexpr int QCOLS = QT * 8;  // columns per CTA

__global__ void features_fold_kernel(const float* __restrict__ t, const float* __restrict__ B, int M, int d,
                                     float* __restrict__ w) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= d) return;
  float s = 0.f;
  for (int j = 0; j < M; ++j) s += B[(size_t)j * d + c];
  w[c] = M > 0 ? t[c] - s / (float)M : t[c];
}

template <typename XT>
__device__ __forceinline__ void load8(const XT* p, float (&v)[8]) {
  if constexpr (sizeof(XT) == 2) {
    unpack_bf16x8(*reinterpret_cast<const uint4*>(p), v);
  } else {
    const float4 a = reinterpret_cast<const float4*>(p)[0], b = reinterpret_cast<const float4*>(p)[1];
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  }
}

// Grid (list slot, quadrant 0..3, column block).  Qsum[slot][q][c] = sum over the quadrant's tokens.
template <typename XT>
__global__ void __launch_bounds__(QT) quad_sum_kernel(const XT* __restrict__ X, int N, int n_v, int d, int g,
                                                      const int* __restrict__ tiles, const int* __restrict__ n_tiles,
                                                      float* __restrict__ Qsum) {
  const int j = blockIdx.x;
  const int n = tiles ? *n_tiles : N;
  if (j >= n) return;
  const int tile = tiles ? tiles[j] : j;
  if (tile < 0 || tile >= N) return;
  const int q = blockIdx.y, h = g / 2;
  const int r0 = (q >> 1) * h, c0 = (q & 1) * h;
  const int col = blockIdx.z * QCOLS + threadIdx.x * 8;
  if (col >= d) return;
  const XT* Xt = X + (size_t)tile * n_v * d;
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int r = r0; r < r0 + h; ++r) {
#pragma unroll 4
    for (int c = c0; c < c0 + h; ++c) {
      float x[8];
      load8(Xt + (size_t)(r * g + c) * d + col, x);
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] += x[e];
    }
  }
  float* out = Qsum + ((size_t)j * 4 + q) * d + col;
  reinterpret_cast<float4*>(out)[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
  reinterpret_cast<float4*>(out)[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
}

__global__ void __launch_bounds__(256) features_final_kernel(const float* __restrict__ Qsum, const float* __restrict__ w,
                                                             const float* __restrict__ token_scores, int N, int n_v,
                                                             int d, const int* __restrict__ tiles,
                                                             const int* __restrict__ n_tiles,
                                                             float* __restrict__ features, float* __restrict__ V) {
  __shared__ float red[32];
  const int j = blockIdx.x;
  const int n = tiles ? *n_tiles : N;
  if (j >= n) return;
  const int tile = tiles ? tiles[j] : j;
  if (tile < 0 || tile >= N) return;
  const float* Q = Qsum + (size_t)j * 4 * d;
  float* f = features + (size_t)j * RIFT_N_FEATURES;
  for (int q = 0; q < 4; ++q) {
    float ss = 0.f, dt = 0.f;
    for (int c = threadIdx.x; c < d; c += blockDim.x) {
      const float v = Q[(size_t)q * d + c];
      ss += v * v;
      dt += v * w[c];
    }
    ss = block_sum(ss, red);
    dt = block_sum(dt, red);
    if (threadIdx.x == 0) f[q] = ss > 0.f ? dt / sqrtf(ss) : 0.f;
  }
  if (V) {
    float ss = 0.f;
    for (int c = threadIdx.x; c < d; c += blockDim.x) {
      const float v = (Q[c] + Q[d + c]) + (Q[2 * d + c] + Q[3 * d + c]);
      ss += v * v;
    }
    ss = block_sum(ss, red);
    const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
    for (int c = threadIdx.x; c < d; c += blockDim.x)
      V[(size_t)j * d + c] = ((Q[c] + Q[d + c]) + (Q[2 * d + c] + Q[3 * d + c])) * inv;
  }
  const float* r = token_scores + (size_t)tile * n_v;
  float mx = -INFINITY, sum = 0.f;
  for (int k = threadIdx.x; k < n_v; k += blockDim.x) {
    mx = fmaxf(mx, r[k]);
    sum += r[k];
  }
  mx = warp_max(mx);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
  __syncthreads();
  mx = red[0];
  for (int w2 = 1; w2 < (int)(blockDim.x >> 5); ++w2) mx = fmaxf(mx, red[w2]);
  const float mean = block_sum(sum, red) / (float)n_v;
  float var = 0.f;
  for (int k = threadIdx.x; k < n_v; k += blockDim.x) var += (r[k] - mean) * (r[k] - mean);
  var = block_sum(var, red) / (float)n_v;
  if (threadIdx.x == 0) {
    f[4] = mx;
    f[5] = mean;
    f[6] = sqrtf(var);
  }
}

}  // namespace ft

FeaturesLayout features_layout(int N, int d) {
  FeaturesLayout L{};
  size_t off = 0;
  auto take = [&](size_t bytes) { size_t o = off; off += (bytes + 255) & ~size_t(255); return o; };
  L.w_off = take((size_t)d * sizeof(float));
  L.qsum_off = take((size_t)N * 4 * d * sizeof(float));
  L.total = off;
  return L;
}

int launch_features(const void* X, rift_dtype xdt, int N, int n_v, int d, int g, const float* t, const float* B, int M,
                    const float* token_scores, const int* tiles, const int* n_tiles, float* features, float* V,
                    char* ws, cudaStream_t st) {
  using namespace ft;
  const FeaturesLayout L = features_layout(N, d);
  float* w = reinterpret_cast<float*>(ws + L.w_off);
  float* Qsum = reinterpret_cast<float*>(ws + L.qsum_off);
  features_fold_kernel<<<(d + 255) / 256, 256, 0, st>>>(t, B, M, d, w);
  const dim3 gq(N, 4, (d + QCOLS - 1) / QCOLS);
  if (xdt == RIFT_BF16)
    quad_sum_kernel<uint16_t><<<gq, QT, 0, st>>>(static_cast<const uint16_t*>(X), N, n_v, d, g, tiles, n_tiles, Qsum);
  else
    quad_sum_kernel<float><<<gq, QT, 0, st>>>(static_cast<const float*>(X), N, n_v, d, g, tiles, n_tiles, Qsum);
  features_final_kernel<<<N, 256, 0, st>>>(Qsum, w, token_scores, N, n_v, d, tiles, n_tiles, features, V);
  return 3;
}

}  // namespace rift
