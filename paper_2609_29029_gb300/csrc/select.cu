// Stage 1 pruning and Stage 2 budgets and token selection on sm_103a.
//
//   prune_budget_kernel  (one CTA) per-scene min-max of the smoothed scores, u_i >= tau,
//                        the kept list (a block scan), the budget argmax of Eq. 2 and the
//                        exclusive scan of the budgets (the varlen offsets of the selection)
//   topb_kernel          (one CTA per kept tile) radix select of the b-th largest token
//                        score over order-preserving integer keys, ties to the lower index,
//                        and an ordered scan that writes the chosen indices ascending
//
// Every fp32 operation that decides an integer is a correctly rounded intrinsic written in
// the order the header documents, so the decisions are fixed by IEEE arithmetic.
#include "rift_internal.h"

namespace rift {

__device__ unsigned int g_err_select;

unsigned int read_clear_err_select() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_err_select, sizeof(v));
  cudaMemcpyToSymbol(g_err_select, &z, sizeof(z));
  return v;
}

constexpr int PB_THREADS = 1024;

// s_range (nullable): the min and max of the whole scene's smoothed scores, when these N tiles are
// one shard of it (the local scores are still checked for non-finite values).
__global__ void __launch_bounds__(PB_THREADS) prune_budget_kernel(
    const float* __restrict__ s, int N, int n_v, const float* __restrict__ p_ext, rift_policy pol,
    const float* __restrict__ s_range, float* __restrict__ u, int* __restrict__ kept, int* __restrict__ n_kept,
    int* __restrict__ budgets, int* __restrict__ sel_off) {
  pdl_trigger();
  pdl_wait();
  __shared__ float rmin[32], rmax[32];
  __shared__ int sh[33];
  __shared__ int s_bad;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  if (tid == 0) s_bad = 0;
  float lo = INFINITY, hi = -INFINITY;
  bool bad = false;
  for (int i = tid; i < N; i += PB_THREADS) {
    float v = s[i];
    if (!isfinite(v)) bad = true;
    lo = fminf(lo, v);
    hi = fmaxf(hi, v);
  }
  lo = warp_min(lo);
  hi = warp_max(hi);
  if (lane == 0) { rmin[wid] = lo; rmax[wid] = hi; }
  __syncthreads();
  if (bad) s_bad = 1;
  if (tid < 32) {
    lo = warp_min(tid < PB_THREADS / 32 ? rmin[tid] : INFINITY);
    hi = warp_max(tid < PB_THREADS / 32 ? rmax[tid] : -INFINITY);
    if (tid == 0) { rmin[0] = lo; rmax[0] = hi; }
  }
  __syncthreads();
  lo = rmin[0];
  hi = rmax[0];
  if (s_range) {
    lo = s_range[0];
    hi = s_range[1];
    if (!isfinite(lo) || !isfinite(hi)) s_bad = 1;  // every thread read s_bad after the barrier above
  }
  __syncthreads();
  if (s_bad) {
    if (tid == 0) { atomicOr(&g_err_select, RIFT_EBIT_NONFINITE); *n_kept = 0; }
    for (int j = tid; j <= N; j += PB_THREADS) sel_off[j] = 0;
    return;
  }
  const float range = __fsub_rn(hi, lo);
  // u, keep flags, compaction in ascending tile order
  int base = 0;
  for (int c0 = 0; c0 < N; c0 += PB_THREADS) {
    const int i = c0 + tid;
    int keep = 0;
    if (i < N) {
      float ui = (hi == lo) ? 1.f : __fdiv_rn(__fsub_rn(s[i], lo), range);
      u[i] = ui;
      keep = ui >= pol.tau ? 1 : 0;
    }
    int total;
    int pos = block_excl_scan(keep, sh, &total);
    if (keep) kept[base + pos] = i;
    base += total;
  }
  const int n = base;
  if (tid == 0) *n_kept = n;
  __syncthreads();
  // budgets: argmax_c U(c), U = ((p a+) + ((1 - p) a-)) - (lambda E), ties to the lower c
  int off = 0;
  for (int c0 = 0; c0 < n; c0 += PB_THREADS) {
    const int j = c0 + tid;
    int b = 0;
    if (j < n) {
      const int i = kept[j];
      const float p = p_ext ? p_ext[i] : u[i];
      if (!isfinite(p)) atomicOr(&g_err_select, RIFT_EBIT_NONFINITE);
      const float q = __fsub_rn(1.f, p);
      int best = 0;
      float bestU = 0.f;
      for (int c = 0; c < pol.n_c; ++c) {
        float acc = __fadd_rn(__fmul_rn(p, pol.alpha_pos[c]), __fmul_rn(q, pol.alpha_neg[c]));
        float Uc = __fsub_rn(acc, __fmul_rn(pol.lambda, pol.energy[c]));
        if (c == 0 || Uc > bestU) { best = c; bestU = Uc; }
      }
      b = pol.C[best];
      budgets[j] = b;
      // with the merge on, c - floor(ctx_num c / ctx_den) of the c tokens are selected (the
      // rest of the budget is contextual tokens); the full budget selects every token
      if (pol.ctx_num > 0 && b < n_v) b -= (pol.ctx_num * b) / pol.ctx_den;
    }
    int total;
    int pos = block_excl_scan(b, sh, &total);
    if (j < n) sel_off[j] = off + pos;
    off += total;
  }
  for (int j = n + tid; j <= N; j += PB_THREADS) sel_off[j] = off;
}

// Order-preserving map of fp32 to uint32 (larger float -> larger key); -0 maps like +0.
__device__ __forceinline__ uint32_t float_key(float f) {
  uint32_t b = __float_as_uint(f);
  if (b == 0x80000000u) b = 0u;
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

constexpr int TB_THREADS = 256;
constexpr int TB_KPT = RIFT_MAX_NV / TB_THREADS;  // keys per thread (4)

__global__ void __launch_bounds__(TB_THREADS) topb_kernel(const float* __restrict__ r, int n_v,
                                                          const int* __restrict__ kept,
                                                          const int* __restrict__ n_kept,
                                                          const int* __restrict__ budgets,
                                                          const int* __restrict__ sel_off,
                                                          int* __restrict__ sel) {
  pdl_trigger();
  pdl_wait();
  __shared__ int hist[256];
  __shared__ int sh[33];
  __shared__ uint32_t s_digit;
  __shared__ int s_rem;
  const int j = blockIdx.x;
  if (j >= *n_kept) return;
  const int tid = threadIdx.x, lane = tid & 31;
  const int tile = kept[j];
  const int b = sel_off[j + 1] - sel_off[j];  // tokens to select (the budget less its contextual tokens)
  uint32_t key[TB_KPT];
  bool valid[TB_KPT];
  bool bad = false;
#pragma unroll
  for (int e = 0; e < TB_KPT; ++e) {
    const int k = tid * TB_KPT + e;  // thread-major: index order = (thread, e)
    valid[e] = k < n_v;
    float f = valid[e] ? r[(size_t)tile * n_v + k] : 0.f;
    if (valid[e] && !isfinite(f)) bad = true;
    key[e] = float_key(f);
  }
  if (bad) atomicOr(&g_err_select, RIFT_EBIT_NONFINITE);

  // Radix select, 8 bits per pass from the top: the b-th largest key and how many of the
  // keys equal to it are taken (the lowest-index ones).
  uint32_t prefix = 0, mask = 0;
  int rem = b;
  for (int shift = 24; shift >= 0; shift -= 8) {
    hist[tid] = 0;
    __syncthreads();
#pragma unroll
    for (int e = 0; e < TB_KPT; ++e)
      if (valid[e] && (key[e] & mask) == prefix) atomicAdd(&hist[(key[e] >> shift) & 255u], 1);
    __syncthreads();
    if (tid < 32) {
      // lane l covers digits 255 - 8l down to 248 - 8l
      int c[8], loc = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) { c[q] = hist[255 - 8 * lane - q]; loc += c[q]; }
      const int inc = warp_incl_scan(loc);
      const int exc = inc - loc;
      if (exc < rem && rem <= inc) {
        int cum = exc;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          if (cum + c[q] >= rem) {
            s_digit = 255u - 8u * lane - q;
            s_rem = rem - cum;
            break;
          }
          cum += c[q];
        }
      }
    }
    __syncthreads();
    prefix |= s_digit << shift;
    mask |= 255u << shift;
    rem = s_rem;
    __syncthreads();
  }
  const uint32_t kth = prefix;
  const int need = rem;  // keys equal to kth that are selected

  int eq_loc = 0;
#pragma unroll
  for (int e = 0; e < TB_KPT; ++e) eq_loc += (valid[e] && key[e] == kth) ? 1 : 0;
  int tot;
  int eq_rank = block_excl_scan(eq_loc, sh, &tot);
  bool take[TB_KPT];
  int sel_loc = 0;
#pragma unroll
  for (int e = 0; e < TB_KPT; ++e) {
    bool eq = valid[e] && key[e] == kth;
    take[e] = valid[e] && (key[e] > kth || (eq && eq_rank < need));
    if (eq) ++eq_rank;
    sel_loc += take[e] ? 1 : 0;
  }
  int pos = block_excl_scan(sel_loc, sh, &tot);
  int* out = sel + sel_off[j];
#pragma unroll
  for (int e = 0; e < TB_KPT; ++e)
    if (take[e]) out[pos++] = tid * TB_KPT + e;
  (void)lane;
}

void launch_select(const float* token_scores, const float* tile_s, int N, int n_v, const float* p,
                   const rift_policy& pol, float* u, int* kept, int* n_kept, int* budgets, int* sel,
                   int* sel_off, cudaStream_t st, const float* s_range) {
  launch_ex(prune_budget_kernel, dim3(1), dim3(PB_THREADS), 0, st, true, tile_s, N, n_v, p, pol, s_range, u, kept,
            n_kept, budgets, sel_off);
  launch_ex(topb_kernel, dim3(N), dim3(TB_THREADS), 0, st, true, token_scores, n_v, (const int*)kept,
            (const int*)n_kept, (const int*)budgets, (const int*)sel_off, sel);
}

}  // namespace rift
