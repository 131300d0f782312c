// Merge of the unselected tokens into contextual tokens on sm_103a (Section 2.3, Stage 2: Rift
// uses VisionZip's mechanism to keep the dominant tokens and merge the remainder).
//
// For kept slot j with m_j = budgets[j] - s_j contextual tokens (s_j selected tokens):
//   merge_plan_kernel     m_j (capped at the R_j unselected tokens) and their offsets ctx_off
//   merge_targets_kernel  the unselected tokens in ascending index, the targets (every
//                         floor(R_j / m_j)-th of them from the first) and the targets' norms
//   merge_assign_kernel   (fp32 tokens) per 64 unselected tokens x 64 targets: fp32 dot products in
//                         32-term chunks, a running top 2 per token; the two are recomputed as
//                         float-float sums (good to ~2^-44) and compared as x.t1 / ||t1|| vs
//                         x.t2 / ||t2|| in fp64, so the decision is the cosine argmax of the exact
//                         arithmetic (ties to the lower target)
//   (bf16 tokens) merge_screen_kernel (gemm_tc.cu) takes the top 2 from a tcgen05 product of
//                         each 128-token block with the slot's target rows, and
//                         merge_decide_kernel makes the same float-float decision between them
//   merge_groups_kernel   the groups as member lists in ascending token index (counting sort)
//   merge_mean_kernel     per contextual token: the fp32 sum of its members' rows in that order,
//                         divided by the group size, stored as bf16
#include "rift_internal.h"

namespace rift {

__device__ unsigned int g_err_merge;

unsigned int read_clear_err_merge() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_err_merge, sizeof(v));
  cudaMemcpyToSymbol(g_err_merge, &z, sizeof(z));
  return v;
}

namespace mg {

constexpr int TB = 64;     // tokens and targets per block of the similarity pass
constexpr int KC = 32;     // d-chunk staged per step (summed in 32-term sub-chunks)

template <typename XT>
__device__ __forceinline__ float load_x(const XT* p) {
  if constexpr (sizeof(XT) == 2)
    return bf16_bits_to_float(*reinterpret_cast<const uint16_t*>(p));
  else
    return *p;
}

// Eight consecutive elements of a row (16-byte aligned) as floats.
template <typename XT>
__device__ __forceinline__ void load8(const XT* p, float (&v)[8]) {
  if constexpr (sizeof(XT) == 2) {
    unpack_bf16x8(*reinterpret_cast<const uint4*>(p), v);
  } else {
    const float4 a = reinterpret_cast<const float4*>(p)[0], b = reinterpret_cast<const float4*>(p)[1];
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  }
}

// Float-float accumulation of a.b over d terms (d % 256 == 0) by one warp (TwoProduct with an
// FMA, TwoSum), eight elements per lane and step, then the lanes' pairs summed in fp64.
template <typename XT>
__device__ double ff_dot(const XT* a, const XT* b, int d, int lane) {
  float hi = 0.f, lo = 0.f;
  for (int k = lane * 8; k < d; k += 256) {
    float x[8], y[8];
    load8(a + k, x);
    load8(b + k, y);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float p = __fmul_rn(x[e], y[e]);
      const float pe = fmaf(x[e], y[e], -p);
      const float s = __fadd_rn(hi, p);
      const float bb = __fsub_rn(s, hi);
      const float er = __fadd_rn(__fsub_rn(hi, __fsub_rn(s, bb)), __fsub_rn(p, bb));
      hi = s;
      lo = __fadd_rn(lo, __fadd_rn(er, pe));
    }
  }
  double acc = (double)hi + (double)lo;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  return acc;
}

// a.b and a.c in one pass over a, each summed as ff_dot does.
template <typename XT>
__device__ double2 ff_dot2(const XT* a, const XT* b, const XT* c, int d, int lane) {
  float hb = 0.f, lb = 0.f, hc = 0.f, lc = 0.f;
  auto step = [](float x, float y, float& hi, float& lo) {
    const float p = __fmul_rn(x, y);
    const float pe = fmaf(x, y, -p);
    const float s = __fadd_rn(hi, p);
    const float bb = __fsub_rn(s, hi);
    const float er = __fadd_rn(__fsub_rn(hi, __fsub_rn(s, bb)), __fsub_rn(p, bb));
    hi = s;
    lo = __fadd_rn(lo, __fadd_rn(er, pe));
  };
  for (int k = lane * 8; k < d; k += 256) {
    float x[8], y[8], z[8];
    load8(a + k, x);
    load8(b + k, y);
    load8(c + k, z);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      step(x[e], y[e], hb, lb);
      step(x[e], z[e], hc, lc);
    }
  }
  double sb = (double)hb + (double)lb, sc = (double)hc + (double)lc;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    sb += __shfl_xor_sync(0xffffffffu, sb, o);
    sc += __shfl_xor_sync(0xffffffffu, sc, o);
  }
  return make_double2(sb, sc);
}

// m_j = min(budgets[j] - s_j, n_v - s_j) and its exclusive prefix sum over the kept slots.  If
// the total exceeds max_ctx, RIFT_EBIT_CAPACITY is set and every m_j is taken as 0 (no contextual
// row is then written or read).
__global__ void __launch_bounds__(1024) merge_plan_kernel(const int* __restrict__ n_kept,
                                                          const int* __restrict__ budgets,
                                                          const int* __restrict__ sel_off, int N, int n_v,
                                                          int max_ctx, int* __restrict__ ctx_off) {
  __shared__ int sh[33];
  const int n = *n_kept;
  auto count = [&](int j) {
    const int s = sel_off[j + 1] - sel_off[j];
    return max(0, min(budgets[j] - s, n_v - s));
  };
  int total_all = 0;
  for (int c0 = 0; c0 < n; c0 += blockDim.x) {
    const int j = c0 + threadIdx.x;
    int total;
    block_excl_scan(j < n ? count(j) : 0, sh, &total);
    total_all += total;
  }
  const bool fits = total_all <= max_ctx;
  if (threadIdx.x == 0 && !fits) atomicOr(&g_err_merge, RIFT_EBIT_CAPACITY);
  int base = 0;
  for (int c0 = 0; c0 < n; c0 += blockDim.x) {
    const int j = c0 + threadIdx.x;
    const int m = (j < n && fits) ? count(j) : 0;
    int total;
    const int pos = block_excl_scan(m, sh, &total);
    if (j < n) ctx_off[j] = base + pos;
    base += total;
  }
  for (int j = n + threadIdx.x; j <= N; j += blockDim.x) ctx_off[j] = base;
}

// One CTA per kept slot: rest[j][0 .. R) = the unselected tokens in ascending index, the targets
// (written to ctx_target) and their norms (tnorm, fp64 from a float-float sum of squares).
template <typename XT>
__global__ void __launch_bounds__(256) merge_targets_kernel(const XT* __restrict__ X, int n_v, int d,
                                                            const int* __restrict__ kept,
                                                            const int* __restrict__ n_kept,
                                                            const int* __restrict__ sel,
                                                            const int* __restrict__ sel_off,
                                                            const int* __restrict__ ctx_off, int max_ctx,
                                                            int* __restrict__ rest, int* __restrict__ ctx_target,
                                                            double* __restrict__ tnorm, int* __restrict__ pos,
                                                            float* __restrict__ tinv, uint16_t* __restrict__ trow) {
  __shared__ unsigned char chosen[RIFT_MAX_NV];
  __shared__ int sh[33];
  const int j = blockIdx.x;
  if (j >= *n_kept) return;
  const int so = sel_off[j], s = sel_off[j + 1] - so;
  const int co = ctx_off[j], m = ctx_off[j + 1] - co;
  for (int k = threadIdx.x; k < n_v; k += blockDim.x) chosen[k] = 0;
  __syncthreads();
  for (int q = threadIdx.x; q < s; q += blockDim.x) {
    const int k = sel[so + q];
    if (k >= 0 && k < n_v) chosen[k] = 1;
  }
  __syncthreads();
  int* rj = rest + (size_t)j * n_v;
  int base = 0;
  for (int c0 = 0; c0 < n_v; c0 += blockDim.x) {
    const int k = c0 + threadIdx.x;
    const int f = (k < n_v && !chosen[k]) ? 1 : 0;
    int total;
    const int at = block_excl_scan(f, sh, &total);
    if (f) rj[base + at] = k;
    if (pos && k < n_v) pos[(size_t)j * n_v + k] = f ? base + at : -1;
    base += total;
  }
  __syncthreads();
  const int R = base;
  if (m == 0 || R == 0) return;
  const int step = R / m;
  const XT* Xt = X + (size_t)kept[j] * n_v * d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int q = warp; q < m; q += blockDim.x / 32) {
    const int t = rj[q * step];
    const double nn = ff_dot(Xt + (size_t)t * d, Xt + (size_t)t * d, d, lane);
    if (co + q >= max_ctx) continue;
    if (lane == 0) {
      ctx_target[co + q] = t;
      tnorm[co + q] = sqrt(nn);
      if (tinv) tinv[co + q] = nn > 0.0 ? (float)(1.0 / sqrt(nn)) : 0.f;  // a zero target has similarity 0
    }
    if (trow) {  // the target's row, for the tensor-core screening (bf16 tokens only)
      const uint4* src = reinterpret_cast<const uint4*>(Xt + (size_t)t * d);
      uint4* dst = reinterpret_cast<uint4*>(trow + (size_t)(co + q) * d);
      for (int c = lane; c < d / 8; c += 32) dst[c] = src[c];
    }
  }
}

// Grid (blocks of 8 unselected positions, kept slot), 8 warps: for the position a of each warp
// (not a target), the better of its two screened candidates cand[j][a] at ~fp64 accuracy:
// x.t1 / ||t1|| vs x.t2 / ||t2|| from float-float dot products (ties to the lower target).
template <typename XT>
__global__ void __launch_bounds__(256) merge_decide_kernel(const XT* __restrict__ X, int n_v, int d,
                                                           const int* __restrict__ kept,
                                                           const int* __restrict__ n_kept,
                                                           const int* __restrict__ sel_off,
                                                           const int* __restrict__ ctx_off, int max_ctx,
                                                           const int* __restrict__ rest,
                                                           const int* __restrict__ ctx_target,
                                                           const double* __restrict__ tnorm,
                                                           const int2* __restrict__ cand, int* __restrict__ assign) {
  const int j = blockIdx.y;
  if (j >= *n_kept) return;
  const int R = n_v - (sel_off[j + 1] - sel_off[j]);
  const int co = ctx_off[j], m = ctx_off[j + 1] - co;
  if (m == 0 || co + m > max_ctx) return;
  const int step = R / m;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int a = blockIdx.x * 8 + warp;
  if (a >= R || (a % step == 0 && a / step < m)) return;  // targets keep their own group
  int2 c = cand[(size_t)j * n_v + a];
  if (c.x < 0 || c.x >= m) {  // no finite similarity (a NaN token): the first target
    if (lane == 0) atomicOr(&g_err_merge, RIFT_EBIT_NONFINITE);
    c = make_int2(0, -1);
  }
  int choice = c.x;
  if (c.y >= 0 && c.y < m) {
    const XT* Xt = X + (size_t)kept[j] * n_v * d;
    const int k = rest[(size_t)j * n_v + a];
    const int t1 = ctx_target[co + c.x], t2 = ctx_target[co + c.y];
    const double2 dd = ff_dot2(Xt + (size_t)k * d, Xt + (size_t)t1 * d, Xt + (size_t)t2 * d, d, lane);
    const double d1 = dd.x, d2 = dd.y;
    const double n1 = tnorm[co + c.x], n2 = tnorm[co + c.y];
    const double s1 = n1 > 0.0 ? d1 / n1 : 0.0, s2 = n2 > 0.0 ? d2 / n2 : 0.0;
    if (s2 > s1 || (s2 == s1 && c.y < c.x)) choice = c.y;
  }
  if (lane == 0) assign[(size_t)j * n_v + a] = choice;
}

// Grid (kept slot, block of TB unselected tokens).  assign[j][a] = target index of rest[a].
template <typename XT>
__global__ void __launch_bounds__(256) merge_assign_kernel(const XT* __restrict__ X, int n_v, int d,
                                                           const int* __restrict__ kept,
                                                           const int* __restrict__ n_kept,
                                                           const int* __restrict__ sel_off,
                                                           const int* __restrict__ ctx_off, int max_ctx,
                                                           const int* __restrict__ rest,
                                                           const int* __restrict__ ctx_target,
                                                           const double* __restrict__ tnorm,
                                                           int* __restrict__ assign) {
  extern __shared__ float ab_sm[];  // As[KC][TB + 4], Bs[KC][TB + 4]
  float (*As)[TB + 4] = reinterpret_cast<float (*)[TB + 4]>(ab_sm);
  float (*Bs)[TB + 4] = reinterpret_cast<float (*)[TB + 4]>(ab_sm + KC * (TB + 4));
  __shared__ float best_v[TB][2];
  __shared__ int best_j[TB][2];
  __shared__ float inv_n[TB];
  const int j = blockIdx.y;  // the token blocks of one slot are adjacent: its target rows stay in L2
  if (j >= *n_kept) return;
  const int s = sel_off[j + 1] - sel_off[j];
  const int R = n_v - s;
  const int co = ctx_off[j], m = ctx_off[j + 1] - co;
  const int a0 = blockIdx.x * TB;
  if (m == 0 || a0 >= R || co + m > max_ctx) return;
  const int* rj = rest + (size_t)j * n_v;
  const XT* Xt = X + (size_t)kept[j] * n_v * d;
  const int tid = threadIdx.x, ti = tid >> 4, tj = tid & 15;
  if (tid < TB) {
    best_v[tid][0] = best_v[tid][1] = -INFINITY;
    best_j[tid][0] = best_j[tid][1] = -1;
  }
  for (int b0 = 0; b0 < m; b0 += TB) {
    if (tid < TB) {
      const double nn = b0 + tid < m ? tnorm[co + b0 + tid] : 0.0;
      inv_n[tid] = nn > 0.0 ? (float)(1.0 / nn) : 0.f;  // a zero target has similarity 0
    }
    float acc[4][4] = {};
    // 64 rows x KC columns per operand and chunk: four 8-column groups per thread and operand,
    // kept packed while the next chunk's loads are in flight
    const int srow = tid >> 2, scol = (tid & 3) * 8;
    const XT* pa = a0 + srow < R ? Xt + (size_t)rj[a0 + srow] * d + scol : nullptr;
    const XT* pb = b0 + srow < m ? Xt + (size_t)ctx_target[co + b0 + srow] * d + scol : nullptr;
    constexpr int NG = KC / 32;  // 8-column groups per thread and operand
    float va[NG][8], vb[NG][8];
    auto fetch = [&](int k0) {
#pragma unroll
      for (int g = 0; g < NG; ++g) {
#pragma unroll
        for (int e = 0; e < 8; ++e) va[g][e] = vb[g][e] = 0.f;
        if (k0 + 32 * g >= d) continue;  // d % 32 == 0: a group is wholly inside the row or past it
        if (pa) load8(pa + k0 + 32 * g, va[g]);
        if (pb) load8(pb + k0 + 32 * g, vb[g]);
      }
    };
    fetch(0);
    for (int k0 = 0; k0 < d; k0 += KC) {
#pragma unroll
      for (int g = 0; g < NG; ++g)
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          As[32 * g + scol + e][srow] = va[g][e];
          Bs[32 * g + scol + e][srow] = vb[g][e];
        }
      __syncthreads();
      if (k0 + KC < d) fetch(k0 + KC);
#pragma unroll 1
      for (int kc = 0; kc < KC; kc += 32) {
        float part[4][4] = {};
#pragma unroll 8
        for (int k = kc; k < kc + 32; ++k) {
          const float4 av = *reinterpret_cast<const float4*>(&As[k][ti * 4]);
          const float4 bv = *reinterpret_cast<const float4*>(&Bs[k][tj * 4]);
          const float aa[4] = {av.x, av.y, av.z, av.w}, bb[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
          for (int r = 0; r < 4; ++r)
#pragma unroll
            for (int c = 0; c < 4; ++c) part[r][c] = fmaf(aa[r], bb[c], part[r][c]);
        }
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
          for (int c = 0; c < 4; ++c) acc[r][c] += part[r][c];
      }
      __syncthreads();
    }
    // running top 2 per token: thread (ti, tj) offers its 4 x 4 candidates row by row
    for (int w = 0; w < 16; ++w) {
      if (tj == w) {
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const int row = ti * 4 + r;
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            const int b = b0 + tj * 4 + c;
            if (b >= m) continue;
            const float v = acc[r][c] * inv_n[tj * 4 + c];
            if (v > best_v[row][0] || (v == best_v[row][0] && b < best_j[row][0])) {
              best_v[row][1] = best_v[row][0];
              best_j[row][1] = best_j[row][0];
              best_v[row][0] = v;
              best_j[row][0] = b;
            } else if (v > best_v[row][1] || (v == best_v[row][1] && b < best_j[row][1])) {
              best_v[row][1] = v;
              best_j[row][1] = b;
            }
          }
        }
      }
      __syncthreads();
    }
  }
  // decide between the top two at ~fp64 accuracy: x.t1 / ||t1|| vs x.t2 / ||t2||
  const int warp = tid >> 5, lane = tid & 31;
  for (int row = warp; row < TB; row += 8) {
    const int a = a0 + row;
    if (a >= R) break;
    const int k = rj[a];
    int choice = best_j[row][0];
    const int j2 = best_j[row][1];
    if (j2 >= 0) {
      const int t1 = ctx_target[co + choice], t2 = ctx_target[co + j2];
      const double d1 = ff_dot(Xt + (size_t)k * d, Xt + (size_t)t1 * d, d, lane);
      const double d2 = ff_dot(Xt + (size_t)k * d, Xt + (size_t)t2 * d, d, lane);
      const double n1 = tnorm[co + choice], n2 = tnorm[co + j2];
      const double s1 = n1 > 0.0 ? d1 / n1 : 0.0, s2 = n2 > 0.0 ? d2 / n2 : 0.0;
      if (s2 > s1 || (s2 == s1 && j2 < choice)) choice = j2;
    }
    if (lane == 0) assign[(size_t)j * n_v + a] = choice;
  }
}

// One CTA per kept slot: the slot's groups as member lists, ascending token index within each
// group (targets at their own index): gstart[j][q] .. gstart[j][q+1] in memb[j].  A counting sort
// whose placement pass runs in token order on one warp.
__global__ void __launch_bounds__(256) merge_groups_kernel(int n_v, const int* __restrict__ n_kept,
                                                           const int* __restrict__ sel_off,
                                                           const int* __restrict__ ctx_off, int max_ctx,
                                                           const int* __restrict__ rest,
                                                           const int* __restrict__ assign, int* __restrict__ memb,
                                                           int* __restrict__ gstart) {
  __shared__ int cnt[RIFT_MAX_NV + 1];
  const int j = blockIdx.x;
  if (j >= *n_kept) return;
  const int R = n_v - (sel_off[j + 1] - sel_off[j]);
  const int co = ctx_off[j], m = ctx_off[j + 1] - co;
  if (m == 0 || co + m > max_ctx) return;
  const int step = R / m;
  const int* rj = rest + (size_t)j * n_v;
  const int* aj = assign + (size_t)j * n_v;
  auto group = [&](int a) {
    if (a % step == 0 && a / step < m) return a / step;
    const int g = aj[a];
    return (g >= 0 && g < m) ? g : 0;  // an unassigned token (no finite similarity) joins the first group
  };
  for (int q = threadIdx.x; q <= m; q += blockDim.x) cnt[q] = 0;
  __syncthreads();
  for (int a = threadIdx.x; a < R; a += blockDim.x) atomicAdd(&cnt[group(a)], 1);
  __syncthreads();
  if (threadIdx.x == 0) {
    int* gs = gstart + (size_t)j * (n_v + 1);
    int acc = 0;
    for (int q = 0; q < m; ++q) {  // cnt becomes each group's next free slot
      const int c = cnt[q];
      gs[q] = acc;
      cnt[q] = acc;
      acc += c;
    }
    gs[m] = acc;
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    // placement in token order by one warp, 32 tokens at a time: a token's slot is its group's
    // next free one plus the number of lower lanes of the same group
    const int lane = threadIdx.x;
    int* mj = memb + (size_t)j * n_v;
    for (int a0 = 0; a0 < R; a0 += 32) {
      const int a = a0 + lane;
      const int g = a < R ? group(a) : -1 - lane;  // idle lanes match no one
      const unsigned same = __match_any_sync(0xffffffffu, g);
      if (a < R) mj[cnt[g] + __popc(same & ((1u << lane) - 1u))] = rj[a];
      __syncwarp();
      if (a < R && (same >> lane) == 1u) cnt[g] += __popc(same);  // the group's highest lane
      __syncwarp();
    }
  }
}

// Grid (kept slot, y), 256 threads: contextual token q = y, y + gridDim.y, ... is the mean of its
// group's rows, summed in fp32 in member order (ascending index), each thread owning d / 256 of
// the columns; stored as bf16.
constexpr int MT = 256, MV = RIFT_MERGE_MAX_D / (MT * 8);
template <typename XT>
__global__ void __launch_bounds__(MT) merge_mean_kernel(const XT* __restrict__ X, int n_v, int d,
                                                        const int* __restrict__ kept, const int* __restrict__ n_kept,
                                                        const int* __restrict__ ctx_off, int max_ctx,
                                                        const int* __restrict__ memb, const int* __restrict__ gstart,
                                                        uint16_t* __restrict__ ctx) {
  const int j = blockIdx.x;
  if (j >= *n_kept) return;
  const int co = ctx_off[j], m = ctx_off[j + 1] - co;
  if (m == 0 || co + m > max_ctx) return;
  const int* gs = gstart + (size_t)j * (n_v + 1);
  const int* mj = memb + (size_t)j * n_v;
  const XT* Xt = X + (size_t)kept[j] * n_v * d;
  for (int q = blockIdx.y; q < m; q += gridDim.y) {
    const int g0 = gs[q], g1 = gs[q + 1];
    float acc[MV][8];
#pragma unroll
    for (int v = 0; v < MV; ++v)
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[v][e] = 0.f;
    for (int g = g0; g < g1; ++g) {
      const XT* row = Xt + (size_t)mj[g] * d;
#pragma unroll
      for (int v = 0; v < MV; ++v) {
        const int c = (threadIdx.x + v * MT) * 8;
        if (c < d) {
          float x[8];
          load8(row + c, x);
#pragma unroll
          for (int e = 0; e < 8; ++e) acc[v][e] += x[e];
        }
      }
    }
    const float inv = 1.f / (float)(g1 - g0);
#pragma unroll
    for (int v = 0; v < MV; ++v) {
      const int c = (threadIdx.x + v * MT) * 8;
      if (c < d) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) w[e] = pack_bf16x2(acc[v][2 * e] * inv, acc[v][2 * e + 1] * inv);
        *reinterpret_cast<uint4*>(ctx + (size_t)(co + q) * d + c) = make_uint4(w[0], w[1], w[2], w[3]);
      }
    }
  }
}

}  // namespace mg

MergeLayout merge_layout(int N, int n_v) {
  MergeLayout L{};
  size_t off = 0;
  auto take = [&](size_t bytes) { size_t o = off; off += (bytes + 255) & ~size_t(255); return o; };
  L.rest_off = take((size_t)N * n_v * sizeof(int));
  L.assign_off = take((size_t)N * n_v * sizeof(int));
  L.tnorm_off = take((size_t)N * n_v * sizeof(double));
  L.memb_off = take((size_t)N * n_v * sizeof(int));
  L.gstart_off = take((size_t)N * (n_v + 1) * sizeof(int));
  L.pos_off = take((size_t)N * n_v * sizeof(int));
  L.tinv_off = take((size_t)N * n_v * sizeof(float));  // at most n_v - 1 targets per slot
  L.cand_off = take((size_t)N * n_v * sizeof(int2));
  L.total = off;
  return L;
}

int launch_merge(const void* X, rift_dtype xdt, int N, int n_v, int d, const int* kept, const int* n_kept,
                 const int* budgets, const int* sel, const int* sel_off, uint16_t* ctx, int max_ctx, int* ctx_off,
                 int* ctx_target, char* ws, cudaStream_t st) {
  using namespace mg;
  const MergeLayout L = merge_layout(N, n_v);
  int* rest = reinterpret_cast<int*>(ws + L.rest_off);
  int* assign = reinterpret_cast<int*>(ws + L.assign_off);
  double* tnorm = reinterpret_cast<double*>(ws + L.tnorm_off);
  int* memb = reinterpret_cast<int*>(ws + L.memb_off);
  int* gstart = reinterpret_cast<int*>(ws + L.gstart_off);
  int* pos = reinterpret_cast<int*>(ws + L.pos_off);
  float* tinv = reinterpret_cast<float*>(ws + L.tinv_off);
  int2* cand = reinterpret_cast<int2*>(ws + L.cand_off);
  merge_plan_kernel<<<1, 1024, 0, st>>>(n_kept, budgets, sel_off, N, n_v, max_ctx, ctx_off);
  const dim3 ga((n_v + TB - 1) / TB, N), gm(N, 32);
  const size_t ab_bytes = 2 * (size_t)KC * (TB + 4) * sizeof(float);
  if (xdt == RIFT_BF16) {
    // bf16 tokens: the target rows go to ctx (overwritten by the means at the end), the top two
    // of every token come from the tensor cores, the choice between them from float-float sums
    const uint16_t* x = static_cast<const uint16_t*>(X);
    merge_targets_kernel<uint16_t><<<N, 256, 0, st>>>(x, n_v, d, kept, n_kept, sel, sel_off, ctx_off, max_ctx, rest,
                                                      ctx_target, tnorm, pos, tinv, ctx);
    if (max_ctx > 0 &&
        launch_merge_screen(x, N, n_v, d, kept, n_kept, sel_off, ctx_off, max_ctx, ctx, tinv, pos, cand, st))
      return -1;
    merge_decide_kernel<uint16_t><<<dim3((n_v + 7) / 8, N), 256, 0, st>>>(x, n_v, d, kept, n_kept, sel_off, ctx_off,
                                                                        max_ctx, rest, ctx_target, tnorm, cand,
                                                                        assign);
    merge_groups_kernel<<<N, 256, 0, st>>>(n_v, n_kept, sel_off, ctx_off, max_ctx, rest, assign, memb, gstart);
    merge_mean_kernel<uint16_t><<<gm, MT, 0, st>>>(x, n_v, d, kept, n_kept, ctx_off, max_ctx, memb, gstart, ctx);
    return max_ctx > 0 ? 6 : 5;
  } else {
    const float* x = static_cast<const float*>(X);
    merge_targets_kernel<float><<<N, 256, 0, st>>>(x, n_v, d, kept, n_kept, sel, sel_off, ctx_off, max_ctx, rest,
                                                   ctx_target, tnorm, nullptr, nullptr, nullptr);
    static std::atomic<unsigned long long> smem_raised{0};
    if (raise_smem_limit(smem_raised, merge_assign_kernel<float>, (int)ab_bytes) != cudaSuccess) return -1;
    merge_assign_kernel<float><<<ga, 256, ab_bytes, st>>>(x, n_v, d, kept, n_kept, sel_off, ctx_off, max_ctx, rest,
                                                   ctx_target, tnorm, assign);
    merge_groups_kernel<<<N, 256, 0, st>>>(n_v, n_kept, sel_off, ctx_off, max_ctx, rest, assign, memb, gstart);
    merge_mean_kernel<float><<<gm, MT, 0, st>>>(x, n_v, d, kept, n_kept, ctx_off, max_ctx, memb, gstart, ctx);
  }
  return 5;
}

}  // namespace rift
