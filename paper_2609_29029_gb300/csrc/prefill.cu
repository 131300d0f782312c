// Decoder prefill over the packed batch (Section 2.1): the per-layer kernel sequence, the
// fused RMSNorm kernels and RoPE.
//
// Per layer, with the residual stream h kept in fp32 and every GEMM operand in fp16:
//   xn  = RMSNorm(h) g_attn                      rmsnorm_kernel            (fp16 out)
//   qkv = xn W_qkv^T, RoPE on q and k            GEMM, RoPE epilogue on the fp32 accumulators
//   a   = causal varlen attention(q, k, v)       attention
//   h  += a W_o^T                                GEMM, fp32 residual epilogue
//   xn  = RMSNorm(h) g_ffn
//   act = SiLU(xn W_g^T) * (xn W_u^T)            GEMM, SwiGLU epilogue (interleaved gate/up)
//   h  += act W_down^T                           GEMM, fp32 residual epilogue
// and finally hidden = RMSNorm(h) g_final in bf16.  Optional outputs: each layer's keys (after
// RoPE) and values copied out of the QKV buffer (the KV cache), and the logits of every
// sequence's last token, RMSNorm(h_last) g_final times the output matrix.
//
// The decode step runs the same layer sequence for one new token per sequence, at position L_i,
// with the attention replaced by decode_attn_kernel over the sequence's cached keys and values
// plus the token's own.
// fp16 rather than bf16 operands: after 32 layers the bf16 rounding of the GEMM inputs alone
// moves the final hidden states by about 3% of their largest magnitude; fp16 (3 more mantissa
// bits, same tensor-core rate, LLaVA-1.5-7B's checkpoint dtype) keeps the whole path near 0.5%.
#include <atomic>
#include <type_traits>

#include "rift_internal.h"

namespace rift {

__device__ unsigned int g_err_prefill;

unsigned int read_clear_err_prefill() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_err_prefill, sizeof(v));
  cudaMemcpyToSymbol(g_err_prefill, &z, sizeof(z));
  return v;
}

constexpr int NORM_THREADS = 256;

// One row of the RMSNorm below.
template <bool IN_BF16, bool OUT_F16, int VPT>
__device__ __forceinline__ void rmsnorm_row(const void* __restrict__ in, float* __restrict__ h32,
                                            const uint16_t* __restrict__ gain, uint16_t* __restrict__ out, int d,
                                            float eps, size_t row, float* red) {
  const int nv = d / 4;
  float4 v[VPT];
  float ss = 0.f;
#pragma unroll
  for (int q = 0; q < VPT; ++q) {
    const int c = threadIdx.x + q * NORM_THREADS;
    if (c < nv) {
      if constexpr (IN_BF16) {
        uint2 raw = reinterpret_cast<const uint2*>(static_cast<const uint16_t*>(in) + row * d)[c];
        v[q] = make_float4(__uint_as_float(raw.x << 16), __uint_as_float(raw.x & 0xffff0000u),
                           __uint_as_float(raw.y << 16), __uint_as_float(raw.y & 0xffff0000u));
        reinterpret_cast<float4*>(h32 + row * d)[c] = v[q];
      } else {
        v[q] = reinterpret_cast<const float4*>(static_cast<const float*>(in) + row * d)[c];
      }
      ss += v[q].x * v[q].x + v[q].y * v[q].y + v[q].z * v[q].z + v[q].w * v[q].w;
    }
  }
  const float inv = rsqrtf(block_sum(ss, red) / (float)d + eps);
#pragma unroll
  for (int q = 0; q < VPT; ++q) {
    const int c = threadIdx.x + q * NORM_THREADS;
    if (c < nv) {
      uint2 gr = reinterpret_cast<const uint2*>(gain)[c];
      const float g0 = __uint_as_float(gr.x << 16), g1 = __uint_as_float(gr.x & 0xffff0000u);
      const float g2 = __uint_as_float(gr.y << 16), g3 = __uint_as_float(gr.y & 0xffff0000u);
      uint2 o;
      if constexpr (OUT_F16) {
        o.x = pack_half2(v[q].x * inv * g0, v[q].y * inv * g1);
        o.y = pack_half2(v[q].z * inv * g2, v[q].w * inv * g3);
      } else {
        o.x = pack_bf16x2(v[q].x * inv * g0, v[q].y * inv * g1);
        o.y = pack_bf16x2(v[q].z * inv * g2, v[q].w * inv * g3);
      }
      reinterpret_cast<uint2*>(out + row * d)[c] = o;
    }
  }
}

// y = h / sqrt(mean(h^2) + eps) * g, one row per CTA at a time: rows blockIdx.x, + gridDim.x,
// ... below the row count (rows_dev: a device count clamped to max_rows, or max_rows itself).
// IN_BF16: h is the bf16 packed input, which is also widened into the fp32 residual stream h32.
// OUT_F16: y in fp16 (the GEMM operand); otherwise bf16 (the final hidden states).  VPT: float4
// per thread, the fewest that cover d (4 at d = 4096, 8 at the widest d = 8192), so the row held
// in registers is no larger than the row: fewer registers, more CTAs per SM and more bytes in
// flight.
template <bool IN_BF16, bool OUT_F16, int VPT>
__global__ void __launch_bounds__(NORM_THREADS, VPT <= 4 ? 8 : 4) rmsnorm_kernel(const void* __restrict__ in,
                                                               float* __restrict__ h32,
                                                               const uint16_t* __restrict__ gain,
                                                               uint16_t* __restrict__ out, int d,
                                                               float eps, const int* __restrict__ rows_dev,
                                                               int max_rows) {
  __shared__ float red[32];
  const int n_rows = rows_dev ? max(0, min(max_rows, *rows_dev)) : max_rows;
  for (size_t row = blockIdx.x; row < (size_t)n_rows; row += gridDim.x)
    rmsnorm_row<IN_BF16, OUT_F16, VPT>(in, h32, gain, out, d, eps, row, red);
}

// cos/sin of pos * theta^(-2j/hd), evaluated in double and rounded once to fp32.
__global__ void rope_table_kernel(float2* __restrict__ tab, int max_len, int half, float theta) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= max_len * half) return;
  const int p = i / half, j = i % half;
  const double inv = pow((double)theta, -2.0 * j / (2.0 * half));
  double s, c;
  sincos((double)p * inv, &s, &c);
  tab[i] = make_float2((float)c, (float)s);
}

// KV cache rows: k_out[r] = qkv[r, d .. 2d), v_out[r] = qkv[r, 2d .. 3d) (fp16, heads contiguous),
// for the rows below the device count rows_dev clamped to rows (all rows without one).
__global__ void kv_store_kernel(const uint16_t* __restrict__ qkv, int rows, const int* __restrict__ rows_dev, int d,
                                uint16_t* __restrict__ k_out, uint16_t* __restrict__ v_out) {
  const int nv = d / 8;  // uint4 per row half
  if (rows_dev) rows = max(0, min(rows, *rows_dev));
  const size_t total = (size_t)rows * 2 * nv;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < total; e += (size_t)gridDim.x * blockDim.x) {
    const size_t r = e / (2 * nv);
    const int c = (int)(e % (2 * nv));
    const uint4 v = reinterpret_cast<const uint4*>(qkv + r * 3 * d + d)[c];
    if (c < nv)
      reinterpret_cast<uint4*>(k_out + r * d)[c] = v;
    else
      reinterpret_cast<uint4*>(v_out + r * d)[c - nv] = v;
  }
}

static void kv_store(const uint16_t* qkv, int rows, const int* rows_dev, int d, uint16_t* k_out, uint16_t* v_out,
                     cudaStream_t st) {
  const size_t total = (size_t)rows * (d / 4);
  const int grid = (int)((total + 255) / 256 < 4096 ? (total + 255) / 256 : 4096);
  kv_store_kernel<<<grid, 256, 0, st>>>(qkv, rows, rows_dev, d, k_out, v_out);
}

// Rows T .. T + n_tail - 1 (clamped to the cap rows of the buffer) of an fp16 [cap, cols] buffer
// set to zero, T = *T_dev.  The attention's last query tile and key block may reach up to 127
// rows past the last packed row, and a masked key still meets its value row in the P V product,
// where 0 x NaN = NaN: so the rows past T that the tensor maps can reach must hold finite values
// (with the row count equal to the capacity they are out of bounds and read as zero instead).
__global__ void zero_tail_kernel(uint16_t* __restrict__ buf, int cols, const int* __restrict__ T_dev, int cap,
                                 int n_tail) {
  const int T = max(0, min(cap, *T_dev));
  const int rows = min(n_tail, cap - T);
  const int nv = cols / 8;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < (size_t)rows * nv;
       e += (size_t)gridDim.x * blockDim.x)
    reinterpret_cast<uint4*>(buf + (size_t)(T + e / nv) * cols)[e % nv] = make_uint4(0, 0, 0, 0);
}

// out[i] = h32[cu[i + 1] - 1]: the residual stream of each sequence's last row (zeros for an
// empty sequence, or one that ends past the row_cap rows the buffers hold), for the sequences
// below the device count n_seq_dev (all gridDim.x of them without one).
__global__ void last_rows_kernel(const float* __restrict__ h32, const int* __restrict__ cu,
                                 const int* __restrict__ n_seq_dev, int row_cap, int d, float* __restrict__ out) {
  const int i = blockIdx.x;
  if (n_seq_dev && i >= *n_seq_dev) return;
  const bool empty = cu[i + 1] <= cu[i] || cu[i + 1] > row_cap;
  const float4* src = reinterpret_cast<const float4*>(h32 + (size_t)(empty ? 0 : cu[i + 1] - 1) * d);
  float4* dst = reinterpret_cast<float4*>(out + (size_t)i * d);
  for (int c = threadIdx.x; c < d / 4; c += blockDim.x) dst[c] = empty ? make_float4(0.f, 0.f, 0.f, 0.f) : src[c];
}

PrefillLayout prefill_layout(const rift_model& m, int max_T, int max_seqs, int max_len) {
  PrefillLayout L{};
  size_t off = 0;
  auto take = [&](size_t bytes) { size_t o = off; off += (bytes + 255) & ~size_t(255); return o; };
  const size_t T = (size_t)max_T;
  L.h32_off = take(T * m.d * 4);
  L.xn_off = take(T * m.d * 2);
  L.qkv_off = take(T * 3 * m.d * 2);
  L.attn_off = take(T * m.d * 2);
  L.act_off = take(T * m.ffn * 2);
  L.rope_off = take((size_t)max_len * (m.head_dim / 2) * sizeof(float2));
  L.max_qblocks = attention_max_qblocks(max_T, max_seqs);
  L.sched_off = take((size_t)(L.max_qblocks + 1) * sizeof(int4));  // + the entry count
  L.last32_off = take((size_t)max_seqs * m.d * 4);
  L.last16_off = take((size_t)max_seqs * m.d * 2);
  L.total = off;
  return L;
}

int launch_gemm(const void* A, const void* B, int M, int N, int K, int epi, void* C, cudaStream_t st,
                const EpiParams& ep, void* split_ws, size_t split_ws_bytes, bool pdl) {
  prof_begin(RIFT_PROF_GEMM, st);
  const int r = launch_gemm_tc(A, B, M, N, K, epi, C, ep, st, split_ws, split_ws_bytes, pdl);
  prof_end(RIFT_PROF_GEMM, st, 1);
  return r;
}

static int sm_count() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

// CTAs of rmsnorm_kernel<IN_BF16, OUT_F16, VPT> resident per SM at once (asked once per
// instantiation; 1 if the query fails).
template <bool IN_BF16, bool OUT_F16, int VPT>
static int norm_resident_ctas() {
  static std::atomic<int> n{0};
  int v = n.load(std::memory_order_relaxed);
  if (v == 0) {
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, rmsnorm_kernel<IN_BF16, OUT_F16, VPT>, NORM_THREADS, 0) !=
            cudaSuccess ||
        v < 1) {
      cudaGetLastError();
      v = 1;
    }
    n.store(v, std::memory_order_relaxed);
  }
  return v;
}

// kind 0: packed bf16 input -> h32 + fp16 xn; 1: h32 -> fp16 xn; 2: h32 -> bf16 final output.
// Rows: min(*rows_dev, T) with a device count, else T.  The grid is four times the CTAs that fit
// on the GPU at once (8 per SM at d <= 4096), each looping over rows: a CTA that finishes early
// frees its slot for another, so the last rows spread over the SMs as with one CTA per row.
static void norm_launch(int kind, int T, const void* in, float* h32, const void* gain, uint16_t* out, int d,
                        float eps, cudaStream_t st, const int* rows_dev = nullptr) {
  prof_begin(RIFT_PROF_NORM, st);
  const uint16_t* g = static_cast<const uint16_t*>(gain);
  const int per_thread = (d / 4 + NORM_THREADS - 1) / NORM_THREADS;  // d <= 8192: at most 8
  auto go = [&](auto vpt) {
    constexpr int V = decltype(vpt)::value;
    auto grid = [&](int per_sm) { return T < 4 * per_sm * sm_count() ? T : 4 * per_sm * sm_count(); };
    if (kind == 0)
      rmsnorm_kernel<true, true, V><<<grid(norm_resident_ctas<true, true, V>()), NORM_THREADS, 0, st>>>(
          in, h32, g, out, d, eps, rows_dev, T);
    else if (kind == 1)
      rmsnorm_kernel<false, true, V><<<grid(norm_resident_ctas<false, true, V>()), NORM_THREADS, 0, st>>>(
          in, nullptr, g, out, d, eps, rows_dev, T);
    else
      rmsnorm_kernel<false, false, V><<<grid(norm_resident_ctas<false, false, V>()), NORM_THREADS, 0, st>>>(
          in, nullptr, g, out, d, eps, rows_dev, T);
  };
  if (per_thread <= 1) go(std::integral_constant<int, 1>{});
  else if (per_thread <= 2) go(std::integral_constant<int, 2>{});
  else if (per_thread <= 4) go(std::integral_constant<int, 4>{});
  else go(std::integral_constant<int, 8>{});
  prof_end(RIFT_PROF_NORM, st, 1);
}

int launch_prefill(const rift_model& m, void* hidden, int T, const int* T_dev, const int* cu_seqlens, int n_seq,
                   const int* n_seq_dev, int max_len, const int* positions, void* kv_out, float* last_logits,
                   char* ws, cudaStream_t st, const void* prefix_kv, int S_pre) {
  if (T == 0 || n_seq == 0) return 0;
  const PrefillLayout L = prefill_layout(m, T, n_seq, max_len);
  float* h32 = reinterpret_cast<float*>(ws + L.h32_off);
  uint16_t* xn = reinterpret_cast<uint16_t*>(ws + L.xn_off);
  uint16_t* qkv = reinterpret_cast<uint16_t*>(ws + L.qkv_off);
  uint16_t* att = reinterpret_cast<uint16_t*>(ws + L.attn_off);
  uint16_t* act = reinterpret_cast<uint16_t*>(ws + L.act_off);
  float2* rope = reinterpret_cast<float2*>(ws + L.rope_off);
  int4* sched = reinterpret_cast<int4*>(ws + L.sched_off);
  const int d = m.d, half = m.head_dim / 2;

  prof_begin(RIFT_PROF_ROPE, st);
  rope_table_kernel<<<(max_len * half + 255) / 256, 256, 0, st>>>(rope, max_len, half, m.rope_theta);
  prof_end(RIFT_PROF_ROPE, st, 1);
  prof_begin(RIFT_PROF_ATTN, st);
  launch_attention_schedule(cu_seqlens, n_seq, n_seq_dev, T, sched, L.max_qblocks, st);
  if (T_dev) zero_tail_kernel<<<64, 256, 0, st>>>(qkv, 3 * d, T_dev, T, 128);
  prof_end(RIFT_PROF_ATTN, st, T_dev ? 2 : 1);
  // every product covers the rows the device count holds (T rows of capacity)
  EpiParams rows_ep;
  rows_ep.m_dev = T_dev;
  EpiParams rope_ep = rows_ep;
  rope_ep.positions = positions;
  rope_ep.rope = rope;
  rope_ep.rope_cols = 2 * d;
  rope_ep.head_dim = m.head_dim;
  rope_ep.max_len = max_len;
  rope_ep.pos_offset = S_pre;
  for (int l = 0; l < m.n_layers; ++l) {
    if (l == 0)
      norm_launch(0, T, hidden, h32, m.g_attn[0], xn, d, m.eps, st, T_dev);
    else
      norm_launch(1, T, h32, nullptr, m.g_attn[l], xn, d, m.eps, st, T_dev);
    if (launch_gemm(xn, m.w_qkv[l], T, 3 * d, d, EPI_QKV_ROPE, qkv, st, rope_ep)) return 1;
    if (kv_out) {
      uint16_t* kl = static_cast<uint16_t*>(kv_out) + (size_t)l * 2 * T * d;
      kv_store(qkv, T, T_dev, d, kl, kl + (size_t)T * d, st);
    }
    prof_begin(RIFT_PROF_ATTN, st);
    const uint16_t* pk = prefix_kv ? static_cast<const uint16_t*>(prefix_kv) + (size_t)l * 2 * S_pre * d : nullptr;
    if (launch_attention(qkv, T, cu_seqlens, n_seq, m.n_heads, m.head_dim, sched, L.max_qblocks, att, st, pk,
                         pk ? pk + (size_t)S_pre * d : nullptr, prefix_kv ? S_pre : 0))
      return 1;
    prof_end(RIFT_PROF_ATTN, st, 1);
    if (launch_gemm(att, m.w_o[l], T, d, d, EPI_RESID_F32, h32, st, rows_ep)) return 1;
    norm_launch(1, T, h32, nullptr, m.g_ffn[l], xn, d, m.eps, st, T_dev);
    if (launch_gemm(xn, m.w_gate_up[l], T, 2 * m.ffn, d, EPI_SWIGLU, act, st, rows_ep)) return 1;
    if (launch_gemm(act, m.w_down[l], T, d, m.ffn, EPI_RESID_F32, h32, st, rows_ep)) return 1;
  }
  norm_launch(2, T, h32, nullptr, m.g_final, static_cast<uint16_t*>(hidden), d, m.eps, st, T_dev);
  if (last_logits) {
    float* last32 = reinterpret_cast<float*>(ws + L.last32_off);
    uint16_t* last16 = reinterpret_cast<uint16_t*>(ws + L.last16_off);
    last_rows_kernel<<<n_seq, 256, 0, st>>>(h32, cu_seqlens, n_seq_dev, T, d, last32);
    norm_launch(1, n_seq, last32, nullptr, m.g_final, last16, d, m.eps, st, n_seq_dev);
    EpiParams seq_ep;
    seq_ep.m_dev = n_seq_dev;
    if (launch_gemm(last16, m.lm_head, n_seq, m.vocab, d, EPI_STORE_F32, last_logits, st, seq_ep)) return 1;
  }
  return 0;
}

// ------------------------------------------------------------------------------------------
// Shared-prefix prefill: the system prompt once, then every sequence's suffix over its cache
// ------------------------------------------------------------------------------------------

// prefix rows = embed[sys_ids] (bf16), cu = {0, S}, positions 0 .. S-1; a bad id sets
// RIFT_EBIT_BADID and gives a zero row.
__global__ void prefix_rows_kernel(const int* __restrict__ sys_ids, int S, const uint16_t* __restrict__ embed,
                                   int vocab, int d, uint16_t* __restrict__ rows, int* __restrict__ cu,
                                   int* __restrict__ pos) {
  const int r = blockIdx.x;
  const int id = sys_ids[r];
  const bool ok = id >= 0 && id < vocab;
  if (threadIdx.x == 0) {
    pos[r] = r;
    if (!ok) atomicOr(&g_err_prefill, RIFT_EBIT_BADID);
    if (r == 0) {
      cu[0] = 0;
      cu[1] = S;
    }
  }
  const uint4* src = reinterpret_cast<const uint4*>(embed + (size_t)(ok ? id : 0) * d);
  uint4* dst = reinterpret_cast<uint4*>(rows + (size_t)r * d);
  for (int c = threadIdx.x; c < d / 8; c += blockDim.x) dst[c] = ok ? src[c] : make_uint4(0, 0, 0, 0);
}

SharedPrefixLayout shared_prefix_layout(const rift_model& m, int max_T, int max_seqs, int max_len, int S) {
  SharedPrefixLayout L{};
  const PrefillLayout P = prefill_layout(m, max_T > S ? max_T : S, max_seqs > 1 ? max_seqs : 1, max_len);
  size_t off = (P.total + 255) & ~size_t(255);
  L.prefill_bytes = P.total;
  L.cu_off = off;
  off += 256;
  L.pos_off = off;
  off += ((size_t)S * sizeof(int) + 255) & ~size_t(255);
  L.total = off;
  return L;
}

int launch_prefill_shared_prefix(const rift_model& m, const int* sys_ids, int S, const void* embed, int vocab,
                                 void* prefix_hidden, void* prefix_kv, void* hidden, int T, const int* T_dev,
                                 const int* cu_seqlens, int n_seq, const int* n_seq_dev, int max_len,
                                 const int* positions, float* last_logits, char* ws, cudaStream_t st) {
  const SharedPrefixLayout L = shared_prefix_layout(m, T, n_seq, max_len, S);
  int* cu_pre = reinterpret_cast<int*>(ws + L.cu_off);
  int* pos_pre = reinterpret_cast<int*>(ws + L.pos_off);
  prefix_rows_kernel<<<S, 128, 0, st>>>(sys_ids, S, static_cast<const uint16_t*>(embed), vocab, m.d,
                                        static_cast<uint16_t*>(prefix_hidden), cu_pre, pos_pre);
  // the prefix as one sequence, keeping its cache; then the suffixes over it (the two share the
  // prefill workspace: they run in order on the stream)
  if (launch_prefill(m, prefix_hidden, S, nullptr, cu_pre, 1, nullptr, max_len, pos_pre, prefix_kv, nullptr, ws, st))
    return 1;
  if (T > 0 && launch_prefill(m, hidden, T, T_dev, cu_seqlens, n_seq, n_seq_dev, max_len, positions, nullptr,
                              last_logits, ws, st, prefix_kv, S))
    return 1;
  return 0;
}

// ------------------------------------------------------------------------------------------
// Decode step: one new token per sequence
// ------------------------------------------------------------------------------------------

constexpr int DEC_CHUNK = 128;  // keys per decode-attention work unit
constexpr int DEC_HG = 8;       // heads per decode-attention CTA (one warp each)

DecodeLayout decode_layout(const rift_model& m, int n_seq, int max_len) {
  DecodeLayout L{};
  size_t off = 0;
  auto take = [&](size_t bytes) { size_t o = off; off += (bytes + 255) & ~size_t(255); return o; };
  const size_t n = (size_t)(n_seq > 0 ? n_seq : 1);
  L.h32_off = take(n * m.d * 4);
  L.x0_off = take(n * m.d * 2);
  L.xn_off = take(n * m.d * 2);
  L.qkv_off = take(n * 3 * m.d * 2);
  L.attn_off = take(n * m.d * 2);
  L.act_off = take(n * m.ffn * 2);
  L.rope_off = take((size_t)max_len * (m.head_dim / 2) * sizeof(float2));
  L.pos_off = take(n * sizeof(int));
  // decode attention partials: (m, l, o[head_dim]) per (sequence, key chunk, head)
  L.dpart_off = take(n * (size_t)((max_len + DEC_CHUNK - 1) / DEC_CHUNK) * m.n_heads * (m.head_dim + 2) * 4);
  // split-K partial products of the few-row GEMMs: up to 16 slices of [min(n, 128), widest
  // output] fp32, at most 128 MB
  const size_t rows = n < 128 ? n : 128;
  size_t widest = (size_t)3 * m.d;
  if ((size_t)2 * m.ffn > widest) widest = (size_t)2 * m.ffn;
  if (m.lm_head && (size_t)m.vocab > widest) widest = (size_t)m.vocab;
  L.split_bytes = 16 * rows * widest * 4;
  if (L.split_bytes > (size_t)128 << 20) L.split_bytes = (size_t)128 << 20;
  // at least one slice of the residual products, which always go through the scratch
  if (L.split_bytes < n * m.d * 4) L.split_bytes = n * m.d * 4;
  L.split_off = take(L.split_bytes);
  L.total = off;
  return L;
}

// x0[i] = embed[ids[i]] (bf16) and pos[i] = L_i = cu[i + 1] - cu[i], the new token's position.
// An id outside [0, vocab) sets RIFT_EBIT_BADID and gives a zero row.
__global__ void decode_embed_kernel(const int* __restrict__ ids, const int* __restrict__ cu,
                                    const uint16_t* __restrict__ embed, int vocab, int d,
                                    uint16_t* __restrict__ x0, int* __restrict__ pos) {
  const int i = blockIdx.x;
  const int id = ids[i];
  const bool ok = id >= 0 && id < vocab;
  if (threadIdx.x == 0) {
    pos[i] = cu[i + 1] - cu[i];
    if (!ok) atomicOr(&g_err_prefill, RIFT_EBIT_BADID);
  }
  uint4* dst = reinterpret_cast<uint4*>(x0 + (size_t)i * d);
  const uint4* src = reinterpret_cast<const uint4*>(embed + (size_t)(ok ? id : 0) * d);
  for (int c = threadIdx.x; c < d / 8; c += blockDim.x) dst[c] = ok ? src[c] : make_uint4(0, 0, 0, 0);
}


// Attention of each sequence's new token over its P = L_i cached rows and itself, split like
// flash decoding: CTA (sequence i, chunk c of DEC_CHUNK keys, group of hg heads: the largest of
// 8, 4, 2, 1 that divides H), one warp per head.  A key row's hg head slices are hg * head_dim * 2
// contiguous bytes, read together by the CTA's warps.  Lanes read 16 bytes (8 head dims) each, so
// one warp-wide load covers KPL = 256 / head_dim keys, LPK = head_dim / 8 lanes per key; each
// lane group keeps its own running maximum m, sum l and output o over its keys (online softmax,
// fp32, log2 units) and the groups are merged at the end of the chunk.  (m, l, o) of the chunk go
// to `part`, and decode_combine_kernel merges a sequence's chunks.  Units past a sequence's last
// key exit at once.
template <int HD>
__global__ void __launch_bounds__(DEC_HG * 32, 3) decode_attn_kernel(const uint16_t* __restrict__ qkv,
                                                                     const uint16_t* __restrict__ Kc,
                                                                     const uint16_t* __restrict__ Vc,
                                                                     const int* __restrict__ cu, int H, int hg,
                                                                     int max_chunks, float scale_log2,
                                                                     float* __restrict__ part) {
  pdl_trigger();
  pdl_wait();
  constexpr int LPK = HD / 8, KPL = 32 / LPK;  // lanes per key, keys per warp-wide load
  constexpr int NL = 4;                        // warp-wide loads of K (and of V) in flight
  const int groups = H / hg;  // hg = blockDim.x / 32 heads per CTA
  const int g = blockIdx.x % groups, c = (blockIdx.x / groups) % max_chunks, i = blockIdx.x / (groups * max_chunks);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = g * hg + warp;
  const int d = H * HD;
  const int s0 = cu[i], P = cu[i + 1] - s0, nk = P + 1;
  const int j_begin = c * DEC_CHUNK, j_end = min(nk, j_begin + DEC_CHUNK);
  if (j_begin >= nk) return;
  const int sub = lane / LPK, dl = (lane % LPK) * 8;  // key within a load, first head dim of the lane
  const uint16_t* self = qkv + (size_t)i * 3 * d + h * HD;  // q, then k at + d, v at + 2d
  auto unpack = [](const uint4& u, float (&x)[8]) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w[e]));
      x[2 * e] = f.x;
      x[2 * e + 1] = f.y;
    }
  };
  float q[8];
  unpack(__ldg(reinterpret_cast<const uint4*>(self + dl)), q);
#pragma unroll
  for (int e = 0; e < 8; ++e) q[e] *= scale_log2;  // scores in log2 units
  float m = -INFINITY, l = 0.f, acc[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) acc[e] = 0.f;
  for (int j0 = j_begin; j0 < j_end; j0 += NL * KPL) {
    uint4 kr[NL], vr[NL];
#pragma unroll
    for (int u = 0; u < NL; ++u) {  // rows past the chunk end read the last row, weight 0
      const int j = min(j0 + u * KPL + sub, j_end - 1);
      const size_t r = (size_t)(s0 + j) * d + h * HD + dl;
      kr[u] = __ldg(reinterpret_cast<const uint4*>(j < P ? Kc + r : self + d + dl));
      vr[u] = __ldg(reinterpret_cast<const uint4*>(j < P ? Vc + r : self + 2 * d + dl));
    }
    float sc[NL];
#pragma unroll
    for (int u = 0; u < NL; ++u) {
      float kx[8];
      unpack(kr[u], kx);
      float dot = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) dot = fmaf(q[e], kx[e], dot);
#pragma unroll
      for (int o = LPK / 2; o >= 1; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
      sc[u] = (j0 + u * KPL + sub < j_end) ? dot : -INFINITY;
    }
    float mx = m;
#pragma unroll
    for (int u = 0; u < NL; ++u) mx = fmaxf(mx, sc[u]);
    // a lane group whose keys are all past the end keeps m = -inf (mx = -inf): nothing to add
    const float corr = mx == -INFINITY ? 1.f : exp2f(m - mx);
    l *= corr;
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] *= corr;
#pragma unroll
    for (int u = 0; u < NL; ++u) {
      const float p = mx == -INFINITY ? 0.f : exp2f(sc[u] - mx);
      float vx[8];
      unpack(vr[u], vx);
      l += p;
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] = fmaf(p, vx[e], acc[e]);
    }
    m = mx;
  }
  // merge the KPL lane groups (lanes l, l + LPK, ... hold the same head dims)
#pragma unroll
  for (int o = LPK; o < 32; o <<= 1) {
    const float mo = __shfl_xor_sync(0xffffffffu, m, o), lo = __shfl_xor_sync(0xffffffffu, l, o);
    const float M = fmaxf(m, mo);
    const float fa = m == -INFINITY ? 0.f : exp2f(m - M), fb = mo == -INFINITY ? 0.f : exp2f(mo - M);
    l = l * fa + lo * fb;
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = acc[e] * fa + __shfl_xor_sync(0xffffffffu, acc[e], o) * fb;
    m = M;
  }
  float* dst = part + (((size_t)i * max_chunks + c) * H + h) * (HD + 2);
  if (lane == 0) {
    dst[0] = m;
    dst[1] = l;
  }
  if (lane < LPK) {
#pragma unroll
    for (int e = 0; e < 8; ++e) dst[2 + dl + e] = acc[e];
  }
}

// out[i, h] = sum_c o_c 2^(m_c - M) / sum_c l_c 2^(m_c - M), chunks in order (M = max_c m_c).
// A sequence with more than max_keys keys sets RIFT_EBIT_CAPACITY and gets zeros.
__global__ void decode_combine_kernel(const float* __restrict__ part, const int* __restrict__ cu, int H, int HD,
                                      int max_chunks, int max_keys, uint16_t* __restrict__ out) {
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x / H, h = blockIdx.x % H;
  const int nk = cu[i + 1] - cu[i] + 1;
  uint16_t* o = out + ((size_t)i * H + h) * HD;
  if (nk > max_keys) {
    if (threadIdx.x == 0) atomicOr(&g_err_prefill, RIFT_EBIT_CAPACITY);
    for (int e = threadIdx.x; e < HD; e += blockDim.x) o[e] = 0;
    return;
  }
  const int nch = (nk + DEC_CHUNK - 1) / DEC_CHUNK;
  const float* p0 = part + ((size_t)i * max_chunks * H + h) * (HD + 2);
  const size_t cstride = (size_t)H * (HD + 2);
  float M = -INFINITY;
  for (int c = 0; c < nch; ++c) M = fmaxf(M, p0[c * cstride]);
  for (int e = threadIdx.x; e < HD; e += blockDim.x) {
    float L = 0.f, v = 0.f;
    for (int c = 0; c < nch; ++c) {
      const float* pc = p0 + c * cstride;
      const float f = exp2f(pc[0] - M);
      L += pc[1] * f;
      v += pc[2 + e] * f;
    }
    o[e] = __half_as_ushort(__float2half_rn(v / L));
  }
}

int launch_decode(const rift_model& m, const void* kv_cache, int T, const int* cu_seqlens, int n_seq, int max_len,
                  const int* token_ids, const void* embed, int vocab_embed, void* hidden_out, void* kv_new,
                  float* logits, char* ws, cudaStream_t st) {
  if (n_seq == 0) return 0;
  const DecodeLayout L = decode_layout(m, n_seq, max_len);
  float* h32 = reinterpret_cast<float*>(ws + L.h32_off);
  uint16_t* x0 = reinterpret_cast<uint16_t*>(ws + L.x0_off);
  uint16_t* xn = reinterpret_cast<uint16_t*>(ws + L.xn_off);
  uint16_t* qkv = reinterpret_cast<uint16_t*>(ws + L.qkv_off);
  uint16_t* att = reinterpret_cast<uint16_t*>(ws + L.attn_off);
  uint16_t* act = reinterpret_cast<uint16_t*>(ws + L.act_off);
  float2* rope = reinterpret_cast<float2*>(ws + L.rope_off);
  int* pos = reinterpret_cast<int*>(ws + L.pos_off);
  void* split = ws + L.split_off;
  const size_t sb = L.split_bytes;
  float* dpart = reinterpret_cast<float*>(ws + L.dpart_off);
  const int max_chunks = (max_len + DEC_CHUNK - 1) / DEC_CHUNK;
  int hg = DEC_HG;
  while (m.n_heads % hg != 0) hg /= 2;
  const int d = m.d, half = m.head_dim / 2, n = n_seq;

  rope_table_kernel<<<(max_len * half + 255) / 256, 256, 0, st>>>(rope, max_len, half, m.rope_theta);
  decode_embed_kernel<<<n, 128, 0, st>>>(token_ids, cu_seqlens, static_cast<const uint16_t*>(embed), vocab_embed, d,
                                         x0, pos);
  EpiParams rope_ep;
  rope_ep.positions = pos;
  rope_ep.rope = rope;
  rope_ep.rope_cols = 2 * d;
  rope_ep.head_dim = m.head_dim;
  rope_ep.max_len = max_len;
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)m.head_dim);
  const uint16_t* kv = static_cast<const uint16_t*>(kv_cache);
  // The residual products carry the RMSNorm that follows them (g_ffn after W_o; the next layer's
  // g_attn, or g_final after the last W_down) into their split-K reduction.
  auto resid_norm = [&](const void* gain) {
    EpiParams e;
    e.norm_gain = gain;
    e.norm_out = xn;
    e.norm_eps = m.eps;
    return e;
  };
  norm_launch(0, n, x0, h32, m.g_attn[0], xn, d, m.eps, st);
  // The layer's kernels are launched as programmatic dependents of the kernel before them: each
  // starts while its predecessor drains (the GEMMs already streaming their first weight tiles)
  // and waits for it before touching activations.
  const bool pdl = true;
  for (int l = 0; l < m.n_layers; ++l) {
    if (launch_gemm(xn, m.w_qkv[l], n, 3 * d, d, EPI_QKV_ROPE, qkv, st, rope_ep, split, sb, pdl)) return 1;
    if (kv_new) {
      uint16_t* kl = static_cast<uint16_t*>(kv_new) + (size_t)l * 2 * n * d;
      kv_store(qkv, n, nullptr, d, kl, kl + (size_t)n * d, st);
    }
    const uint16_t* Kc = kv + (size_t)l * 2 * T * d;
    const uint16_t* Vc = Kc + (size_t)T * d;
    prof_begin(RIFT_PROF_ATTN, st);
    const int units = n * max_chunks * (m.n_heads / hg);
    cudaError_t e;
    if (m.head_dim == 128)
      e = launch_ex(decode_attn_kernel<128>, dim3(units), dim3(hg * 32), 0, st, pdl, (const uint16_t*)qkv, Kc, Vc,
                    cu_seqlens, (int)m.n_heads, hg, max_chunks, scale_log2, dpart);
    else
      e = launch_ex(decode_attn_kernel<64>, dim3(units), dim3(hg * 32), 0, st, pdl, (const uint16_t*)qkv, Kc, Vc,
                    cu_seqlens, (int)m.n_heads, hg, max_chunks, scale_log2, dpart);
    if (e != cudaSuccess) return 1;
    if (launch_ex(decode_combine_kernel, dim3(n * m.n_heads), dim3(m.head_dim), 0, st, pdl, (const float*)dpart,
                  cu_seqlens, (int)m.n_heads, (int)m.head_dim, max_chunks, max_len, att) != cudaSuccess)
      return 1;
    prof_end(RIFT_PROF_ATTN, st, 2);
    if (launch_gemm(att, m.w_o[l], n, d, d, EPI_RESID_F32, h32, st, resid_norm(m.g_ffn[l]), split, sb, pdl)) return 1;
    if (launch_gemm(xn, m.w_gate_up[l], n, 2 * m.ffn, d, EPI_SWIGLU, act, st, EpiParams(), split, sb, pdl)) return 1;
    const void* next_gain = l + 1 < m.n_layers ? m.g_attn[l + 1] : m.g_final;
    if (launch_gemm(act, m.w_down[l], n, d, m.ffn, EPI_RESID_F32, h32, st, resid_norm(next_gain), split, sb, pdl))
      return 1;
  }
  // xn now holds RMSNorm(h) g_final in fp16 (the logits operand)
  if (hidden_out) norm_launch(2, n, h32, nullptr, m.g_final, static_cast<uint16_t*>(hidden_out), d, m.eps, st);
  if (logits) {
    if (launch_gemm(xn, m.lm_head, n, m.vocab, d, EPI_STORE_F32, logits, st, EpiParams(), split, sb, pdl)) return 1;
  }
  return 0;
}

}  // namespace rift
