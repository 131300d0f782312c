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
// and finally hidden = RMSNorm(h) g_final in bf16.
// fp16 rather than bf16 operands: after 32 layers the bf16 rounding of the GEMM inputs alone
// moves the final hidden states by about 3% of their largest magnitude; fp16 (3 more mantissa
// bits, same tensor-core rate, LLaVA-1.5-7B's checkpoint dtype) keeps the whole path near 0.5%.
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
constexpr int NORM_MAXV = 8;  // float4 per thread: d <= 8192

// y = h / sqrt(mean(h^2) + eps) * g, one CTA per row.  IN_BF16: h is the bf16 packed input,
// which is also widened into the fp32 residual stream h32.  OUT_F16: y in fp16 (the GEMM
// operand); otherwise bf16 (the final hidden states).
template <bool IN_BF16, bool OUT_F16>
__global__ void __launch_bounds__(NORM_THREADS) rmsnorm_kernel(const void* __restrict__ in,
                                                               float* __restrict__ h32,
                                                               const uint16_t* __restrict__ gain,
                                                               uint16_t* __restrict__ out, int d,
                                                               float eps) {
  __shared__ float red[32];
  const size_t row = blockIdx.x;
  const int nv = d / 4;
  float4 v[NORM_MAXV];
  float ss = 0.f;
#pragma unroll
  for (int q = 0; q < NORM_MAXV; ++q) {
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
  for (int q = 0; q < NORM_MAXV; ++q) {
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
  L.sched_off = take((size_t)L.max_qblocks * sizeof(int2));
  L.total = off;
  return L;
}

int launch_gemm(const void* A, const void* B, int M, int N, int K, int epi, void* C, cudaStream_t st,
                const EpiParams& ep) {
  prof_begin(RIFT_PROF_GEMM, st);
  const int r = launch_gemm_tc(A, B, M, N, K, epi, C, ep, st);
  prof_end(RIFT_PROF_GEMM, st, 1);
  return r;
}

// kind 0: packed bf16 input -> h32 + fp16 xn; 1: h32 -> fp16 xn; 2: h32 -> bf16 final output.
static void norm_launch(int kind, int T, const void* in, float* h32, const void* gain, uint16_t* out, int d,
                        float eps, cudaStream_t st) {
  prof_begin(RIFT_PROF_NORM, st);
  const uint16_t* g = static_cast<const uint16_t*>(gain);
  if (kind == 0)
    rmsnorm_kernel<true, true><<<T, NORM_THREADS, 0, st>>>(in, h32, g, out, d, eps);
  else if (kind == 1)
    rmsnorm_kernel<false, true><<<T, NORM_THREADS, 0, st>>>(in, nullptr, g, out, d, eps);
  else
    rmsnorm_kernel<false, false><<<T, NORM_THREADS, 0, st>>>(in, nullptr, g, out, d, eps);
  prof_end(RIFT_PROF_NORM, st, 1);
}

int launch_prefill(const rift_model& m, void* hidden, int T, const int* cu_seqlens, int n_seq,
                   int max_len, const int* positions, char* ws, cudaStream_t st) {
  if (T == 0) return 0;
  const PrefillLayout L = prefill_layout(m, T, n_seq, max_len);
  float* h32 = reinterpret_cast<float*>(ws + L.h32_off);
  uint16_t* xn = reinterpret_cast<uint16_t*>(ws + L.xn_off);
  uint16_t* qkv = reinterpret_cast<uint16_t*>(ws + L.qkv_off);
  uint16_t* att = reinterpret_cast<uint16_t*>(ws + L.attn_off);
  uint16_t* act = reinterpret_cast<uint16_t*>(ws + L.act_off);
  float2* rope = reinterpret_cast<float2*>(ws + L.rope_off);
  int2* sched = reinterpret_cast<int2*>(ws + L.sched_off);
  const int d = m.d, half = m.head_dim / 2;

  prof_begin(RIFT_PROF_ROPE, st);
  rope_table_kernel<<<(max_len * half + 255) / 256, 256, 0, st>>>(rope, max_len, half, m.rope_theta);
  prof_end(RIFT_PROF_ROPE, st, 1);
  prof_begin(RIFT_PROF_ATTN, st);
  launch_attention_schedule(cu_seqlens, n_seq, sched, L.max_qblocks, st);
  prof_end(RIFT_PROF_ATTN, st, 1);
  EpiParams rope_ep;
  rope_ep.positions = positions;
  rope_ep.rope = rope;
  rope_ep.rope_cols = 2 * d;
  rope_ep.head_dim = m.head_dim;
  rope_ep.max_len = max_len;
  for (int l = 0; l < m.n_layers; ++l) {
    if (l == 0)
      norm_launch(0, T, hidden, h32, m.g_attn[0], xn, d, m.eps, st);
    else
      norm_launch(1, T, h32, nullptr, m.g_attn[l], xn, d, m.eps, st);
    if (launch_gemm(xn, m.w_qkv[l], T, 3 * d, d, EPI_QKV_ROPE, qkv, st, rope_ep)) return 1;
    prof_begin(RIFT_PROF_ATTN, st);
    if (launch_attention(qkv, T, cu_seqlens, n_seq, m.n_heads, m.head_dim, sched, L.max_qblocks, att, st)) return 1;
    prof_end(RIFT_PROF_ATTN, st, 1);
    if (launch_gemm(att, m.w_o[l], T, d, d, EPI_RESID_F32, h32, st)) return 1;
    norm_launch(1, T, h32, nullptr, m.g_ffn[l], xn, d, m.eps, st);
    if (launch_gemm(xn, m.w_gate_up[l], T, 2 * m.ffn, d, EPI_SWIGLU, act, st)) return 1;
    if (launch_gemm(act, m.w_down[l], T, d, m.ffn, EPI_RESID_F32, h32, st)) return 1;
  }
  norm_launch(2, T, h32, nullptr, m.g_final, static_cast<uint16_t*>(hidden), d, m.eps, st);
  return 0;
}

}  // namespace rift
