// Varlen causal attention over the packed per-tile sequences (sm_103a, warp-level tensor
// path).  Each packed sequence attends only to itself; the q-block schedule is built on the
// device from cu_seqlens so the launch needs no host-side lengths.
//
// CTA = (q-block of 64 rows of one sequence, one head), 4 warps x 16 query rows.  K/V tiles
// of 64 keys are double-buffered through shared memory with cp.async; S = Q K^T and O = P V
// run on mma.sync m16n8k16 (fp16 in, fp32 accumulate) with an online softmax in fp32 (exp2,
// scale folded with log2 e).  P is re-used from the S accumulators as the A operand (fp16).
#include "rift_internal.h"

namespace rift {

namespace attn {

constexpr int BQ = 64, BKV = 64, THREADS = 128;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool pred) {
  const int n = pred ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(n));
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void mma_f16(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// One entry per 64-row q-block: (sequence, first row within the sequence); the rest are
// (-1, 0).  One CTA scans the sequence lengths.
__global__ void __launch_bounds__(1024) schedule_kernel(const int* __restrict__ cu, int n_seq,
                                                        int2* __restrict__ sched, int n_max) {
  __shared__ int sh[33];
  int base = 0;
  for (int c0 = 0; c0 < n_seq; c0 += blockDim.x) {
    const int s = c0 + threadIdx.x;
    int nb = 0;
    if (s < n_seq) nb = (cu[s + 1] - cu[s] + BQ - 1) / BQ;
    int total;
    int off = block_excl_scan(nb, sh, &total);
    for (int b = 0; b < nb; ++b)
      if (base + off + b < n_max) sched[base + off + b] = make_int2(s, b * BQ);
    base += total;
  }
  for (int i = base + threadIdx.x; i < n_max; i += blockDim.x) sched[i] = make_int2(-1, 0);
}

template <int HD>
__global__ void __launch_bounds__(THREADS) attn_kernel(const uint16_t* __restrict__ qkv,
                                                       const int* __restrict__ cu,
                                                       const int2* __restrict__ sched, int H,
                                                       float scale_log2, uint16_t* __restrict__ out) {
  constexpr int LD = HD + 8;  // padded rows: conflict-free ldmatrix
  constexpr int NV = HD / 8;  // 16-byte chunks per row
  extern __shared__ __align__(128) uint16_t sm[];
  uint16_t* Qs = sm;                     // [BQ][LD]
  uint16_t* Ks = Qs + BQ * LD;           // [2][BKV][LD]
  uint16_t* Vs = Ks + 2 * BKV * LD;      // [2][BKV][LD]

  const int2 job = sched[blockIdx.x];
  if (job.x < 0) return;
  const int h = blockIdx.y;
  const int seq0 = cu[job.x];
  const int L = cu[job.x + 1] - seq0;
  const int q0 = job.y;
  const int d = H * HD;
  const size_t rs = 3 * (size_t)d;  // qkv row stride
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  // Q tile
  for (int c = tid; c < BQ * NV; c += THREADS) {
    const int r = c / NV, v = c % NV;
    const bool ok = q0 + r < L;
    const uint16_t* src = qkv + (size_t)(seq0 + (ok ? q0 + r : 0)) * rs + h * HD + v * 8;
    cp_async16(smem_u32(Qs + r * LD + v * 8), src, ok);
  }
  auto load_kv = [&](int buf, int k0) {
    for (int c = tid; c < BKV * NV; c += THREADS) {
      const int r = c / NV, v = c % NV;
      const bool ok = k0 + r < L;
      const size_t row = (size_t)(seq0 + (ok ? k0 + r : 0)) * rs;
      cp_async16(smem_u32(Ks + (buf * BKV + r) * LD + v * 8), qkv + row + d + h * HD + v * 8, ok);
      cp_async16(smem_u32(Vs + (buf * BKV + r) * LD + v * 8), qkv + row + 2 * d + h * HD + v * 8, ok);
    }
  };
  load_kv(0, 0);
  asm volatile("cp.async.commit_group;\n");

  const int q_last = min(L, q0 + BQ) - 1;        // last query row of this block
  const int n_kv = q_last / BKV + 1;              // causal: key blocks 0 .. n_kv-1
  uint32_t qf[HD / 16][4];
  float o[HD / 8][4];
#pragma unroll
  for (int j = 0; j < HD / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  float m_r[2] = {-INFINITY, -INFINITY}, l_r[2] = {0.f, 0.f};
  const int g = lane >> 2, c2 = (lane & 3) * 2;
  const int qrow0 = q0 + warp * 16 + g;  // this thread's rows: qrow0 and qrow0 + 8

  for (int kb = 0; kb < n_kv; ++kb) {
    const int buf = kb & 1;
    if (kb + 1 < n_kv) load_kv(buf ^ 1, (kb + 1) * BKV);
    asm volatile("cp.async.commit_group;\n");
    asm volatile("cp.async.wait_group 1;\n");
    __syncthreads();
    if (kb == 0) {
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk) {
        const int row = warp * 16 + (lane & 15);
        const int col = kk * 16 + (lane >> 4) * 8;
        ldsm_x4(smem_u32(Qs + row * LD + col), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
      }
    }
    // S = Q K^T  (16 x 64 per warp)
    float s[BKV / 8][4];
#pragma unroll
    for (int j = 0; j < BKV / 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int jp = 0; jp < BKV / 16; ++jp) {
        const int row = jp * 16 + (lane & 7) + ((lane >> 4) << 3);
        const int col = kk * 16 + ((lane >> 3) & 1) * 8;
        uint32_t r0, r1, r2, r3;
        ldsm_x4(smem_u32(Ks + (buf * BKV + row) * LD + col), r0, r1, r2, r3);
        mma_f16(s[2 * jp], qf[kk], r0, r1);
        mma_f16(s[2 * jp + 1], qf[kk], r2, r3);
      }
    }
    // mask (causal + sequence end), online softmax
    const int k0 = kb * BKV;
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int j = 0; j < BKV / 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = k0 + j * 8 + c2 + (e & 1);
        const int qr = qrow0 + (e >> 1) * 8;
        float v = s[j][e] * scale_log2;
        if (key > qr || key >= L) v = -INFINITY;
        s[j][e] = v;
        mx[e >> 1] = fmaxf(mx[e >> 1], v);
      }
    }
    float corr[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
      const float mn = fmaxf(m_r[r], mx[r]);
      // rows past the sequence end see only -inf; keep them finite
      const float base = (mn == -INFINITY) ? 0.f : mn;
      corr[r] = exp2f(m_r[r] - base);
      m_r[r] = mn;
      mx[r] = base;
    }
    float rsum[2] = {0.f, 0.f};
    uint32_t pf[BKV / 16][4];
#pragma unroll
    for (int j = 0; j < BKV / 8; ++j) {
      const float p0 = exp2f(s[j][0] - mx[0]), p1 = exp2f(s[j][1] - mx[0]);
      const float p2 = exp2f(s[j][2] - mx[1]), p3 = exp2f(s[j][3] - mx[1]);
      rsum[0] += p0 + p1;
      rsum[1] += p2 + p3;
      pf[j >> 1][(j & 1) * 2 + 0] = pack_half2(p0, p1);
      pf[j >> 1][(j & 1) * 2 + 1] = pack_half2(p2, p3);
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      rsum[r] += __shfl_xor_sync(0xffffffffu, rsum[r], 1);
      rsum[r] += __shfl_xor_sync(0xffffffffu, rsum[r], 2);
      l_r[r] = l_r[r] * corr[r] + rsum[r];
    }
#pragma unroll
    for (int j = 0; j < HD / 8; ++j) {
      o[j][0] *= corr[0]; o[j][1] *= corr[0];
      o[j][2] *= corr[1]; o[j][3] *= corr[1];
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < BKV / 16; ++kk) {
      // A fragment of P for keys 16kk..16kk+15: n-tiles 2kk (a0,a1) and 2kk+1 (a2,a3)
      uint32_t a[4] = {pf[kk][0], pf[kk][1], pf[kk][2], pf[kk][3]};
#pragma unroll
      for (int jp = 0; jp < HD / 16; ++jp) {
        const int row = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int col = jp * 16 + (lane >> 4) * 8;
        uint32_t r0, r1, r2, r3;
        ldsm_x4_t(smem_u32(Vs + (buf * BKV + row) * LD + col), r0, r1, r2, r3);
        mma_f16(o[2 * jp], a, r0, r1);
        mma_f16(o[2 * jp + 1], a, r2, r3);
      }
    }
    __syncthreads();  // the buffer is refilled two iterations later
  }
  asm volatile("cp.async.wait_group 0;\n");
  // normalise and store
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int qr = qrow0 + r * 8;
    if (qr >= L) continue;
    const float inv = 1.f / l_r[r];
    uint16_t* dst = out + (size_t)(seq0 + qr) * d + h * HD;
#pragma unroll
    for (int j = 0; j < HD / 8; ++j)
      *reinterpret_cast<uint32_t*>(dst + j * 8 + c2) = pack_half2(o[j][2 * r] * inv, o[j][2 * r + 1] * inv);
  }
}

}  // namespace attn

void launch_attention_schedule(const int* cu_seqlens, int n_seq, int2* sched, int n_sched_max, cudaStream_t st) {
  attn::schedule_kernel<<<1, 1024, 0, st>>>(cu_seqlens, n_seq, sched, n_sched_max);
}

void launch_attention(const void* qkv, int T, const int* cu_seqlens, int n_seq, int n_heads,
                      int head_dim, const int2* sched, int n_sched_max, void* out, cudaStream_t st) {
  using namespace attn;
  (void)T;
  (void)n_seq;
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)head_dim);
  dim3 grid(n_sched_max, n_heads);
  if (head_dim == 128) {
    const size_t smem = (size_t)(BQ + 4 * BKV) * (128 + 8) * 2;
    cudaFuncSetAttribute(attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    attn_kernel<128><<<grid, THREADS, smem, st>>>(static_cast<const uint16_t*>(qkv), cu_seqlens, sched,
                                                  n_heads, scale_log2, static_cast<uint16_t*>(out));
  } else {
    const size_t smem = (size_t)(BQ + 4 * BKV) * (64 + 8) * 2;
    cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    attn_kernel<64><<<grid, THREADS, smem, st>>>(static_cast<const uint16_t*>(qkv), cu_seqlens, sched,
                                                 n_heads, scale_log2, static_cast<uint16_t*>(out));
  }
}

}  // namespace rift
