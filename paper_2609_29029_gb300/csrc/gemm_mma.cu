// Reference-grade bf16 GEMM on the warp-level tensor path (mma.sync m16n8k16), used for the
// shapes the tcgen05 kernel does not take (K or N tails) and as its cross-check.
//
// C[M, N] = A[M, K] . B[N, K]^T, both operands K-major, fp32 accumulation, fused epilogues:
// bf16 store, fp32 residual add, or SwiGLU over 16-column gate/up groups.
// 128 x 128 x 32 CTA tile, 8 warps (2 x 4, 64 x 32 each), 4-stage cp.async pipeline,
// zero-filled tails; CTAs are rasterised in bands of 16 M-tiles so a band's A rows stay in L2
// while the weight tiles stream past.
#include "rift_internal.h"

namespace rift {

namespace mma_gemm {

constexpr int BM = 128, BN = 128, BK = 32, STAGES = 4, THREADS = 256;
constexpr int LDS = BK + 8;  // padded row (80 bytes): conflict-free ldmatrix
constexpr int GROUP_M = 16;
constexpr size_t SMEM = (size_t)STAGES * (BM + BN) * LDS * 2;

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

__device__ __forceinline__ void mma_bf16(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ float silu(float g) { return g / (1.f + expf(-g)); }

template <int EPI>
__global__ void __launch_bounds__(THREADS) gemm_kernel(const uint16_t* __restrict__ A,
                                                       const uint16_t* __restrict__ B, int M, int N,
                                                       int K, void* __restrict__ Cv) {
  extern __shared__ __align__(128) uint16_t smem[];
  uint16_t* As = smem;
  uint16_t* Bs = smem + STAGES * BM * LDS;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int wm = warp >> 2, wn = warp & 3;

  // grouped rasterisation
  const int mt = (M + BM - 1) / BM, nt = (N + BN - 1) / BN;
  const int bid = blockIdx.x;
  const int per_group = GROUP_M * nt;
  const int grp = bid / per_group;
  const int first_m = grp * GROUP_M;
  const int gsz = min(mt - first_m, GROUP_M);
  const int m_blk = first_m + (bid % per_group) % gsz;
  const int n_blk = (bid % per_group) / gsz;
  const int m0 = m_blk * BM, n0 = n_blk * BN;

  const int KT = (K + BK - 1) / BK;
  auto load_tile = [&](int stage, int kt) {
    const int k0 = kt * BK;
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int c = tid + q * THREADS;  // 512 chunks of 16 bytes per operand
      const int row = c >> 2, kc = (c & 3) * 8;
      const int gk = k0 + kc;
      {
        const int gr = m0 + row;
        const bool ok = gr < M && gk < K;
        const uint16_t* src = ok ? A + (size_t)gr * K + gk : A;
        cp_async16(smem_u32(As + (stage * BM + row) * LDS + kc), src, ok);
      }
      {
        const int gr = n0 + row;
        const bool ok = gr < N && gk < K;
        const uint16_t* src = ok ? B + (size_t)gr * K + gk : B;
        cp_async16(smem_u32(Bs + (stage * BN + row) * LDS + kc), src, ok);
      }
    }
  };

  float acc[4][4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[i][j][e] = 0.f;

#pragma unroll
  for (int s = 0; s < STAGES - 1; ++s) {
    if (s < KT) load_tile(s, s);
    asm volatile("cp.async.commit_group;\n");
  }
  for (int kt = 0; kt < KT; ++kt) {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(STAGES - 2));
    __syncthreads();
    {
      const int nk = kt + STAGES - 1;
      if (nk < KT) load_tile(nk % STAGES, nk);
      asm volatile("cp.async.commit_group;\n");
    }
    const int st = kt % STAGES;
#pragma unroll
    for (int kk = 0; kk < BK; kk += 16) {
      uint32_t af[4][4], bfr[4][2];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int row = wm * 64 + i * 16 + (lane & 15);
        const int col = kk + (lane >> 4) * 8;
        ldsm_x4(smem_u32(As + (st * BM + row) * LDS + col), af[i][0], af[i][1], af[i][2], af[i][3]);
      }
#pragma unroll
      for (int jp = 0; jp < 2; ++jp) {
        const int row = wn * 32 + jp * 16 + (lane & 7) + ((lane >> 4) << 3);
        const int col = kk + ((lane >> 3) & 1) * 8;
        uint32_t r0, r1, r2, r3;
        ldsm_x4(smem_u32(Bs + (st * BN + row) * LDS + col), r0, r1, r2, r3);
        bfr[2 * jp][0] = r0; bfr[2 * jp][1] = r1;
        bfr[2 * jp + 1][0] = r2; bfr[2 * jp + 1][1] = r3;
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) mma_bf16(acc[i][j], af[i], bfr[j][0], bfr[j][1]);
    }
  }
  asm volatile("cp.async.wait_group 0;\n");

  // epilogue
  const int g = lane >> 2, c2 = (lane & 3) * 2;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int row = m0 + wm * 64 + i * 16 + g + h * 8;
      if (row >= M) continue;
      if constexpr (EPI == EPI_SWIGLU) {
        const int col0 = n0 + wn * 32;  // 16 gate columns then 16 up columns
        if (col0 >= N) continue;
        uint16_t* C = static_cast<uint16_t*>(Cv);
        const int F = N / 2;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const float g0 = acc[i][j][2 * h], g1 = acc[i][j][2 * h + 1];
          const float u0 = acc[i][j + 2][2 * h], u1 = acc[i][j + 2][2 * h + 1];
          const int oc = col0 / 2 + j * 8 + c2;
          *reinterpret_cast<uint32_t*>(C + (size_t)row * F + oc) = pack_bf16x2(silu(g0) * u0, silu(g1) * u1);
        }
      } else {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int col = n0 + wn * 32 + j * 8 + c2;
          if (col >= N) continue;
          const float v0 = acc[i][j][2 * h], v1 = acc[i][j][2 * h + 1];
          if constexpr (EPI == EPI_STORE_BF16) {
            uint16_t* C = static_cast<uint16_t*>(Cv);
            *reinterpret_cast<uint32_t*>(C + (size_t)row * N + col) = pack_bf16x2(v0, v1);
          } else {
            float* R = static_cast<float*>(Cv);
            float2* p = reinterpret_cast<float2*>(R + (size_t)row * N + col);
            float2 r = *p;
            r.x += v0;
            r.y += v1;
            *p = r;
          }
        }
      }
    }
  }
}

}  // namespace mma_gemm

int launch_gemm_mma(const void* A, const void* B, int M, int N, int K, int epi, void* C, cudaStream_t st) {
  using namespace mma_gemm;
  const int mt = (M + BM - 1) / BM, nt = (N + BN - 1) / BN;
  const int grid = mt * nt;
  if (grid == 0) return 0;
  const uint16_t* a = static_cast<const uint16_t*>(A);
  const uint16_t* b = static_cast<const uint16_t*>(B);
  switch (epi) {
    case EPI_STORE_BF16:
      cudaFuncSetAttribute(gemm_kernel<EPI_STORE_BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM);
      gemm_kernel<EPI_STORE_BF16><<<grid, THREADS, SMEM, st>>>(a, b, M, N, K, C);
      break;
    case EPI_RESID_F32:
      cudaFuncSetAttribute(gemm_kernel<EPI_RESID_F32>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM);
      gemm_kernel<EPI_RESID_F32><<<grid, THREADS, SMEM, st>>>(a, b, M, N, K, C);
      break;
    case EPI_SWIGLU:
      cudaFuncSetAttribute(gemm_kernel<EPI_SWIGLU>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM);
      gemm_kernel<EPI_SWIGLU><<<grid, THREADS, SMEM, st>>>(a, b, M, N, K, C);
      break;
    default:
      return 1;
  }
  return 0;
}

}  // namespace rift
