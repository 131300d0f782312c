// The prefill GEMMs on Blackwell's fifth-generation tensor cores (tcgen05, sm_103a).
//
// C[M, N] = A[M, K] . B[N, K]^T with fp16 operands (both K-major) and fp32 accumulation in
// tensor memory, plus the fused epilogues of the decoder layer (fp16 store with RoPE on q and
// k, fp32 residual add, SwiGLU over 16-column gate/up groups).
//
// Persistent, warp-specialised kernel, one CTA per SM (192 threads):
//   warp 0      one thread issues TMA tile loads (128B-swizzled) into a 4-stage shared-memory ring
//   warp 1      allocates 512 TMEM columns; one thread issues tcgen05.mma (M = 128, N = 256, K = 16)
//               into one of two 256-column fp32 accumulators and commits to mbarriers
//   warps 2..5  epilogue: tcgen05.ld of their 32 TMEM lanes (one row per thread), fused op, store
// Two accumulators let the epilogue of one tile overlap the main loop of the next.  Tiles are
// visited in bands of M-tiles whose A rows fit in L2 (48 MB), so each weight tile is read from
// DRAM once per band.
// Split-K (for few rows, where the tiles alone would leave most SMs idle, as in the decode
// step): the work units are (tile, K-slice) pairs, each unit stores its fp32 partial product
// into a caller workspace, and splitk_reduce_kernel sums the slices in a fixed order and
// applies the epilogue.
// Every mbarrier wait is bounded (RIFT_SPIN_LIMIT iterations, ~4 s of globaltimer): on timeout
// the kernel sets RIFT_EBIT_TIMEOUT, lets every role fall through, waits for its issued copies
// and frees its tensor memory.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "rift_internal.h"

namespace rift {

__device__ unsigned int g_err_gemm;

unsigned int read_clear_err_gemm() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_err_gemm, sizeof(v));
  cudaMemcpyToSymbol(g_err_gemm, &z, sizeof(z));
  return v;
}

namespace tc {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;  // 16 KB
constexpr int THREADS = 192;
// Instruction descriptor (per kernel instance), kind::f16: D fp32 (bits 4-5 = 1), A fp16 (bits
// 7-9 = 0), B fp16 (bits 10-12 = 0), both K-major (bits 15, 16 = 0), N >> 3 at bits 17-22, M >> 4
// at bits 24-28.

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Shared-memory matrix descriptor for a K-major tile written by TMA with 128-byte swizzling:
// start address >> 4 (bits 0-13), leading byte offset 16 B (unused for this layout), stride
// byte offset 1024 B between 8-row groups (bits 32-45), descriptor version 1 (bit 46),
// swizzle mode 2 = 128B (bits 61-63).
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr) {
  return (uint64_t)((addr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.b32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
      " selp.b32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait for the phase of parity `parity` (CL: acquire at cluster scope, for a barrier the
// other CTA of the pair arrives on).  Returns false if the kernel is aborting or the wait ran out
// (which starts the abort).
template <bool CL = false>
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  auto tw = [&]() { return CL ? mbar_try_wait_cluster(bar, parity) : mbar_try_wait(bar, parity); };
  if (tw()) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t i = 0; i < RIFT_SPIN_LIMIT; ++i) {
    if (tw()) return true;
    if ((i & 255u) == 255u) {
      if (*abort_flag) return false;
      if (globaltimer() - t0 > 4000000000ull) break;
    }
  }
  atomicOr(&g_err_gemm, RIFT_EBIT_TIMEOUT);
  *abort_flag = 1;
  return false;
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];\n" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void umma_f16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accum) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accum));
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(bar)
               : "memory");
}
// The SM-pair forms (cta_group::2): the two CTAs of a 2-CTA cluster share one M = 256 product.
// The even CTA issues the MMA; each CTA holds its own 128 rows of A and 128 of the 256 B rows
// in shared memory at the same offsets, and its own 128 accumulator rows in tensor memory.
__device__ __forceinline__ void umma_f16_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                              uint32_t accum) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accum));
}
// Arrive on the mbarrier at this offset in both CTAs of the pair once the pair's MMAs are done.
__device__ __forceinline__ void umma_commit_pair(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;\n" ::"r"(
          bar),
      "h"((uint16_t)3)
      : "memory");
}
// TMA load into this CTA's shared memory whose completion is counted on an mbarrier of either
// CTA of the pair (bar: a shared::cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, "
      "%3}], [%4];\n" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;\n" : "=r"(r));
  return r;
}
// The shared::cluster address of this CTA's shared variable at `addr` in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t d;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;\n" : "=r"(d) : "r"(addr), "r"(rank));
  return d;
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];\n" ::"r"(cluster_addr) : "memory");
}
__device__ __forceinline__ void cluster_sync() {
  __syncwarp();
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;\n" ::: "memory");
}
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }

// 32 consecutive fp32 accumulator columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
}

// Tile order.  group > 0: bands of `group` M-tiles, M fastest within a band, so the band's A rows
// stay in L2 while every B tile streams past them once per band.  group < 0: bands of -group
// N-tiles, N fastest, so the band's B rows stay in L2 and A streams once per band (the better
// order when B is the smaller operand: traffic A + B x bands vs B + A x bands).
__device__ __forceinline__ void tile_coords(int tile, int mt, int nt, int group, int& m_blk, int& n_blk) {
  const bool n_major = group < 0;
  const int g = n_major ? -group : group;
  const int inner = n_major ? nt : mt, outer = n_major ? mt : nt;
  const int per_group = g * outer;
  const int grp = tile / per_group;
  const int first = grp * g;
  const int gsz = min(inner - first, g);
  const int r = tile - grp * per_group;
  const int a = first + r % gsz, b = r / gsz;
  m_blk = n_major ? b : a;
  n_blk = n_major ? a : b;
}

// Tile t of the upper triangle (bi <= bj) of an mt x mt tile grid, row by row.
__device__ __forceinline__ void tri_coords(int t, int mt, int& bi, int& bj) {
  int b = 0;
  while (b < mt - 1 && t >= mt - b) {
    t -= mt - b;
    ++b;
  }
  bi = b;
  bj = b + t;
}

__device__ __forceinline__ float silu(float g) { return g / (1.f + expf(-g)); }

// Epilogue for one row of one 32-column chunk (columns n0 .. n0 + 31 of the tile).
template <int EPI>
__device__ __forceinline__ void epilogue_chunk(const uint32_t (&r)[32], int row, int col, int N, void* C,
                                               float out_scale = 1.f) {
  if constexpr (EPI == EPI_STORE_F32) {
    float* out = static_cast<float*>(C) + (size_t)row * N + col;
    if (col + 32 <= N) {
      float4* o4 = reinterpret_cast<float4*>(out);
#pragma unroll
      for (int q = 0; q < 8; ++q)
        o4[q] = make_float4(__uint_as_float(r[4 * q]) * out_scale, __uint_as_float(r[4 * q + 1]) * out_scale,
                            __uint_as_float(r[4 * q + 2]) * out_scale, __uint_as_float(r[4 * q + 3]) * out_scale);
    } else {
      for (int j = 0; j < 32 && col + j < N; ++j) out[j] = __uint_as_float(r[j]) * out_scale;
    }
  } else if constexpr (EPI == EPI_STORE_BF16) {
    uint16_t* out = static_cast<uint16_t*>(C) + (size_t)row * N + col;
    if (col + 32 <= N) {
      uint4* o4 = reinterpret_cast<uint4*>(out);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        o4[q] = make_uint4(pack_half2(__uint_as_float(r[8 * q + 0]), __uint_as_float(r[8 * q + 1])),
                           pack_half2(__uint_as_float(r[8 * q + 2]), __uint_as_float(r[8 * q + 3])),
                           pack_half2(__uint_as_float(r[8 * q + 4]), __uint_as_float(r[8 * q + 5])),
                           pack_half2(__uint_as_float(r[8 * q + 6]), __uint_as_float(r[8 * q + 7])));
    } else {
#pragma unroll
      for (int j = 0; j < 32; j += 2)
        if (col + j < N)
          *reinterpret_cast<uint32_t*>(out + j) = pack_half2(__uint_as_float(r[j]), __uint_as_float(r[j + 1]));
    }
  } else if constexpr (EPI == EPI_RESID_F32) {
    float* out = static_cast<float*>(C) + (size_t)row * N + col;
    if (col + 32 <= N) {
      float4* o4 = reinterpret_cast<float4*>(out);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        float4 v = o4[q];
        v.x += __uint_as_float(r[4 * q + 0]);
        v.y += __uint_as_float(r[4 * q + 1]);
        v.z += __uint_as_float(r[4 * q + 2]);
        v.w += __uint_as_float(r[4 * q + 3]);
        o4[q] = v;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (col + j < N) out[j] += __uint_as_float(r[j]);
    }
  } else if constexpr (EPI == EPI_SWIGLU) {  // columns col..col+15 gate, col+16..col+31 the matching up
    if (col >= N) return;
    const int F = N / 2;
    uint16_t* out = static_cast<uint16_t*>(C) + (size_t)row * F + col / 2;
    uint32_t p[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float g0 = __uint_as_float(r[2 * j]), g1 = __uint_as_float(r[2 * j + 1]);
      const float u0 = __uint_as_float(r[16 + 2 * j]), u1 = __uint_as_float(r[16 + 2 * j + 1]);
      p[j] = pack_half2(silu(g0) * u0, silu(g1) * u1);
    }
    uint4* o4 = reinterpret_cast<uint4*>(out);
    o4[0] = make_uint4(p[0], p[1], p[2], p[3]);
    o4[1] = make_uint4(p[4], p[5], p[6], p[7]);
  }
}

// Rotate-half RoPE on fp32 accumulators: r1 holds dims j0..j0+31 of a head, r2 the partner
// dims j0+half..; y1 = x1 cos - x2 sin, y2 = x2 cos + x1 sin, rounded once to fp16.
__device__ __forceinline__ void rope_chunk(const uint32_t (&r1)[32], const uint32_t (&r2)[32], int row, int col,
                                           int half, int N, int pos, const float2* __restrict__ tab, void* C) {
  uint16_t* out = static_cast<uint16_t*>(C) + (size_t)row * N + col;
  const int head_dim = 2 * half;
  const int j0 = col % head_dim;
  const float2* cs = tab + (size_t)pos * half + j0;
  uint32_t p1[16], p2[16];
#pragma unroll
  for (int e = 0; e < 32; e += 2) {
    const float2 c0 = cs[e], c1 = cs[e + 1];
    const float a0 = __uint_as_float(r1[e]), a1 = __uint_as_float(r1[e + 1]);
    const float b0 = __uint_as_float(r2[e]), b1 = __uint_as_float(r2[e + 1]);
    p1[e / 2] = pack_half2(a0 * c0.x - b0 * c0.y, a1 * c1.x - b1 * c1.y);
    p2[e / 2] = pack_half2(b0 * c0.x + a0 * c0.y, b1 * c1.x + a1 * c1.y);
  }
  uint4* o1 = reinterpret_cast<uint4*>(out);
  uint4* o2 = reinterpret_cast<uint4*>(out + half);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    o1[q] = make_uint4(p1[4 * q], p1[4 * q + 1], p1[4 * q + 2], p1[4 * q + 3]);
    o2[q] = make_uint4(p2[4 * q], p2[4 * q + 1], p2[4 * q + 2], p2[4 * q + 3]);
  }
}

// K-block k of an operand read through EpiParams' remap (mode 1: [hi | hi | lo], 2: [hi | lo | hi]
// over a stored [hi | lo] row of D blocks each; 0: k).
__device__ __forceinline__ int kblock(int mode, int D, int k) {
  return mode == 1 ? (k < D ? k : k - D) : mode == 2 ? (k < 2 * D ? k : k - 2 * D) : k;
}

// BN_ x STAGES_: 256 x 4 for the prefill on one SM; 128 x 6 for few-row products with the
// operands swapped (weights as the 128-row operand, the few activation rows as the N side;
// EPI_STORE_F32_T).  PAIR: 2-CTA clusters on an SM pair, 256 x 256 tiles (cta_group::2): each SM
// stages 128 rows of A and 128 of the 256 B rows per k-block, half the B traffic of one SM per
// tile row, and the even CTA issues the M = 256 MMAs into both SMs' tensor memory.
template <int EPI, int BN_, int STAGES_, bool PAIR = false>
__global__ void __launch_bounds__(THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, int M_cap,
                   int N, int K, void* C, const EpiParams ep, int group_m, int splits, size_t split_stride,
                   int a_const) {
  constexpr int BN = BN_, STAGES = STAGES_;  // this instance's tile width and ring depth
  constexpr int TM = PAIR ? 2 * BM : BM;     // rows of a tile (both CTAs of the pair)
  constexpr int B_ROWS = PAIR ? BN / 2 : BN; // B rows staged by this CTA
  constexpr int B_BYTES = B_ROWS * BK * 2, STAGE_BYTES = A_BYTES + B_BYTES;
  constexpr int ACC_COLS = BN, TMEM_COLS = 2 * ACC_COLS;
  constexpr uint32_t IDESC_T = (1u << 4) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(TM >> 4) << 24);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 4);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t bar0 = smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
  auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * STAGES + b); };
  auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * STAGES + 2 + b); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull_bar(b), 1);
      mbar_init(tempty_bar(b), PAIR ? 256 : 128);  // the epilogue threads of every CTA that drains it
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
  }
  const uint32_t rank = PAIR ? cluster_ctarank() : 0u;
  if constexpr (PAIR) cluster_sync();  // both CTAs' barriers initialised before any remote arrival
  if (warp == 1) {
    if constexpr (PAIR) {
      asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(
                       smem_u32(tmem_slot)),
                   "r"(TMEM_COLS)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;\n" ::: "memory");
    } else {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(
                       smem_u32(tmem_slot)),
                   "r"(TMEM_COLS)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
    }
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_trigger();
  // The producer waits after prefetching constant A tiles; with a device row count every role
  // waits first, since the count is written by an earlier kernel.
  if (warp != 0 || ep.m_dev) pdl_wait();
  // Rows: M_cap (host), or the device count ep.m_dev clamped to it (the rows the TMA map covers).
  const int M = ep.m_dev ? max(0, min(M_cap, *ep.m_dev)) : M_cap;

  const int mt = (M + TM - 1) / TM, nt = (N + BN - 1) / BN, kt = (K + BK - 1) / BK;
  const int n_tiles = ep.symmetric ? mt * (mt + 1) / 2 : mt * nt;
  auto coords = [&](int tile, int& m_blk, int& n_blk) {
    if (ep.symmetric) tri_coords(tile, mt, m_blk, n_blk);
    else tile_coords(tile, mt, nt, group_m, m_blk, n_blk);
  };
  // unit u: tile u / splits, K-blocks [k0, k1) of slice u % splits (the host makes every slice
  // non-empty)
  const int n_units = n_tiles * splits, k_per = (kt + splits - 1) / splits;
  auto unit_k = [&](int u, int& k0, int& k1) {
    k0 = (u % splits) * k_per;
    k1 = min(kt, k0 + k_per);
  };

  // the pair walks the units together, one unit per cluster
  const int u_first = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  const int u_step = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer (PAIR: both CTAs load their halves; the even CTA's full
      // barrier counts the bytes of both)
      // a_const: A does not depend on earlier kernels (weights), so the first ring round of this
      // CTA's first unit takes its A tiles before waiting for the kernel before this one.
      int n_pre = 0;
      if (!PAIR && a_const && !ep.m_dev && u_first < n_units) {
        int m_blk, n_blk, k0, k1;
        coords(u_first / splits, m_blk, n_blk);
        unit_k(u_first, k0, k1);
        n_pre = min(STAGES, k1 - k0);
        for (int j = 0; j < n_pre; ++j) {
          mbar_expect_tx(full_bar(j), STAGE_BYTES);
          tma_load_2d(smem_u32(sA + j * A_BYTES), &tmA, kblock(ep.kmap_a, ep.kmap_d, k0 + j) * BK, m_blk * BM,
                      full_bar(j));
        }
      }
      pdl_wait();
      int it = 0;
      bool ok = true;
      for (int u = u_first; u < n_units && ok; u += u_step) {
        int m_blk, n_blk, k0, k1;
        coords(u / splits, m_blk, n_blk);
        unit_k(u, k0, k1);
        for (int k = k0; k < k1; ++k, ++it) {
          const int s = it % STAGES;
          const uint32_t round = it / STAGES;
          if (it < n_pre) {  // A already requested (first round: the stage is free)
            tma_load_2d(smem_u32(sB + s * B_BYTES), &tmB, kblock(ep.kmap_b, ep.kmap_d, k) * BK, n_blk * BN,
                        full_bar(s));
            continue;
          }
          if (!mbar_wait(empty_bar(s), (round & 1u) ^ 1u, abort_flag)) { ok = false; break; }
          if constexpr (PAIR) {
            const uint32_t fb = mapa_shared(full_bar(s), 0);
            if (rank == 0) mbar_expect_tx(full_bar(s), 2 * STAGE_BYTES);
            tma_load_2d_pair(smem_u32(sA + s * A_BYTES), &tmA, kblock(ep.kmap_a, ep.kmap_d, k) * BK,
                             m_blk * TM + (int)rank * BM, fb);
            tma_load_2d_pair(smem_u32(sB + s * B_BYTES), &tmB, kblock(ep.kmap_b, ep.kmap_d, k) * BK,
                             n_blk * BN + (int)rank * B_ROWS, fb);
          } else {
            mbar_expect_tx(full_bar(s), STAGE_BYTES);
            tma_load_2d(smem_u32(sA + s * A_BYTES), &tmA, kblock(ep.kmap_a, ep.kmap_d, k) * BK, m_blk * BM, full_bar(s));
            tma_load_2d(smem_u32(sB + s * B_BYTES), &tmB, kblock(ep.kmap_b, ep.kmap_d, k) * BK, n_blk * BN, full_bar(s));
          }
        }
      }
      // Before leaving, make sure no copy this thread issued is still in flight (bounded).  PAIR:
      // the copies are counted on the even CTA's barrier, so wait instead for the MMAs' releases
      // of the last stages, which also keeps this CTA alive until they have all arrived.
      for (int j = 1; j <= STAGES && it - j >= 0; ++j) {
        const int i2 = it - j;
        const int s = i2 % STAGES;
        const uint32_t round = i2 / STAGES;
        const uint32_t bar = PAIR ? empty_bar(s) : full_bar(s);
        for (uint32_t w = 0; w < (1u << 22) && !mbar_try_wait(bar, round & 1u); ++w) {
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // ---------------- MMA issuer (PAIR: the even CTA only)
      int it = 0, tl = 0;
      bool ok = true;
      for (int u = u_first; u < n_units && ok; u += u_step, ++tl) {
        int k0, k1;
        unit_k(u, k0, k1);
        const int b = tl & 1;
        const uint32_t use = tl >> 1;
        if (!mbar_wait<PAIR>(tempty_bar(b), (use & 1u) ^ 1u, abort_flag)) break;
        fence_after();
        const uint32_t tmem_d = tmem_base + (uint32_t)(b * ACC_COLS);
        for (int k = k0; k < k1; ++k, ++it) {
          const int s = it % STAGES;
          const uint32_t round = it / STAGES;
          if (!mbar_wait(full_bar(s), round & 1u, abort_flag)) { ok = false; break; }
          fence_after();
          const uint64_t ad = smem_desc(smem_u32(sA + s * A_BYTES));
          const uint64_t bd = smem_desc(smem_u32(sB + s * B_BYTES));
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {  // +32 bytes along K per step (encoded >> 4)
            if constexpr (PAIR)
              umma_f16_pair(tmem_d, ad + 2 * kk, bd + 2 * kk, IDESC_T, (k != k0 || kk != 0) ? 1u : 0u);
            else
              umma_f16(tmem_d, ad + 2 * kk, bd + 2 * kk, IDESC_T, (k != k0 || kk != 0) ? 1u : 0u);
          }
          if constexpr (PAIR) umma_commit_pair(empty_bar(s));
          else umma_commit(empty_bar(s));
        }
        if (ok) {
          if constexpr (PAIR) umma_commit_pair(tfull_bar(b));
          else umma_commit(tfull_bar(b));
        }
      }
      if constexpr (PAIR) {
        // the last two accumulators' releases (the odd CTA's arrivals among them) have landed
        for (int t = tl - 1; t >= 0 && t >= tl - 2; --t)
          for (uint32_t w = 0; w < (1u << 22) && !mbar_try_wait_cluster(tempty_bar(t & 1), (t >> 1) & 1u); ++w) {
          }
      }
    }
  } else {
    // ---------------- epilogue (warps 2..5 -> TMEM lane quarters 2, 3, 0, 1)
    const int quarter = warp & 3;
    const uint32_t tempty_even0 = PAIR ? mapa_shared(tempty_bar(0), 0) : tempty_bar(0);
    const uint32_t tempty_even1 = PAIR ? mapa_shared(tempty_bar(1), 0) : tempty_bar(1);
    int tl = 0;
    for (int u = u_first; u < n_units; u += u_step, ++tl) {
      int m_blk, n_blk;
      coords(u / splits, m_blk, n_blk);
      // split-K partials (EPI_STORE_F32 only): slice u % splits at C + slice * split_stride
      void* Cu = splits > 1 ? static_cast<void*>(static_cast<float*>(C) + (size_t)(u % splits) * split_stride) : C;
      const int b = tl & 1;
      const uint32_t use = tl >> 1;
      if (!mbar_wait(tfull_bar(b), use & 1u, abort_flag)) break;
      fence_after();
      const int row = m_blk * TM + (int)rank * BM + quarter * 32 + lane;
      const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(b * ACC_COLS);
      if constexpr (EPI == EPI_QKV_ROPE) {
        const int half = ep.head_dim >> 1;
        const int pos = (row < M) ? ep.positions[row] + ep.pos_offset : 0;
        const bool pos_ok = pos >= 0 && pos < ep.max_len;
        if (row < M && !pos_ok) atomicOr(&g_err_gemm, RIFT_EBIT_BADID);
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          const int col = n_blk * BN + c;
          if (col >= N) break;
          if (col < ep.rope_cols) {
            if ((c % ep.head_dim) >= half) continue;  // done with its partner c - half
            uint32_t r1[32], r2[32];
            tmem_ld32(taddr + c, r1);
            tmem_ld32(taddr + c + half, r2);
            if (row < M && pos_ok) rope_chunk(r1, r2, row, col, half, N, pos, ep.rope, C);
          } else {
            uint32_t r[32];
            tmem_ld32(taddr + c, r);
            if (row < M) epilogue_chunk<EPI_STORE_BF16>(r, row, col, N, C);
          }
        }
      } else {
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          uint32_t r[32];
          tmem_ld32(taddr + c, r);
          if constexpr (EPI == EPI_STORE_F32_T) {  // C[col][row] (transposed), col < N, row < M
            const int col = n_blk * BN + c;
            if (row < M) {
              float* out = static_cast<float*>(Cu) + row;
#pragma unroll
              for (int e = 0; e < 32; ++e)
                if (col + e < N) out[(size_t)(col + e) * M] = __uint_as_float(r[e]);
            }
          } else {
            if (row < M) epilogue_chunk<EPI>(r, row, n_blk * BN + c, N, Cu, ep.out_scale);
            if constexpr (EPI == EPI_STORE_F32) {
              // symmetric product: the off-diagonal tile also fills its mirror (a warp's lanes hold
              // consecutive rows, so each transposed store is 32 consecutive floats)
              if (ep.symmetric && m_blk != n_blk && row < M) {
                float* out = static_cast<float*>(Cu);
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                  const int col = n_blk * BN + c + e;
                  if (col < M) out[(size_t)col * N + row] = __uint_as_float(r[e]) * ep.out_scale;
                }
              }
            }
          }
        }
      }
      fence_before();
      if constexpr (PAIR) mbar_arrive_cluster(b ? tempty_even1 : tempty_even0);
      else mbar_arrive(tempty_bar(b));
    }
  }
  fence_before();
  __syncthreads();
  if constexpr (PAIR) cluster_sync();  // neither CTA frees its tensor memory or exits before the other is done
  if (warp == 1) {
    fence_after();
    if constexpr (PAIR)
      asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_base), "r"(TMEM_COLS)
                   : "memory");
    else
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_base), "r"(TMEM_COLS)
                   : "memory");
  }
}

// ---------------------------------------------------------------- merge screening (Stage 2)
// Similarity of every token of a kept tile to the tile's merge targets on the tensor cores: per
// (kept slot j, 128-token block) a 128 x 128 x d bf16 product against 128 target rows at a time,
// one token row per epilogue thread, which keeps the two best targets by x.t / ||t|| (fp32, ties
// to the lower target) for each unselected token that is not itself a target.  The choice
// between the two is then made at ~fp64 accuracy outside (merge.cu).  Rows of the block past the
// tile's tokens and target columns past the slot's m are computed and ignored.
namespace ms {
constexpr int STAGES = 3, THREADS = 192, COLS = 128;
constexpr int A_BYTES = 128 * BK * 2, B_BYTES = COLS * BK * 2, STAGE_BYTES = A_BYTES + B_BYTES;
constexpr size_t SMEM = (size_t)STAGES * STAGE_BYTES + 1024 + 256;
// kind::f16 with bf16 A and B (bits 7-9 and 10-12 = 1), fp32 D, K-major, M = N = 128
constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(COLS >> 3) << 17) | ((128u >> 4) << 24);
}  // namespace ms

__global__ void __launch_bounds__(ms::THREADS, 2)
    merge_screen_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmT, int n_v,
                        int d, const int* __restrict__ kept, const int* __restrict__ n_kept,
                        const int* __restrict__ sel_off, const int* __restrict__ ctx_off, int max_ctx,
                        const float* __restrict__ tinv, const int* __restrict__ pos, int2* __restrict__ cand) {
  constexpr int STAGES = ms::STAGES, COLS = ms::COLS, A_BYTES = ms::A_BYTES, B_BYTES = ms::B_BYTES,
                STAGE_BYTES = ms::STAGE_BYTES;
  constexpr uint32_t IDESC = ms::IDESC;
  const int j = blockIdx.y, mb = blockIdx.x;
  if (j >= *n_kept) return;
  const int co = ctx_off[j], m = ctx_off[j + 1] - co;
  if (m == 0 || co + m > max_ctx) return;  // uniform over the CTA, before any setup
  const int R = n_v - (sel_off[j + 1] - sel_off[j]);
  const int step = R / m;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t bar0 = smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
  const uint32_t tfull = bar0 + 8u * (2 * STAGES), tempty = bar0 + 8u * (2 * STAGES + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s2 = 0; s2 < STAGES; ++s2) {
      mbar_init(full_bar(s2), 1);
      mbar_init(empty_bar(s2), 1);
    }
    mbar_init(tfull, 1);
    mbar_init(tempty, 128);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(tmem_slot)),
                 "r"(COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int kt = d / BK, nblk = (m + COLS - 1) / COLS;
  const int xrow = kept[j] * n_v + mb * 128;

  if (warp == 0) {
    if (lane == 0) {
      int it = 0;
      bool ok = true;
      for (int nb = 0; nb < nblk && ok; ++nb)
        for (int k = 0; k < kt; ++k, ++it) {
          const int s2 = it % STAGES;
          const uint32_t round = it / STAGES;
          if (!mbar_wait(empty_bar(s2), (round & 1u) ^ 1u, abort_flag)) { ok = false; break; }
          mbar_expect_tx(full_bar(s2), STAGE_BYTES);
          tma_load_2d(smem_u32(sA + s2 * A_BYTES), &tmX, k * BK, xrow, full_bar(s2));
          tma_load_2d(smem_u32(sB + s2 * B_BYTES), &tmT, k * BK, co + nb * COLS, full_bar(s2));
        }
      for (int q = 1; q <= STAGES && it - q >= 0; ++q) {  // no copy left in flight (bounded)
        const int i2 = it - q;
        for (uint32_t w = 0; w < (1u << 22) && !mbar_try_wait(full_bar(i2 % STAGES), (i2 / STAGES) & 1u); ++w) {
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int it = 0;
      bool ok = true;
      for (int nb = 0; nb < nblk && ok; ++nb) {
        if (!mbar_wait(tempty, (nb & 1) ^ 1, abort_flag)) break;
        fence_after();
        for (int k = 0; k < kt; ++k, ++it) {
          const int s2 = it % STAGES;
          if (!mbar_wait(full_bar(s2), (it / STAGES) & 1u, abort_flag)) { ok = false; break; }
          fence_after();
          const uint64_t ad = smem_desc(smem_u32(sA + s2 * A_BYTES));
          const uint64_t bd = smem_desc(smem_u32(sB + s2 * B_BYTES));
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            umma_f16(tmem_base, ad + 2 * kk, bd + 2 * kk, IDESC, (k != 0 || kk != 0) ? 1u : 0u);
          umma_commit(empty_bar(s2));
        }
        if (ok) umma_commit(tfull);
      }
    }
  } else {
    // epilogue: warps 2..5 -> TMEM lane quarters 2, 3, 0, 1; thread = token row
    const int quarter = warp & 3, r = quarter * 32 + lane;
    const int tok = mb * 128 + r;
    const int a = tok < n_v ? pos[(size_t)j * n_v + tok] : -1;
    const bool want = a >= 0 && !(a % step == 0 && a / step < m);
    float v1 = -INFINITY, v2 = -INFINITY;
    int b1 = -1, b2 = -1;
    bool ok = true;
    for (int nb = 0; nb < nblk; ++nb) {
      const int c0 = nb * COLS, nc = min(COLS, m - c0);
      const float* inv_n = tinv + co + c0;  // 1 / ||t|| (0 for a zero target: similarity 0)
      if (!mbar_wait(tfull, nb & 1, abort_flag)) { ok = false; break; }
      fence_after();
      const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16);
      for (int c = 0; c < nc; c += 32) {
        uint32_t acc[32];
        tmem_ld32(taddr + c, acc);
        if (want) {
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            if (c + e < nc) {
              const float v = __uint_as_float(acc[e]) * inv_n[c + e];
              const int b = c0 + c + e;
              if (v > v1) {
                v2 = v1;
                b2 = b1;
                v1 = v;
                b1 = b;
              } else if (v > v2) {
                v2 = v;
                b2 = b;
              }
            }
          }
        }
      }
      fence_before();
      mbar_arrive(tempty);
    }
    if (ok && want) cand[(size_t)j * n_v + a] = make_int2(b1, b2);
  }
  fence_before();
  __syncthreads();
  if (warp == 1) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_base), "r"(COLS) : "memory");
  }
}

// ------------------------------------------------------------------------------------------ host

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D fp16 tensor [rows, inner] (row-major, inner contiguous), box [box_rows, 64], 128B swizzle,
// out-of-bounds elements read as zero.
static bool make_map(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows,
                     CUtensorMapDataType dt = CU_TENSOR_MAP_DATA_TYPE_FLOAT16) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {(cuuint32_t)BK, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, dt, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
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

// L2 band of the tile order (tile_coords): as many tiles of the resident operand as keep its rows
// within kBandBytes of L2 (lo..hi tiles).  The resident operand is the larger one when
// kOrientBands (the smaller one is then streamed once per band), else always A.
constexpr size_t kBandBytes = (size_t)48 << 20;
constexpr bool kOrientBands = true;
static int band_group(int M, int N, int K, int tm, int tn, int lo, int hi) {
  const bool n_major = kOrientBands && (size_t)N < (size_t)M;
  int g = (int)(kBandBytes / ((size_t)(n_major ? tn : tm) * K * 2));
  g = g < lo ? lo : (g > hi ? hi : g);
  return n_major ? -g : g;
}

// pdl: launched as a programmatic dependent of the kernel before it; a_const: A is constant weights.
template <int EPI, int BN_ = BN, int STAGES_ = STAGES>
static int launch(const CUtensorMap& a, const CUtensorMap& b, int M, int N, int K, void* C, const EpiParams& ep,
                  cudaStream_t st, int splits = 1, bool pdl = false, int a_const = 0) {
  constexpr size_t smem = (size_t)STAGES_ * (A_BYTES + BN_ * BK * 2) + 1024 + 256;
  static std::atomic<unsigned long long> smem_raised{0};
  if (raise_smem_limit(smem_raised, gemm_tc_kernel<EPI, BN_, STAGES_>, (int)smem) != cudaSuccess) return 1;
  const int units = ((M + BM - 1) / BM) * ((N + BN_ - 1) / BN_) * splits;
  const int grid = units < sm_count() ? units : sm_count();
  const int group_m = band_group(M, N, K, BM, BN_, 8, 64);
  return launch_ex(gemm_tc_kernel<EPI, BN_, STAGES_>, dim3(grid), dim3(THREADS), smem, st, pdl, a, b, M, N, K, C, ep,
                   group_m, splits, (size_t)M * N, a_const) != cudaSuccess;
}

// The paired kernel (2-CTA clusters, 256 x 256 tiles), persistent over as many clusters as can be
// resident at once.  b: the B map with 128-row boxes.  Returns -1 if no cluster can be resident
// (the caller then uses one SM per tile).
constexpr int PAIR_STAGES = 6;
template <int EPI>
static int launch_pair(const CUtensorMap& a, const CUtensorMap& b, int M, int N, int K, void* C, const EpiParams& ep,
                       cudaStream_t st) {
  constexpr size_t smem = (size_t)PAIR_STAGES * (A_BYTES + (BN / 2) * BK * 2) + 1024 + 256;
  auto kern = gemm_tc_kernel<EPI, BN, PAIR_STAGES, true>;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // per device: the raised shared-memory limit, and how many 2-CTA clusters fit at once (+1; 0 = not
  // asked yet)
  static std::atomic<unsigned long long> smem_raised{0};
  static std::atomic<int> clusters_plus1[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  int known = (dev >= 0 && dev < 64) ? clusters_plus1[dev].load(std::memory_order_acquire) : 0;
  if (known == 0) {
    int n = 0;
    cfg.gridDim = dim3(2, 1, 1);
    if (raise_smem_limit(smem_raised, kern, (int)smem) != cudaSuccess ||
        cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
      cudaGetLastError();
      n = 0;
    }
    known = n + 1;
    if (dev >= 0 && dev < 64) clusters_plus1[dev].store(known, std::memory_order_release);
  } else if (raise_smem_limit(smem_raised, kern, (int)smem) != cudaSuccess) {
    return 1;
  }
  const int max_clusters = known - 1;
  if (max_clusters <= 0) return -1;
  const int units = ((M + 2 * BM - 1) / (2 * BM)) * ((N + BN - 1) / BN);
  const int clusters = units < max_clusters ? units : max_clusters;
  const int group_m = band_group(M, N, K, 2 * BM, BN, 4, 32);
  cfg.gridDim = dim3(2 * clusters, 1, 1);
  cfg.stream = st;
  return cudaLaunchKernelEx(&cfg, kern, a, b, M, N, K, C, ep, group_m, 1, (size_t)M * N, 0) == cudaSuccess ? 0 : 1;
}

// Sum of the split-K slices (in slice order) and the epilogue EPI, four consecutive outputs per
// thread and step (float4 partial reads): the same arithmetic as epilogue_chunk / rope_chunk on
// the summed accumulator.  N % 8 == 0, so a group of four never straddles a row, a SwiGLU
// 16-column group or a RoPE half.
template <int EPI>
__global__ void splitk_reduce_kernel(const float* __restrict__ part, int splits, int M, int N, void* C,
                                     const EpiParams ep) {
  pdl_trigger();
  pdl_wait();
  const size_t stride = (size_t)M * N;
  const int n_out = EPI == EPI_SWIGLU ? N / 2 : N;
  const int q_out = n_out / 4;
  const size_t total = (size_t)M * q_out;
  auto acc4 = [&](int row, int col) {
    const float* p = part + (size_t)row * N + col;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
    for (int sp = 0; sp < splits; ++sp) {
      const float4 f = *reinterpret_cast<const float4*>(p + sp * stride);
      v.x += f.x;
      v.y += f.y;
      v.z += f.z;
      v.w += f.w;
    }
    return v;
  };
  auto store_h4 = [](void* dst, float a, float b, float c, float d) {
    *reinterpret_cast<uint2*>(dst) = make_uint2(pack_half2(a, b), pack_half2(c, d));
  };
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < total; e += (size_t)gridDim.x * blockDim.x) {
    const int row = (int)(e / q_out), col = (int)(e % q_out) * 4;
    if constexpr (EPI == EPI_STORE_F32) {
      const float4 v = acc4(row, col);
      *reinterpret_cast<float4*>(static_cast<float*>(C) + (size_t)row * N + col) =
          make_float4(v.x * ep.out_scale, v.y * ep.out_scale, v.z * ep.out_scale, v.w * ep.out_scale);
    } else if constexpr (EPI == EPI_RESID_F32) {
      const float4 v = acc4(row, col);
      float4* o = reinterpret_cast<float4*>(static_cast<float*>(C) + (size_t)row * N + col);
      float4 r = *o;
      r.x += v.x;
      r.y += v.y;
      r.z += v.z;
      r.w += v.w;
      *o = r;
    } else if constexpr (EPI == EPI_STORE_BF16) {
      const float4 v = acc4(row, col);
      store_h4(static_cast<uint16_t*>(C) + (size_t)row * N + col, v.x, v.y, v.z, v.w);
    } else if constexpr (EPI == EPI_SWIGLU) {  // outputs f..f+3: gate column 32 (f / 16) + f % 16, up 16 further
      const int gc = 32 * (col / 16) + col % 16;
      const float4 g = acc4(row, gc), u = acc4(row, gc + 16);
      store_h4(static_cast<uint16_t*>(C) + (size_t)row * n_out + col, silu(g.x) * u.x, silu(g.y) * u.y,
               silu(g.z) * u.z, silu(g.w) * u.w);
    } else if constexpr (EPI == EPI_QKV_ROPE) {
      float4 y = acc4(row, col);
      if (col < ep.rope_cols) {
        const int half = ep.head_dim >> 1, j = col % ep.head_dim;
        const int pos = ep.positions[row] + ep.pos_offset;
        if (pos < 0 || pos >= ep.max_len) {
          if (j == 0) atomicOr(&g_err_gemm, RIFT_EBIT_BADID);
          continue;  // as the fused epilogue: q and k of a row without a valid position stay unwritten
        }
        const float2* cs = ep.rope + (size_t)pos * half + (j < half ? j : j - half);
        const float4 x = acc4(row, j < half ? col + half : col - half);  // the partner dims
        const float sg = j < half ? -1.f : 1.f;  // first half: x cos - x' sin; second: x cos + x' sin
        y = make_float4(y.x * cs[0].x + sg * x.x * cs[0].y, y.y * cs[1].x + sg * x.y * cs[1].y,
                        y.z * cs[2].x + sg * x.z * cs[2].y, y.w * cs[3].x + sg * x.w * cs[3].y);
      }
      store_h4(static_cast<uint16_t*>(C) + (size_t)row * N + col, y.x, y.y, y.z, y.w);
    }
  }
}

// The residual add of a split-K product fused with the RMSNorm that follows it: one CTA per row,
// h[row] += sum of the slices (in slice order), then out[row] = fp16(h / sqrt(mean(h^2) + eps) g)
// with the bf16 gain g (the arithmetic of the standalone RMSNorm kernel).  N % 4 == 0, N <= 8192.
// The rows are few (one per sequence in a decode step), so the kernel is latency-bound: a CTA has
// up to 1024 threads and each holds VPT float4 columns of its row (1 at N = 4096), so that all of
// a thread's loads (its columns of h and of every slice) are independent and issue together.
template <int VPT>
__global__ void __launch_bounds__(1024) splitk_resid_norm_kernel(const float* __restrict__ part, int splits, int M,
                                                                 int N, float* __restrict__ h32,
                                                                 const uint16_t* __restrict__ gain, float eps,
                                                                 uint16_t* __restrict__ out) {
  __shared__ float red[32];
  pdl_trigger();
  pdl_wait();
  const size_t row = blockIdx.x, stride = (size_t)M * N;
  const int nv = N / 4;
  float4 v[VPT];
  float ss = 0.f;
#pragma unroll
  for (int q = 0; q < VPT; ++q) {
    const int c = threadIdx.x + q * blockDim.x;
    if (c < nv) {
      float4 a = reinterpret_cast<const float4*>(h32 + row * N)[c];
      const float4* p = reinterpret_cast<const float4*>(part + row * N) + c;
#pragma unroll 4
      for (int sp = 0; sp < splits; ++sp) {
        const float4 f = p[sp * stride / 4];
        a.x += f.x;
        a.y += f.y;
        a.z += f.z;
        a.w += f.w;
      }
      reinterpret_cast<float4*>(h32 + row * N)[c] = a;
      v[q] = a;
      ss += a.x * a.x + a.y * a.y + a.z * a.z + a.w * a.w;
    }
  }
  const float inv = rsqrtf(block_sum(ss, red) / (float)N + eps);
#pragma unroll
  for (int q = 0; q < VPT; ++q) {
    const int c = threadIdx.x + q * blockDim.x;
    if (c < nv) {
      const uint2 gr = reinterpret_cast<const uint2*>(gain)[c];
      const float g0 = __uint_as_float(gr.x << 16), g1 = __uint_as_float(gr.x & 0xffff0000u);
      const float g2 = __uint_as_float(gr.y << 16), g3 = __uint_as_float(gr.y & 0xffff0000u);
      reinterpret_cast<uint2*>(out + row * N)[c] =
          make_uint2(pack_half2(v[q].x * inv * g0, v[q].y * inv * g1), pack_half2(v[q].z * inv * g2, v[q].w * inv * g3));
    }
  }
}

// Split count for an M x N x K product whose tiles leave SMs idle: the K-slice count (1..16, at
// least 4 K-blocks a slice, partials within the workspace) that minimises the makespan, i.e. the
// rounds of units over the SMs times the K-blocks of a slice.  1 = no split.
// With `unit_cost` > 0 (the swapped few-row path, whose units always store partials) every slice
// count is weighed, each unit costing its K-blocks plus unit_cost K-blocks' worth of traffic and
// overhead; otherwise only products whose tiles leave SMs idle are split.
static int choose_splits(int M, int N, int K, size_t ws_bytes, int bn = BN, double unit_cost = 0.0) {
  const int sms = sm_count();
  const int tiles = ((M + BM - 1) / BM) * ((N + bn - 1) / bn), kt = (K + BK - 1) / BK;
  if (tiles >= sms && unit_cost == 0.0) return 1;
  int best = 1;
  double best_cost = (double)((tiles + sms - 1) / sms) * (kt + unit_cost);
  for (int s = 2; s <= 16 && kt / s >= 4; ++s) {
    if ((size_t)s * M * N * sizeof(float) > ws_bytes) break;
    const int per = (kt + s - 1) / s;
    const int se = (kt + per - 1) / per;  // every slice non-empty
    const double cost = (double)((tiles * se + sms - 1) / sms) * (per + unit_cost);
    if (cost < best_cost) {
      best_cost = cost;
      best = se;
    }
  }
  return best;
}

// A wait that can never complete (an mbarrier nobody arrives at), through the same bounded
// mbar_wait as the GEMM's pipeline: it gives up after ~4 s of globaltimer, sets
// RIFT_EBIT_TIMEOUT and returns, leaving the context usable.
__global__ void wait_timeout_check_kernel() {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  abort_flag = 0;
  mbar_init(smem_u32(&bar), 1);
  asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
  mbar_wait(smem_u32(&bar), 0, reinterpret_cast<volatile int*>(&abort_flag));
}

// The slices' partial products [splits][M][N] summed in slice order with the epilogue epi (a
// residual product with ep.norm_out also applies the following RMSNorm).
static int reduce_slices(const float* part, int splits, int M, int N, int epi, void* C, const EpiParams& ep,
                         cudaStream_t st, bool pdl) {
  if (epi == EPI_RESID_F32 && ep.norm_out) {
    float* h = static_cast<float*>(C);
    const uint16_t* g = static_cast<const uint16_t*>(ep.norm_gain);
    const cudaError_t e =
        N / 4 <= 1024
            ? launch_ex(splitk_resid_norm_kernel<1>, dim3(M), dim3((N / 4 + 31) / 32 * 32), 0, st, pdl, part, splits,
                        M, N, h, g, ep.norm_eps, ep.norm_out)
            : launch_ex(splitk_resid_norm_kernel<2>, dim3(M), dim3(1024), 0, st, pdl, part, splits, M, N, h, g,
                        ep.norm_eps, ep.norm_out);
    return e != cudaSuccess;
  }
  const size_t n_out = (size_t)M * (epi == EPI_SWIGLU ? N / 2 : N) / 4;
  const dim3 grid((unsigned)((n_out + 255) / 256 < 2048 ? (n_out + 255) / 256 : 2048));
  cudaError_t e;
  switch (epi) {
    case EPI_STORE_BF16: e = launch_ex(splitk_reduce_kernel<EPI_STORE_BF16>, grid, dim3(256), 0, st, pdl, part, splits, M, N, C, ep); break;
    case EPI_RESID_F32: e = launch_ex(splitk_reduce_kernel<EPI_RESID_F32>, grid, dim3(256), 0, st, pdl, part, splits, M, N, C, ep); break;
    case EPI_SWIGLU: e = launch_ex(splitk_reduce_kernel<EPI_SWIGLU>, grid, dim3(256), 0, st, pdl, part, splits, M, N, C, ep); break;
    case EPI_QKV_ROPE: e = launch_ex(splitk_reduce_kernel<EPI_QKV_ROPE>, grid, dim3(256), 0, st, pdl, part, splits, M, N, C, ep); break;
    case EPI_STORE_F32: e = launch_ex(splitk_reduce_kernel<EPI_STORE_F32>, grid, dim3(256), 0, st, pdl, part, splits, M, N, C, ep); break;
    default: return 1;
  }
  return e != cudaSuccess;
}

}  // namespace tc

int launch_merge_screen(const uint16_t* X, int N, int n_v, int d, const int* kept, const int* n_kept,
                        const int* sel_off, const int* ctx_off, int max_ctx, const uint16_t* targets,
                        const float* tinv, const int* pos, int2* cand, cudaStream_t st) {
  using namespace tc;
  CUtensorMap mx, mt;
  if (!make_map(&mx, X, (uint64_t)d, (uint64_t)N * n_v, 128, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16) ||
      !make_map(&mt, targets, (uint64_t)d, (uint64_t)max_ctx, ms::COLS, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16))
    return 1;
  static std::atomic<unsigned long long> smem_raised{0};
  if (raise_smem_limit(smem_raised, merge_screen_kernel, (int)ms::SMEM) != cudaSuccess) return 1;
  merge_screen_kernel<<<dim3((n_v + 127) / 128, N), ms::THREADS, ms::SMEM, st>>>(
      mx, mt, n_v, d, kept, n_kept, sel_off, ctx_off, max_ctx, tinv, pos, cand);
  return 0;
}

int launch_wait_timeout_check(cudaStream_t st) {
  tc::wait_timeout_check_kernel<<<1, 32, 0, st>>>();
  return 0;
}

// Requirements: K % 8 == 0 (16-byte row pitch), N % 8 == 0 (N % 32 == 0 for SwiGLU, N % 64 == 0 for
// the RoPE epilogue), A, B and C 16-byte aligned.
int launch_gemm_tc(const void* A, const void* B, int M, int N, int K, int epi, void* C, const EpiParams& ep,
                   cudaStream_t st, void* split_ws, size_t split_ws_bytes, bool pdl, bool b_const) {
  using namespace tc;
  if (M <= 0 || N <= 0 || K <= 0) return 0;
  if (K % 8 != 0 || N % 8 != 0 || (epi == EPI_SWIGLU && N % 32 != 0)) return 1;
  if (ep.m_dev && split_ws) return 1;  // a device row count is for the unsplit products only
  if (epi == EPI_QKV_ROPE && (N % 64 != 0 || (ep.head_dim != 64 && ep.head_dim != 128) || !ep.positions || !ep.rope))
    return 1;
  // Few rows (<= 128, with scratch: the decode step): the operands swapped so that the weights
  // stream as the 128-row operand in 128-row tiles and the rows sit on the N side (128 wide); the
  // slices' fp32 partials are stored transposed ([M, N] as the reductions below read them).
  // The operands' stored row width: K, or 2 kmap_d blocks when read through the K-block remap.
  if (ep.kmap_d && K != 3 * ep.kmap_d * BK) return 1;
  const uint64_t Ks = ep.kmap_d ? (uint64_t)2 * ep.kmap_d * BK : (uint64_t)K;
  EpiParams kp;  // the remap alone, for the partial products
  kp.kmap_d = ep.kmap_d;
  kp.kmap_a = ep.kmap_a;
  kp.kmap_b = ep.kmap_b;
  if (split_ws && M <= 128 && (size_t)M * N * sizeof(float) <= split_ws_bytes) {
    constexpr int SW_BN = 128, SW_STAGES = 6;
    CUtensorMap mw, mx;
    if (!make_map(&mw, B, Ks, (uint64_t)N, BM) || !make_map(&mx, A, Ks, (uint64_t)M, SW_BN)) return 1;
    EpiParams ks = kp;  // the operands swapped: the kernel's A is B
    ks.kmap_a = ep.kmap_b;
    ks.kmap_b = ep.kmap_a;
    // a unit's partials (M x 128 fp32, written and read back) cost M / 16 K-blocks of weight
    // traffic; its fill and drain about 1.5 more
    const int splits = choose_splits(N, M, K, split_ws_bytes, SW_BN, M / 16.0 + 1.5);
    // constant weights (b_const) are requested before the wait on the kernel before this one
    if (launch<EPI_STORE_F32_T, SW_BN, SW_STAGES>(mw, mx, N, M, K, split_ws, ks, st, splits, pdl, b_const ? 1 : 0))
      return 1;
    EpiParams e = ep;
    e.symmetric = 0;
    return reduce_slices(static_cast<const float*>(split_ws), splits, M, N, epi, C, e, st, pdl);
  }
  CUtensorMap ma, mb;
  if (!make_map(&ma, A, Ks, (uint64_t)M, BM) || !make_map(&mb, B, Ks, (uint64_t)N, BN)) return 1;
  // The residual product with a following RMSNorm (ep.norm_out) always goes through the
  // scratch, one slice or more, into the fused reduction + norm kernel.
  const bool fuse_norm = epi == EPI_RESID_F32 && ep.norm_out;
  if (fuse_norm && (!split_ws || N > 8192 || (size_t)M * N * sizeof(float) > split_ws_bytes)) return 1;
  const int splits = split_ws ? choose_splits(M, N, K, split_ws_bytes) : 1;
  if (splits > 1 || fuse_norm) {
    if (launch<EPI_STORE_F32>(ma, mb, M, N, K, split_ws, kp, st, splits, pdl)) return 1;
    EpiParams e = ep;
    e.symmetric = 0;
    return reduce_slices(static_cast<const float*>(split_ws), splits, M, N, epi, C, e, st, pdl);
  }
  // Many rows: 256 x 256 tiles on SM pairs.
  if (M >= 1024) {
    CUtensorMap mb2;
    if (!make_map(&mb2, B, Ks, (uint64_t)N, BN / 2)) return 1;
    int r = -1;
    switch (epi) {
      case EPI_STORE_BF16: r = launch_pair<EPI_STORE_BF16>(ma, mb2, M, N, K, C, ep, st); break;
      case EPI_RESID_F32: r = launch_pair<EPI_RESID_F32>(ma, mb2, M, N, K, C, ep, st); break;
      case EPI_SWIGLU: r = launch_pair<EPI_SWIGLU>(ma, mb2, M, N, K, C, ep, st); break;
      case EPI_QKV_ROPE: r = launch_pair<EPI_QKV_ROPE>(ma, mb2, M, N, K, C, ep, st); break;
      case EPI_STORE_F32: r = launch_pair<EPI_STORE_F32>(ma, mb2, M, N, K, C, ep, st); break;
      default: return 1;
    }
    if (r >= 0) return r;
  }
  EpiParams e1 = ep;  // one SM per tile: 128 x 256 tiles, every tile computed
  e1.symmetric = 0;
  switch (epi) {
    case EPI_STORE_BF16: return launch<EPI_STORE_BF16>(ma, mb, M, N, K, C, e1, st);
    case EPI_RESID_F32: return launch<EPI_RESID_F32>(ma, mb, M, N, K, C, e1, st);
    case EPI_SWIGLU: return launch<EPI_SWIGLU>(ma, mb, M, N, K, C, e1, st);
    case EPI_QKV_ROPE: return launch<EPI_QKV_ROPE>(ma, mb, M, N, K, C, e1, st);
    case EPI_STORE_F32: return launch<EPI_STORE_F32>(ma, mb, M, N, K, C, e1, st);
    default: return 1;
  }
}

}  // namespace rift
