// Varlen causal attention on Blackwell's tcgen05 tensor cores (sm_103a).
//
// Work item = (128-row q-block of one packed sequence, one head).  Persistent CTAs walk the
// items; tensor memory and barriers are set up once per CTA.  Two shapes share one kernel:
//   KB = 64   keys per block, two CTAs per SM (96 KB shared memory, 256 TMEM columns each): while
//             one CTA waits on a load, a product or its softmax, the other keeps the SM busy
//   KB = 128  keys per block, one CTA per SM, 3-stage rings and two O buffers
// Per CTA, 192 threads:
//   warp 0      TMA, two threads: lane 0 loads K tiles (KB keys) into a ring, lane 1 loads the
//               item's Q tile and the V tiles into their own ring (fp16, 128B swizzle; a 64-column
//               box per 64 head dims)
//   warp 1      one thread issues S_j = Q K_j^T (M = 128, N = KB) into one of two TMEM S buffers,
//               and O += P_j V_j with P_j read from tensor memory (the A operand of the TS form) and
//               V_j from shared memory as an MN-major operand
//   warps 2..5  softmax, one query row per thread (TMEM lane = row): scale, causal and
//               sequence-end mask, online softmax with a stale maximum (O is rescaled in TMEM
//               only when a row's maximum grows by more than 2^8), P_j written back as packed fp16
//               over the first KB / 2 columns of its own S buffer; at the end of an item O / l is
//               stored as fp16.
// K is released as soon as its S product completes and V after its PV product; S/P is
// double-buffered, so the softmax of block j overlaps S_{j+1} and PV_{j-1}.  S_{j+2} is issued
// only once PV_j (the reader of P_j in the same columns) has completed.  Every mbarrier wait is
// bounded; on timeout the kernel sets RIFT_EBIT_TIMEOUT and every role falls through.
//
// With a shared prefix (S_pre > 0: a system prompt prefilled once), every item first runs over
// the prefix's key/value blocks, loaded from their own tensor maps and masked only past S_pre, and
// then over its own sequence's blocks, causal as above.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "rift_internal.h"

namespace rift {

__device__ unsigned int g_err_attn;

unsigned int read_clear_err_attn() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_err_attn, sizeof(v));
  cudaMemcpyToSymbol(g_err_attn, &z, sizeof(z));
  return v;
}

namespace fa {

constexpr int BQ = 128, THREADS = 192;
constexpr float STALE = 8.f;  // log2 units: P <= 2^8 before a rescale is forced

template <int HD, int KB>
struct Cfg {
  static constexpr int CTAS = KB == 64 ? 2 : 1;  // CTAs per SM
  static constexpr int NST = KB == 64 ? 2 : 3;   // K and V ring stages
  static constexpr int NO = KB == 64 ? 1 : 2;    // O buffers in TMEM
  static constexpr int TMEM_COLS = NO * 128 + 2 * KB;
  static constexpr uint32_t S_COL0 = NO * 128;   // S/P buffers after the O buffers
  static constexpr int Q_BYTES = BQ * HD * 2;
  static constexpr int K_BYTES = KB * HD * 2;
  static constexpr int V_BYTES = KB * HD * 2;
  static constexpr size_t SMEM = (size_t)Q_BYTES + NST * (K_BYTES + V_BYTES) + 1024 + 512;
  // kind::f16 instruction descriptors: fp32 D, fp16 A and B, M = 128.
  // S = Q K^T: both K-major, N = KB keys.  O += P V: P K-major (in TMEM), V MN-major (bit 16),
  // N = HD.
  static constexpr uint32_t IDESC_S = (1u << 4) | ((uint32_t)(KB >> 3) << 17) | ((uint32_t)(BQ >> 4) << 24);
  static constexpr uint32_t IDESC_O =
      (1u << 4) | (1u << 16) | ((uint32_t)(HD >> 3) << 17) | ((uint32_t)(BQ >> 4) << 24);
  static_assert(TMEM_COLS == 256 || TMEM_COLS == 512, "TMEM allocation must be a power of two");
  static_assert(SMEM * CTAS <= 232448, "shared memory per SM");
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
// K-major, 128B swizzle: rows of 128 B, 8-row groups 1024 B apart (stride byte offset).
__device__ __forceinline__ uint64_t desc_kmajor(uint32_t addr) {
  return (uint64_t)((addr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
// MN-major, 128B swizzle: 64 contiguous MN elements (128 B) per row, 8 K-rows per 1024 B group
// (stride byte offset 1024), the next 64-wide MN block `lbo` bytes on (leading byte offset).
__device__ __forceinline__ uint64_t desc_mnmajor(uint32_t addr, uint32_t lbo) {
  return (uint64_t)((addr & 0x3FFFFu) >> 4) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
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
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  if (mbar_try_wait(bar, parity)) return true;
  uint64_t t0;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t0));
  for (uint32_t i = 0; i < RIFT_SPIN_LIMIT; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 255u) == 255u) {
      if (*abort_flag) return false;
      uint64_t t;
      asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
      if (t - t0 > 4000000000ull) break;
    }
  }
  atomicOr(&g_err_attn, RIFT_EBIT_TIMEOUT);
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
__device__ __forceinline__ void umma(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t accum) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(idesc), "r"(accum));
}
// A from tensor memory (TS form): row i of A in lane i, two fp16 per 32-bit column.
__device__ __forceinline__ void umma_ts(uint32_t tmem_d, uint32_t tmem_a, uint64_t b, uint32_t idesc, uint32_t accum) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(tmem_d),
      "r"(tmem_a), "l"(b), "r"(idesc), "r"(accum));
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(bar)
               : "memory");
}
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};\n" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]),
      "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]),
      "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
// 2^x on the special-function unit (flushes subnormal results to zero).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Three-input maximum and packed pairs of fp32 (Blackwell's f32x2 FMA-pipe forms).
__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
__device__ __forceinline__ uint64_t f2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ float2 unf2(uint64_t v) {
  float2 r;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(r.x), "=f"(r.y) : "l"(v));
  return r;
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};\n" ::"r"(
          taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

// 32-byte global store (address 32-byte aligned).
__device__ __forceinline__ void st_global_v8(void* p, const uint32_t* r) {
  asm volatile("st.global.v8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};\n" ::"l"(p), "r"(r[0]), "r"(r[1]), "r"(r[2]),
               "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
               : "memory");
}

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;\n" ::: "memory"); }

// Item i -> (schedule entry, head): entries are q-blocks (sequence, first row); heads inner.
template <int HD, int KB>
__global__ void __launch_bounds__(THREADS, Cfg<HD, KB>::CTAS)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kv,
                   const __grid_constant__ CUtensorMap tm_pk, const __grid_constant__ CUtensorMap tm_pv, int S_pre,
                   const int4* __restrict__ sched, int n_entries, int H, float scale_log2,
                   uint16_t* __restrict__ out) {
  using CF = Cfg<HD, KB>;
  constexpr int NST = CF::NST, NO = CF::NO, NC = KB / 32;  // NC: 32-key chunks per block
  constexpr uint32_t S_COL0 = CF::S_COL0;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sK = smem + CF::Q_BYTES;             // stage s at sK + s * K_BYTES
  uint8_t* sV = sK + NST * CF::K_BYTES;         // stage s at sV + s * V_BYTES
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV + NST * CF::V_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 32);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t b0 = smem_u32(bars);
  // barrier k lives at b0 + 8 k; rings and buffers are indexed by the stage or buffer
  const uint32_t Q_FULL = b0, Q_EMPTY = b0 + 8;
  auto BAR = [&](int base, int i) { return b0 + 8u * (uint32_t)(base + i); };
  enum { K_FULL = 2, K_EMPTY = K_FULL + NST, V_FULL = K_EMPTY + NST, V_EMPTY = V_FULL + NST, S_FULL = V_EMPTY + NST,
         P_FULL = S_FULL + 2, PV_DONE = P_FULL + 2, O_FULL = PV_DONE + 2, O_EMPTY = O_FULL + NO, N_BARS = O_EMPTY + NO };
  static_assert(N_BARS <= 32, "barrier slots");

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(Q_FULL, 1);
    mbar_init(Q_EMPTY, 1);
    for (int b = 0; b < NST; ++b) {
      mbar_init(BAR(K_FULL, b), 1);
      mbar_init(BAR(K_EMPTY, b), 1);
      mbar_init(BAR(V_FULL, b), 1);
      mbar_init(BAR(V_EMPTY, b), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(BAR(S_FULL, b), 1);
      mbar_init(BAR(P_FULL, b), 128);
      mbar_init(BAR(PV_DONE, b), 1);
    }
    for (int b = 0; b < NO; ++b) {
      mbar_init(BAR(O_FULL, b), 1);
      mbar_init(BAR(O_EMPTY, b), 128);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(tmem_slot)),
                 "r"(CF::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tmem_slot;
  const int n_items = min(n_entries, sched[n_entries].x) * H;  // entries in use (the schedule's count)
  const int d = H * HD;
  const int np = (S_pre + KB - 1) / KB;  // prefix blocks ahead of every sequence's own

  // An item's sequence start, length, first row, head and number of KB-key blocks (causal:
  // keys up to the block's last valid row).  Every role fetches the next item's schedule entry
  // (one 16-byte load, no branch on it) while it works on the current one, and decodes it only
  // when that item starts, so the load's latency is hidden behind a whole item.
  struct Item {
    int seq0, L, q0, h, nkv;
  };
  auto fetch_item = [&](int item) -> int4 {
    return item < n_items ? sched[item / H] : make_int4(0, 0, 0, 0);
  };
  auto decode_item = [&](const int4& e, int item) -> Item {
    Item it;
    it.h = item % H;
    it.seq0 = e.x;
    it.L = e.y;
    it.q0 = e.z;
    it.nkv = (item < n_items && e.y > 0) ? np + (min(e.y, e.z + BQ) - 1) / KB + 1 : 0;
    return it;
  };
  // Counters shared by every role: g counts KB-key blocks, t counts items of this CTA.  Block g
  // uses K/V stage g % NST (phase (g / NST) & 1) and S/P buffer g & 1 (phase (g >> 1) & 1); item t
  // uses O buffer t % NO (phase (t / NO) & 1).

  if (warp == 0) {
    if (lane < 2) {
      // ---------------- TMA producers: lane 0 K tiles; lane 1 Q and V tiles
      uint32_t g = 0, t = 0;
      bool ok = true;
      int4 nxt = fetch_item(blockIdx.x);
      for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
        const Item cur = decode_item(nxt, item);
        nxt = fetch_item(item + gridDim.x);
        if (cur.nkv == 0) continue;
        if (lane == 1) {
          if (!mbar_wait(Q_EMPTY, (t & 1u) ^ 1u, abort_flag)) { ok = false; break; }
          mbar_expect_tx(Q_FULL, CF::Q_BYTES);
          for (int c = 0; c < HD / 64; ++c)
            tma_load_2d(smem_u32(sQ + c * BQ * 128), &tm_q, cur.h * HD + c * 64, cur.seq0 + cur.q0, Q_FULL);
        }
        for (int j = 0; j < cur.nkv; ++j, ++g) {
          const int s = g % NST;
          const uint32_t ph = (g / NST) & 1u;
          const int base = lane == 0 ? K_EMPTY : V_EMPTY;
          if (!mbar_wait(BAR(base, s), ph ^ 1u, abort_flag)) { ok = false; break; }
          const uint32_t full = BAR(lane == 0 ? K_FULL : V_FULL, s);
          mbar_expect_tx(full, CF::K_BYTES);
          uint8_t* dst = (lane == 0 ? sK + s * CF::K_BYTES : sV + s * CF::V_BYTES);
          // prefix blocks from the prefix's [S_pre, d] K / V maps (rows past S_pre read as zero),
          // then the sequence's own rows of the qkv map
          const bool pre = j < np;
          const CUtensorMap* map = pre ? (lane == 0 ? &tm_pk : &tm_pv) : &tm_kv;
          const int col = (pre ? 0 : (lane == 0 ? d : 2 * d)) + cur.h * HD;
          const int row = pre ? j * KB : cur.seq0 + (j - np) * KB;
          for (int c = 0; c < HD / 64; ++c) tma_load_2d(smem_u32(dst + c * KB * 128), map, col + c * 64, row, full);
        }
        ++t;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      uint32_t g = 0, t = 0;
      bool ok = true;
      auto issue_s = [&](uint32_t gg) -> bool {
        const int st = gg % NST, sb = gg & 1;
        if (!mbar_wait(BAR(K_FULL, st), (gg / NST) & 1u, abort_flag)) return false;
        // S/P buffer sb is free once PV_{gg-2}, the reader of P_{gg-2}, has completed
        if (gg >= 2 && !mbar_wait(BAR(PV_DONE, sb), ((gg - 2) >> 1) & 1u, abort_flag)) return false;
        fence_after();
        const uint32_t kb = smem_u32(sK + st * CF::K_BYTES);
        const uint32_t qb = smem_u32(sQ);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {  // 16 of the head dims per step
          const uint32_t koff = (kk & 3) * 32;
          umma(tmem + S_COL0 + (uint32_t)KB * sb, desc_kmajor(qb + (kk >> 2) * (BQ * 128) + koff),
               desc_kmajor(kb + (kk >> 2) * (KB * 128) + koff), CF::IDESC_S, kk > 0);
        }
        umma_commit(BAR(S_FULL, sb));
        umma_commit(BAR(K_EMPTY, st));
        return true;
      };
      int4 nxt = fetch_item(blockIdx.x);
      for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
        const int nkv = decode_item(nxt, item).nkv;
        nxt = fetch_item(item + gridDim.x);
        if (nkv == 0) continue;
        const int ob = t % NO;
        if (!mbar_wait(Q_FULL, t & 1u, abort_flag)) break;
        fence_after();
        if (!issue_s(g)) break;
        for (int j = 0; j < nkv; ++j, ++g) {
          if (j + 1 < nkv) {
            if (!issue_s(g + 1)) { ok = false; break; }
          } else {
            umma_commit(Q_EMPTY);  // Q is free once the item's S products complete
          }
          const int st = g % NST, sb = g & 1;
          if (!mbar_wait(BAR(P_FULL, sb), (g >> 1) & 1u, abort_flag)) { ok = false; break; }
          if (j == 0 && !mbar_wait(BAR(O_EMPTY, ob), ((t / NO) & 1u) ^ 1u, abort_flag)) { ok = false; break; }
          if (!mbar_wait(BAR(V_FULL, st), (g / NST) & 1u, abort_flag)) { ok = false; break; }
          fence_after();
          const uint32_t vb = smem_u32(sV + st * CF::V_BYTES);
#pragma unroll
          for (int kk = 0; kk < KB / 16; ++kk) {  // 16 keys (8 TMEM columns of P) per step
            const uint64_t bdesc = desc_mnmajor(vb + kk * 2048, KB * 128);
            umma_ts(tmem + 128u * ob, tmem + S_COL0 + (uint32_t)KB * sb + 8u * kk, bdesc, CF::IDESC_O,
                    (j > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit(BAR(PV_DONE, sb));
          umma_commit(BAR(V_EMPTY, st));
        }
        if (!ok) break;
        umma_commit(BAR(O_FULL, ob));
        ++t;
      }
    }
  } else {
    // ---------------- softmax and output: thread = query row (TMEM lane)
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t lane_base = tmem + ((uint32_t)(quarter * 32) << 16);
    uint32_t g = 0, t = 0;
    bool ok = true;
    int4 nxt = fetch_item(blockIdx.x);
    for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
      const Item cur = decode_item(nxt, item);
      nxt = fetch_item(item + gridDim.x);
      const int L = cur.L, q0 = cur.q0, nkv = cur.nkv;
      if (nkv == 0) continue;
      const int ob = t % NO;
      const uint32_t o_base = lane_base + 128u * ob;
      const int qrow = q0 + r;  // row within the sequence
      float m = -INFINITY, l = 0.f;  // running maximum (log2 units, scaled) and sum
      for (int j = 0; j < nkv; ++j, ++g) {
        const int sb = g & 1;
        if (!mbar_wait(BAR(S_FULL, sb), (g >> 1) & 1u, abort_flag)) { ok = false; break; }
        fence_after();
        const uint32_t sbase = lane_base + S_COL0 + (uint32_t)KB * sb;
        uint32_t sv[NC][32];
#pragma unroll
        for (int c = 0; c < NC; ++c) tmem_ld32(sbase + 32u * c, sv[c]);
        tmem_wait_ld();
        // Own blocks: only the diagonal blocks and the block holding the sequence end need the
        // mask, key valid iff key <= qrow and key < L (uniform over the CTA).  Prefix blocks: key
        // valid iff key < S_pre.  Within a masked block a 32-key chunk is touched only where some
        // row of the warp ends inside or before it.
        const bool pre = j < np;
        const int k0 = pre ? j * KB : (j - np) * KB;
        if (pre ? k0 + KB > S_pre : (k0 + KB - 1 > q0 || k0 + KB > L)) {
          const int lim = pre ? S_pre - 1 - k0 : min(qrow, L - 1) - k0;  // last valid column of this row
#pragma unroll
          for (int c = 0; c < NC; ++c)
            if (__any_sync(0xffffffffu, lim < 32 * c + 31)) {
#pragma unroll
              for (int e = 0; e < 32; ++e)
                if (32 * c + e > lim) sv[c][e] = __float_as_uint(-INFINITY);
            }
        }
        // row maximum over four independent chains of three-input maxima
        float mc[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int c = 0; c < NC; ++c)
#pragma unroll
          for (int e = 0; e < 32; e += 2)
            mc[(e >> 1) & 3] = max3(mc[(e >> 1) & 3], __uint_as_float(sv[c][e]), __uint_as_float(sv[c][e + 1]));
        float mx = max3(fmaxf(mc[0], mc[1]), mc[2], mc[3]);
        mx *= scale_log2;  // scale > 0: the maximum of the scaled scores
        float m_use = m, corr = 1.f;
        if (j == 0) {
          m_use = mx;
        } else if (mx > m + STALE) {
          m_use = mx;
          corr = ex2(m - mx);
        }
        const float nb = (m_use == -INFINITY) ? 0.f : -m_use;  // p = 2^(s * scale - m)
        const uint64_t sc2 = f2(scale_log2, scale_log2), nb2 = f2(nb, nb);
        uint64_t acc[4] = {0, 0, 0, 0};  // four independent pair sums (0 is +0.0f, +0.0f)
        // P_g as packed fp16 over the first KB / 2 columns of S buffer sb, 32 keys (16 columns) at
        // a time: chunk c lands in columns [16c, 16c + 16), whose S values are already in
        // registers (PV_{g-2}, the previous reader of these columns, completed before S_g was
        // issued)
#pragma unroll
        for (int c = 0; c < NC; ++c) {
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            const float2 x = unf2(fma2(f2(__uint_as_float(sv[c][e]), __uint_as_float(sv[c][e + 1])), sc2, nb2));
            const float p0 = ex2(x.x), p1 = ex2(x.y);
            acc[(e >> 1) & 3] = add2(acc[(e >> 1) & 3], f2(p0, p1));
            pk[e / 2] = pack_half2(p0, p1);
          }
          tmem_st16(sbase + 16u * c, pk);
        }
        const float2 a01 = unf2(add2(acc[0], acc[1])), a23 = unf2(add2(acc[2], acc[3]));
        const float rs = (a01.x + a01.y) + (a23.x + a23.y);
        if (__any_sync(0xffffffffu, corr != 1.f)) {  // rare: rescale this warp's O rows
          // O must hold PV_{g-1} complete (j >= 1 here) before it is rescaled
          if (!mbar_wait(BAR(PV_DONE, (g - 1) & 1), ((g - 1) >> 1) & 1u, abort_flag)) { ok = false; break; }
          fence_after();
#pragma unroll 1
          for (int c = 0; c < HD / 32; ++c) {
            uint32_t ov[32];
            tmem_ld32(o_base + 32u * c, ov);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 32; ++e) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * corr);
            tmem_st32(o_base + 32u * c, ov);
          }
        }
        l = l * corr + rs;
        m = m_use;
        tmem_wait_st();
        fence_before();
        mbar_arrive(BAR(P_FULL, sb));
      }
      if (!ok) break;
      // output: wait for the item's last PV product, O / l
      if (!mbar_wait(BAR(O_FULL, ob), (t / NO) & 1u, abort_flag)) break;
      fence_after();
      const float inv = 1.f / l;
      uint16_t* dst = out + (size_t)(cur.seq0 + qrow) * d + cur.h * HD;
      const bool v8 = (reinterpret_cast<uintptr_t>(out) & 31u) == 0;  // rows then start on 32 B
#pragma unroll 1
      for (int c = 0; c < HD / 32; ++c) {
        uint32_t ov[32];
        tmem_ld32(o_base + 32u * c, ov);
        tmem_wait_ld();
        uint32_t hv[16];
#pragma unroll
        for (int q = 0; q < 16; ++q) hv[q] = pack_half2(__uint_as_float(ov[2 * q]) * inv, __uint_as_float(ov[2 * q + 1]) * inv);
        if (qrow < L) {
          if (v8) {  // one full 32-byte sector per row and store
#pragma unroll
            for (int q = 0; q < 2; ++q)
              st_global_v8(dst + 32 * c + 16 * q, hv + 8 * q);
          } else {
            uint4* d4 = reinterpret_cast<uint4*>(dst + 32 * c);
#pragma unroll
            for (int q = 0; q < 4; ++q) d4[q] = make_uint4(hv[4 * q], hv[4 * q + 1], hv[4 * q + 2], hv[4 * q + 3]);
          }
        }
      }
      fence_before();
      mbar_arrive(BAR(O_EMPTY, ob));
      ++t;
    }
  }
  fence_before();
  __syncthreads();
  if (warp == 1) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem), "r"(CF::TMEM_COLS) : "memory");
  }
}

// One entry per 128-row q-block: (first row of its sequence in the packed batch, sequence length,
// first row of the block within the sequence, 0); the rest (0, 0, 0, 0), which the kernel skips.
// Entry n_max holds the number of entries in use (.x), so the attention visits only those.  The
// sequence count is n_seq_dev's value when given (a count written by an earlier kernel), clamped
// to n_seq; a sequence that ends past row_cap (the rows the buffers hold) and the sequences after
// it are left out and RIFT_EBIT_CAPACITY is set.  Longer sequences' entries are not reordered:
// items are interleaved across CTAs by the persistent loop.
__global__ void __launch_bounds__(1024) schedule128_kernel(const int* __restrict__ cu, int n_seq,
                                                           const int* __restrict__ n_seq_dev, int row_cap,
                                                           int4* __restrict__ sched, int n_max) {
  __shared__ int sh[33];
  __shared__ int s_cut;
  int n = n_seq;
  if (n_seq_dev) {
    const int nd = *n_seq_dev;
    if (nd > n_seq && threadIdx.x == 0) atomicOr(&g_err_attn, RIFT_EBIT_CAPACITY);
    n = max(0, min(n_seq, nd));
  }
  if (threadIdx.x == 0) s_cut = n;
  __syncthreads();
  // the first sequence that does not fit in row_cap rows ends the schedule
  for (int s = threadIdx.x; s < n; s += blockDim.x)
    if (cu[s + 1] > row_cap || cu[s + 1] < cu[s]) atomicMin(&s_cut, s);
  __syncthreads();
  if (s_cut < n) {
    if (threadIdx.x == 0) atomicOr(&g_err_attn, RIFT_EBIT_CAPACITY);
    n = s_cut;
  }
  int base = 0;
  for (int c0 = 0; c0 < n; c0 += blockDim.x) {
    const int s = c0 + threadIdx.x;
    int nb = 0, s0 = 0, len = 0;
    if (s < n) {
      s0 = cu[s];
      len = cu[s + 1] - s0;
      nb = (len + BQ - 1) / BQ;
    }
    int total;
    int off = block_excl_scan(nb, sh, &total);
    for (int b = 0; b < nb; ++b)
      if (base + off + b < n_max) sched[base + off + b] = make_int4(s0, len, b * BQ, 0);
    base += total;
  }
  for (int i = base + threadIdx.x; i < n_max; i += blockDim.x) sched[i] = make_int4(0, 0, 0, 0);
  if (threadIdx.x == 0) sched[n_max] = make_int4(min(base, n_max), 0, 0, 0);
}

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

}  // namespace fa

// q-block schedule of the tcgen05 attention (one entry per 128 rows of a sequence)
void launch_attention_schedule(const int* cu_seqlens, int n_seq, const int* n_seq_dev, int row_cap, int4* sched,
                               int n_sched_max, cudaStream_t st) {
  fa::schedule128_kernel<<<1, 1024, 0, st>>>(cu_seqlens, n_seq, n_seq_dev, row_cap, sched, n_sched_max);
}

int attention_max_qblocks(int max_T, int max_seqs) { return (max_T + fa::BQ - 1) / fa::BQ + max_seqs; }

namespace {

// Keys per block of the launched kernel shape (64: two CTAs per SM; 128: one).
constexpr int kAttnKB = 64;

template <int HD, int KB>
int launch_shape(const CUtensorMap& mq, const CUtensorMap& mkv, const CUtensorMap& mpk, const CUtensorMap& mpv,
                 int S_pre, const int4* sched, int n_sched_max, int n_heads, float scale_log2, void* out,
                 cudaStream_t st) {
  using namespace fa;
  using CF = Cfg<HD, KB>;
  static std::atomic<unsigned long long> smem_raised{0};
  if (raise_smem_limit(smem_raised, attn_tc_kernel<HD, KB>, (int)CF::SMEM) != cudaSuccess) return 1;
  const int items = n_sched_max * n_heads;
  const int slots = CF::CTAS * sm_count();
  const int grid = items < slots ? items : slots;
  attn_tc_kernel<HD, KB><<<grid, THREADS, CF::SMEM, st>>>(mq, mkv, mpk, mpv, S_pre, sched, n_sched_max, n_heads,
                                                          scale_log2, static_cast<uint16_t*>(out));
  return 0;
}

// fp16 [rows, cols] (row-major) as a 2-D tensor map of 64-column x box_rows boxes, 128B swizzle.
bool make_attn_map(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows) {
  auto fn = fa::encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

// qkv fp16 [T, 3 H hd] (q | k | v, heads contiguous), out fp16 [T, H hd]; optional prefix keys and
// values fp16 [S_pre, H hd] attended to by every sequence before its own rows.
int launch_attention(const void* qkv, int T, const int* cu_seqlens, int n_seq, int n_heads, int head_dim,
                     const int4* sched, int n_sched_max, void* out, cudaStream_t st, const void* prefix_k,
                     const void* prefix_v, int S_pre) {
  using namespace fa;
  (void)n_seq;
  (void)cu_seqlens;  // the schedule entries carry the sequence bounds
  if (T <= 0) return 0;
  if (head_dim != 64 && head_dim != 128) return 1;
  if (S_pre > 0 && (!prefix_k || !prefix_v)) return 1;
  const int d = n_heads * head_dim;
  // Q tiles of 128 rows and K/V tiles of kAttnKB rows, each a 64-column (128-byte) box
  CUtensorMap mq, mkv, mpk, mpv;
  if (!make_attn_map(&mq, qkv, 3 * d, T, BQ) || !make_attn_map(&mkv, qkv, 3 * d, T, kAttnKB)) return 1;
  if (S_pre > 0) {
    if (!make_attn_map(&mpk, prefix_k, d, S_pre, kAttnKB) || !make_attn_map(&mpv, prefix_v, d, S_pre, kAttnKB)) return 1;
  } else {
    mpk = mkv;  // unused without a prefix
    mpv = mkv;
  }
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)head_dim);
  if (head_dim == 128)
    return launch_shape<128, kAttnKB>(mq, mkv, mpk, mpv, S_pre, sched, n_sched_max, n_heads, scale_log2, out, st);
  return launch_shape<64, kAttnKB>(mq, mkv, mpk, mpv, S_pre, sched, n_sched_max, n_heads, scale_log2, out, st);
}

}  // namespace rift
