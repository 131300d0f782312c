// Varlen causal attention on Blackwell's tcgen05 tensor cores (sm_103a).
//
// Work item = (128-row q-block of one packed sequence, one head).  Persistent CTAs (one per SM)
// walk the items; tensor memory and barriers are set up once per CTA.  Per CTA, 192 threads:
//   warp 0      TMA: the item's Q tile, then K and V tiles of 128 keys into two stages
//               (fp16, 128B swizzle; a 128-column box pair per 128-wide head)
//   warp 1      one thread issues S_j = Q K_j^T (M = 128, N = 128 keys) into one of two TMEM
//               S buffers, and O += P_j V_j (N = head_dim, V read as an MN-major operand)
//   warps 2..5  softmax, one query row per thread (TMEM lane = row): scale, causal and
//               sequence-end mask, online softmax with a stale maximum (O is rescaled in TMEM
//               only when a row's maximum grows by more than 2^8), P_j written as fp16 into a
//               swizzled shared tile for the PV product; at the end O / l is stored as fp16.
// TMEM: O in columns [0, 128), S buffers at 128 and 256.  Every mbarrier wait is bounded; on
// timeout the kernel sets RIFT_EBIT_TIMEOUT and every role falls through.
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

constexpr int BQ = 128, BKV = 128, THREADS = 192;
constexpr int TMEM_COLS = 512;
constexpr uint32_t S_COL0 = 128;  // S buffers at columns 128 and 256; O at 0
constexpr float STALE = 8.f;      // log2 units: P <= 2^8 before a rescale is forced

template <int HD>
struct Cfg {
  static constexpr int Q_BYTES = BQ * HD * 2;
  static constexpr int K_BYTES = BKV * HD * 2;
  static constexpr int V_BYTES = BKV * HD * 2;
  static constexpr int P_BYTES = BQ * BKV * 2;
  static constexpr int STAGE = K_BYTES + V_BYTES;
  static constexpr size_t SMEM = (size_t)Q_BYTES + 2 * STAGE + P_BYTES + 1024 + 256;
  // kind::f16 instruction descriptors: fp32 D, fp16 A and B, M = 128.
  // S = Q K^T: both K-major, N = 128 keys.  O += P V: P K-major, V MN-major (bit 16), N = HD.
  static constexpr uint32_t IDESC_S = (1u << 4) | ((uint32_t)(BKV >> 3) << 17) | ((uint32_t)(BQ >> 4) << 24);
  static constexpr uint32_t IDESC_O =
      (1u << 4) | (1u << 16) | ((uint32_t)(HD >> 3) << 17) | ((uint32_t)(BQ >> 4) << 24);
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

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;\n" ::: "memory"); }

// Item i -> (schedule entry, head): entries are q-blocks (sequence, first row); heads inner.
template <int HD>
__global__ void __launch_bounds__(THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm, const int* __restrict__ cu, const int2* __restrict__ sched,
                   int n_entries, int H, float scale_log2, uint16_t* __restrict__ out) {
  using CF = Cfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sKV = smem + CF::Q_BYTES;                 // stage s: K at sKV + s*STAGE, V after it
  uint8_t* sP = sKV + 2 * CF::STAGE;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sP + CF::P_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 16);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t b0 = smem_u32(bars);
  const uint32_t Q_FULL = b0, Q_EMPTY = b0 + 8, P_FULL = b0 + 16, PV_DONE = b0 + 24, O_EMPTY = b0 + 32;
  auto KV_FULL = [&](int s) { return b0 + 40 + 8u * s; };
  auto KV_EMPTY = [&](int s) { return b0 + 56 + 8u * s; };
  auto S_FULL = [&](int s) { return b0 + 72 + 8u * s; };
  auto S_EMPTY = [&](int s) { return b0 + 88 + 8u * s; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(Q_FULL, 1);
    mbar_init(Q_EMPTY, 1);
    mbar_init(P_FULL, 128);
    mbar_init(PV_DONE, 1);
    mbar_init(O_EMPTY, 128);
    for (int s = 0; s < 2; ++s) {
      mbar_init(KV_FULL(s), 1);
      mbar_init(KV_EMPTY(s), 1);
      mbar_init(S_FULL(s), 1);
      mbar_init(S_EMPTY(s), 128);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tmem_slot;
  const int n_items = n_entries * H;
  const int d = H * HD;

  // An item's sequence start, length, first row, head and number of 128-key blocks (causal:
  // keys up to the block's last valid row).  Every role reads the next item's entry while it
  // works on the current one.
  struct Item {
    int seq0, L, q0, h, nkv;
  };
  auto load_item = [&](int item) -> Item {
    Item it{0, 0, 0, 0, 0};
    if (item >= n_items) return it;
    const int2 e = sched[item / H];
    it.h = item % H;
    if (e.x < 0) return it;
    it.seq0 = cu[e.x];
    it.L = cu[e.x + 1] - it.seq0;
    it.q0 = e.y;
    it.nkv = (min(it.L, it.q0 + BQ) - 1) / BKV + 1;
    return it;
  };

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      uint32_t g = 0, it_local = 0;
      bool ok = true;
      Item nxt = load_item(blockIdx.x);
      for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
        const Item cur = nxt;
        nxt = load_item(item + gridDim.x);
        const int seq0 = cur.seq0, q0 = cur.q0, h = cur.h, nkv = cur.nkv;
        if (nkv == 0) continue;
        if (!mbar_wait(Q_EMPTY, (it_local & 1u) ^ 1u, abort_flag)) { ok = false; break; }
        mbar_expect_tx(Q_FULL, CF::Q_BYTES);
        for (int c = 0; c < HD / 64; ++c)
          tma_load_2d(smem_u32(sQ + c * BQ * 128), &tm, h * HD + c * 64, seq0 + q0, Q_FULL);
        for (int j = 0; j < nkv; ++j, ++g) {
          const int s = g & 1;
          if (!mbar_wait(KV_EMPTY(s), ((g >> 1) & 1u) ^ 1u, abort_flag)) { ok = false; break; }
          mbar_expect_tx(KV_FULL(s), CF::STAGE);
          uint8_t* sK = sKV + s * CF::STAGE;
          uint8_t* sV = sK + CF::K_BYTES;
          for (int c = 0; c < HD / 64; ++c) {
            tma_load_2d(smem_u32(sK + c * BKV * 128), &tm, d + h * HD + c * 64, seq0 + j * BKV, KV_FULL(s));
            tma_load_2d(smem_u32(sV + c * BKV * 128), &tm, 2 * d + h * HD + c * 64, seq0 + j * BKV, KV_FULL(s));
          }
        }
        ++it_local;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      uint32_t g = 0, it_local = 0;
      bool ok = true;
      auto issue_s = [&](uint32_t gg) -> bool {
        const int s = gg & 1;
        if (!mbar_wait(KV_FULL(s), (gg >> 1) & 1u, abort_flag)) return false;
        if (!mbar_wait(S_EMPTY(s), ((gg >> 1) & 1u) ^ 1u, abort_flag)) return false;
        fence_after();
        const uint32_t sK = smem_u32(sKV + s * CF::STAGE);
        const uint32_t sQa = smem_u32(sQ);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {  // 16 of the head dims per step
          const uint32_t off = (kk >> 2) * (BQ * 128) + (kk & 3) * 32;
          umma(tmem + S_COL0 + 128u * s, desc_kmajor(sQa + off), desc_kmajor(sK + off), CF::IDESC_S, kk > 0);
        }
        umma_commit(S_FULL(s));
        return true;
      };
      Item nxt = load_item(blockIdx.x);
      for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
        const int nkv = nxt.nkv;
        nxt = load_item(item + gridDim.x);
        if (nkv == 0) continue;
        if (!mbar_wait(Q_FULL, it_local & 1u, abort_flag)) break;
        fence_after();
        if (!issue_s(g)) break;
        for (int j = 0; j < nkv; ++j, ++g) {
          if (j + 1 < nkv) {
            if (!issue_s(g + 1)) { ok = false; break; }
          } else {
            umma_commit(Q_EMPTY);  // Q is free once the item's S products complete
          }
          if (!mbar_wait(P_FULL, g & 1u, abort_flag)) { ok = false; break; }
          if (j == 0 && !mbar_wait(O_EMPTY, (it_local & 1u) ^ 1u, abort_flag)) { ok = false; break; }
          fence_after();
          const int s = g & 1;
          const uint32_t sV = smem_u32(sKV + s * CF::STAGE + CF::K_BYTES);
          const uint32_t sPa = smem_u32(sP);
#pragma unroll
          for (int kk = 0; kk < BKV / 16; ++kk) {  // 16 keys per step
            const uint64_t a = desc_kmajor(sPa + (kk >> 2) * (BQ * 128) + (kk & 3) * 32);
            const uint64_t b = desc_mnmajor(sV + kk * 2048, BKV * 128);
            umma(tmem, a, b, CF::IDESC_O, (j > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit(PV_DONE);
          umma_commit(KV_EMPTY(s));
        }
        ++it_local;
      }
    }
  } else {
    // ---------------- softmax: thread = query row (TMEM lane)
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t lane_base = tmem + ((uint32_t)(quarter * 32) << 16);
    uint32_t g = 0, it_local = 0;
    bool ok = true;
    Item nxt = load_item(blockIdx.x);
    for (int item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
      const Item cur = nxt;
      nxt = load_item(item + gridDim.x);
      const int seq0 = cur.seq0, L = cur.L, q0 = cur.q0, h = cur.h, nkv = cur.nkv;
      if (nkv == 0) continue;
      const int qrow = q0 + r;  // row within the sequence
      float m = -INFINITY, l = 0.f;  // running maximum (log2 units, scaled) and sum
      for (int j = 0; j < nkv; ++j, ++g) {
        const int s = g & 1;
        if (!mbar_wait(S_FULL(s), (g >> 1) & 1u, abort_flag)) { ok = false; break; }
        fence_after();
        uint32_t sv[4][32];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(lane_base + S_COL0 + 128u * s + 32u * c, sv[c]);
        tmem_wait_ld();
        fence_before();
        mbar_arrive(S_EMPTY(s));
        const int k0 = j * BKV;
        // Only the diagonal block and the block holding the sequence end need the mask: key
        // valid iff key <= qrow and key < L (this branch is uniform over the CTA).
        if (k0 + BKV - 1 > q0 || k0 + BKV > L) {
          const int lim = min(qrow, L - 1) - k0;  // last valid column of this row
#pragma unroll
          for (int c = 0; c < 4; ++c)
#pragma unroll
            for (int e = 0; e < 32; ++e)
              if (32 * c + e > lim) sv[c][e] = __float_as_uint(-INFINITY);
        }
        float mx = -INFINITY;
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int e = 0; e < 32; ++e) mx = fmaxf(mx, __uint_as_float(sv[c][e]));
        mx *= scale_log2;  // scale > 0: the maximum of the scaled scores
        float m_use = m, corr = 1.f;
        if (j == 0) {
          m_use = mx;
        } else if (mx > m + STALE) {
          m_use = mx;
          corr = ex2(m - mx);
        }
        const float nb = (m_use == -INFINITY) ? 0.f : -m_use;  // p = 2^(s * scale - m)
        float rs = 0.f;
        uint32_t pk[64];
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            const float p0 = ex2(fmaf(__uint_as_float(sv[c][e]), scale_log2, nb));
            const float p1 = ex2(fmaf(__uint_as_float(sv[c][e + 1]), scale_log2, nb));
            rs += p0 + p1;
            pk[c * 16 + e / 2] = pack_half2(p0, p1);
          }
        // P buffer and O are free once the previous PV product completed
        if (g > 0 && !mbar_wait(PV_DONE, (g - 1) & 1u, abort_flag)) { ok = false; break; }
        fence_after();
        if (__any_sync(0xffffffffu, corr != 1.f)) {  // rare: rescale this warp's O rows
#pragma unroll 1
          for (int c = 0; c < HD / 32; ++c) {
            uint32_t ov[32];
            tmem_ld32(lane_base + 32u * c, ov);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 32; ++e) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * corr);
            tmem_st32(lane_base + 32u * c, ov);
          }
          tmem_wait_st();
        }
        l = l * corr + rs;
        m = m_use;
        // P row r: 16 chunks of 8 fp16; chunk c lives in key-atom c/8 at position (c%8)^(r%8)
#pragma unroll
        for (int c = 0; c < 16; ++c) {
          uint8_t* dst = sP + (c >> 3) * (BQ * 128) + r * 128 + ((((c & 7) ^ (r & 7))) << 4);
          *reinterpret_cast<uint4*>(dst) = make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
        }
        asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
        fence_before();
        mbar_arrive(P_FULL);
      }
      if (!ok) break;
      // output: wait for the item's last PV product, O / l
      if (!mbar_wait(PV_DONE, (g - 1) & 1u, abort_flag)) break;
      fence_after();
      const float inv = 1.f / l;
      uint16_t* dst = out + (size_t)(seq0 + qrow) * d + h * HD;
#pragma unroll 1
      for (int c = 0; c < HD / 32; ++c) {
        uint32_t ov[32];
        tmem_ld32(lane_base + 32u * c, ov);
        tmem_wait_ld();
        if (qrow < L) {
          uint4* d4 = reinterpret_cast<uint4*>(dst + 32 * c);
#pragma unroll
          for (int q = 0; q < 4; ++q)
            d4[q] = make_uint4(pack_half2(__uint_as_float(ov[8 * q]) * inv, __uint_as_float(ov[8 * q + 1]) * inv),
                               pack_half2(__uint_as_float(ov[8 * q + 2]) * inv, __uint_as_float(ov[8 * q + 3]) * inv),
                               pack_half2(__uint_as_float(ov[8 * q + 4]) * inv, __uint_as_float(ov[8 * q + 5]) * inv),
                               pack_half2(__uint_as_float(ov[8 * q + 6]) * inv, __uint_as_float(ov[8 * q + 7]) * inv));
        }
      }
      fence_before();
      mbar_arrive(O_EMPTY);
      ++it_local;
    }
  }
  fence_before();
  __syncthreads();
  if (warp == 1) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
  }
}

// One entry per 128-row q-block, (sequence, first row); the rest (-1, 0).  Longer sequences'
// entries are not reordered: items are interleaved across CTAs by the persistent loop.
__global__ void __launch_bounds__(1024) schedule128_kernel(const int* __restrict__ cu, int n_seq,
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
void launch_attention_schedule(const int* cu_seqlens, int n_seq, int2* sched, int n_sched_max, cudaStream_t st) {
  fa::schedule128_kernel<<<1, 1024, 0, st>>>(cu_seqlens, n_seq, sched, n_sched_max);
}

int attention_max_qblocks(int max_T, int max_seqs) { return (max_T + fa::BQ - 1) / fa::BQ + max_seqs; }

// qkv fp16 [T, 3 H hd] (q | k | v, heads contiguous), out fp16 [T, H hd].
int launch_attention(const void* qkv, int T, const int* cu_seqlens, int n_seq, int n_heads, int head_dim,
                     const int2* sched, int n_sched_max, void* out, cudaStream_t st) {
  using namespace fa;
  (void)n_seq;
  if (T <= 0) return 0;
  auto fn = encode_fn();
  if (!fn) return 1;
  const int d = n_heads * head_dim;
  CUtensorMap map;
  cuuint64_t dims[2] = {(cuuint64_t)(3 * d), (cuuint64_t)T};
  cuuint64_t strides[1] = {(cuuint64_t)(3 * d) * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)BQ};
  cuuint32_t estr[2] = {1, 1};
  if (fn(&map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(qkv), dims, strides, box, estr,
         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return 1;
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)head_dim);
  const int items = n_sched_max * n_heads;
  const int grid = items < sm_count() ? items : sm_count();
  if (head_dim == 128) {
    static bool attr = false;
    if (!attr) {
      cudaFuncSetAttribute(attn_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<128>::SMEM);
      attr = true;
    }
    attn_tc_kernel<128><<<grid, THREADS, Cfg<128>::SMEM, st>>>(map, cu_seqlens, sched, n_sched_max, n_heads,
                                                               scale_log2, static_cast<uint16_t*>(out));
  } else if (head_dim == 64) {
    static bool attr = false;
    if (!attr) {
      cudaFuncSetAttribute(attn_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<64>::SMEM);
      attr = true;
    }
    attn_tc_kernel<64><<<grid, THREADS, Cfg<64>::SMEM, st>>>(map, cu_seqlens, sched, n_sched_max, n_heads,
                                                             scale_log2, static_cast<uint16_t*>(out));
  } else {
    return 1;
  }
  return 0;
}

}  // namespace rift
