// Ragged packing on sm_103a: one sequence per kept tile, [system | selected tokens | contextual
// tokens (when merged) | query], back to back, with cu_seqlens and per-row positions.
//
// Each packed row is an 8 KB (d = 4096, bf16) copy.  For bf16 tokens a CTA owns 64 rows of one
// sequence and one thread streams them through an 8-slot shared-memory ring with bulk copies
// (cp.async.bulk global -> shared, completion on an mbarrier; shared -> global, completion by
// bulk group), keeping 7 row loads in flight.  fp32 tokens (rounded to bf16 on the way) go
// through a warp-per-row copy.  The system and query rows come from the embedding table and stay
// in L2 across sequences; the vision rows stream from X once.
#include "rift_internal.h"

namespace rift {

__device__ unsigned int g_err_pack;

unsigned int read_clear_err_pack() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_err_pack, sizeof(v));
  cudaMemcpyToSymbol(g_err_pack, &z, sizeof(z));
  return v;
}

constexpr int PK_ROWS = 32;
constexpr int PK_THREADS = 256;

// The sequence offsets of the prefill, written by thread 0 of CTA (j, 0) of the packing kernels:
// cu_seqlens[j] = row_base + min(j, n) (S + Q) + sel_off[min(j, n)] + ctx_off[min(j, n)], and CTA
// (N - 1, 0) also writes cu_seqlens[N] and T = cu_seqlens[N] - row_base (row_base: rows of the
// queries packed before this one); T over max_T sets RIFT_EBIT_CAPACITY.  (The packing itself
// computes each sequence's first row the same way.)
__device__ __forceinline__ void write_offsets(int j, int n, int N, const int* __restrict__ sel_off,
                                              const int* __restrict__ ctx_off, int S, int Q, int max_T, int row_base,
                                              int* __restrict__ cu, int* __restrict__ T) {
  auto off = [&](int jj) { return jj * (S + Q) + sel_off[jj] + (ctx_off ? ctx_off[jj] : 0); };
  cu[j] = row_base + off(min(j, n));
  if (j == N - 1) {
    const int v = off(min(N, n));
    cu[N] = row_base + v;
    *T = v;
    if (v > max_T) atomicOr(&g_err_pack, RIFT_EBIT_CAPACITY);
  }
}

template <typename XT>
__global__ void __launch_bounds__(PK_THREADS) pack_kernel(
    const XT* __restrict__ X, int N, int n_v, int d, const int* __restrict__ kept,
    const int* __restrict__ n_kept, const int* __restrict__ sel, const int* __restrict__ sel_off,
    const int* __restrict__ sys_ids, int S, const int* __restrict__ query_ids, int Q,
    const uint16_t* __restrict__ embed, int vocab, const uint16_t* __restrict__ ctx,
    const int* __restrict__ ctx_off, uint16_t* __restrict__ packed, int max_T, int* __restrict__ positions,
    int row_base, int* __restrict__ cu, int* __restrict__ T) {
  pdl_trigger();
  pdl_wait();
  const int j = blockIdx.x;
  const int nk = *n_kept;
  if (blockIdx.y == 0 && threadIdx.x == 0) write_offsets(j, nk, N, sel_off, ctx_off, S, Q, max_T, row_base, cu, T);
  if (j >= nk) return;
  const int so = sel_off[j];
  const int dom = sel_off[j + 1] - so;  // selected tokens, then m contextual ones
  const int co = ctx_off ? ctx_off[j] : 0, m = ctx_off ? ctx_off[j + 1] - co : 0;
  const int b = dom + m;
  const int L = S + b + Q;
  const int base = j * (S + Q) + so + co;
  const int tile = kept[j];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int r_end = min(L, (blockIdx.y + 1) * PK_ROWS);
  for (int r = blockIdx.y * PK_ROWS + wid; r < r_end; r += PK_THREADS / 32) {
    const int dst = base + r;
    if (dst >= max_T) {
      if (lane == 0) atomicOr(&g_err_pack, RIFT_EBIT_CAPACITY);
      continue;
    }
    uint4* out = reinterpret_cast<uint4*>(packed + (size_t)dst * d);
    const int nv8 = d / 8;
    if (r < S || r >= S + b) {
      const int id = (r < S) ? sys_ids[r] : query_ids[r - S - b];
      if (id < 0 || id >= vocab) {
        if (lane == 0) atomicOr(&g_err_pack, RIFT_EBIT_BADID);
        continue;
      }
      const uint4* src = reinterpret_cast<const uint4*>(embed + (size_t)id * d);
      for (int q = lane; q < nv8; q += 32) out[q] = src[q];
    } else if (r >= S + dom) {
      const uint4* src = reinterpret_cast<const uint4*>(ctx + (size_t)(co + r - S - dom) * d);
      for (int q = lane; q < nv8; q += 32) out[q] = src[q];
    } else {
      const int k = sel[so + r - S];
      if (k < 0 || k >= n_v || tile < 0 || tile >= N) {
        if (lane == 0) atomicOr(&g_err_pack, RIFT_EBIT_BADID);
        continue;
      }
      const XT* row = X + ((size_t)tile * n_v + k) * d;
      if constexpr (sizeof(XT) == 2) {
        const uint4* src = reinterpret_cast<const uint4*>(row);
        for (int q = lane; q < nv8; q += 32) out[q] = __ldcs(src + q);
      } else {
        const float4* src = reinterpret_cast<const float4*>(row);
        for (int q = lane; q < nv8; q += 32) {
          float4 a = __ldcs(src + 2 * q), c = __ldcs(src + 2 * q + 1);
          out[q] = make_uint4(pack_bf16x2(a.x, a.y), pack_bf16x2(a.z, a.w), pack_bf16x2(c.x, c.y),
                              pack_bf16x2(c.z, c.w));
        }
      }
    }
    if (lane == 0) positions[dst] = r;
  }
}

constexpr int PKB_ROWS = 64;   // rows per CTA
constexpr int PKB_SLOTS = 8;   // row buffers

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Bounded wait on an mbarrier phase; false if it ran out (~1 s).
__device__ __forceinline__ bool pk_wait(uint32_t bar, uint32_t parity) {
  uint64_t t0;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t0));
  for (uint32_t i = 0; i < RIFT_SPIN_LIMIT; ++i) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.b32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    if (ok) return true;
    if ((i & 255u) == 255u) {
      uint64_t t;
      asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
      if (t - t0 > 1000000000ull) break;
    }
  }
  return false;
}

__global__ void __launch_bounds__(64) pack_bulk_kernel(
    const uint16_t* __restrict__ X, int N, int n_v, int d, const int* __restrict__ kept,
    const int* __restrict__ n_kept, const int* __restrict__ sel, const int* __restrict__ sel_off,
    const int* __restrict__ sys_ids, int S, const int* __restrict__ query_ids, int Q,
    const uint16_t* __restrict__ embed, int vocab, const uint16_t* __restrict__ ctx,
    const int* __restrict__ ctx_off, uint16_t* __restrict__ packed, int max_T, int* __restrict__ positions,
    int row_base, int* __restrict__ cu, int* __restrict__ T) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ __align__(128) uint8_t ring[];
  __shared__ __align__(8) uint64_t bars[PKB_SLOTS];
  const int j = blockIdx.x;
  const int nk = *n_kept;
  if (blockIdx.y == 0 && threadIdx.x == 0) write_offsets(j, nk, N, sel_off, ctx_off, S, Q, max_T, row_base, cu, T);
  if (j >= nk) return;
  const int so = sel_off[j];
  const int dom = sel_off[j + 1] - so;  // selected tokens, then m contextual ones
  const int co = ctx_off ? ctx_off[j] : 0, m = ctx_off ? ctx_off[j + 1] - co : 0;
  const int b = dom + m;
  const int L = S + b + Q;
  const int base = j * (S + Q) + so + co;
  const int tile = kept[j];
  const int r0 = blockIdx.y * PKB_ROWS;
  const int n = min(L - r0, PKB_ROWS);
  if (n <= 0) return;
  for (int q = threadIdx.x; q < n; q += blockDim.x)
    if (base + r0 + q < max_T) positions[base + r0 + q] = r0 + q;
  if (threadIdx.x != 0) return;

  const uint32_t row_bytes = (uint32_t)d * 2u;
  // source row of packed row r (nullptr: bad id or past capacity, reported and skipped)
  auto src_of = [&](int r) -> const uint16_t* {
    if (base + r >= max_T) { atomicOr(&g_err_pack, RIFT_EBIT_CAPACITY); return nullptr; }
    if (r < S || r >= S + b) {
      const int id = (r < S) ? sys_ids[r] : query_ids[r - S - b];
      if (id < 0 || id >= vocab) { atomicOr(&g_err_pack, RIFT_EBIT_BADID); return nullptr; }
      return embed + (size_t)id * d;
    }
    if (r >= S + dom) return ctx + (size_t)(co + r - S - dom) * d;
    const int k = sel[so + r - S];
    if (k < 0 || k >= n_v || tile < 0 || tile >= N) { atomicOr(&g_err_pack, RIFT_EBIT_BADID); return nullptr; }
    return X + ((size_t)tile * n_v + k) * d;
  };
  for (int q = 0; q < PKB_SLOTS; ++q)
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;\n" ::"r"(smem_u32(&bars[q])) : "memory");
  asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
  asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");

  uint32_t uses[PKB_SLOTS];   // issued loads per slot (sets the parity to wait for)
  bool issued[PKB_ROWS];
  for (int q = 0; q < PKB_SLOTS; ++q) uses[q] = 0;
  auto issue = [&](int i) {
    const uint16_t* src = src_of(r0 + i);
    issued[i] = src != nullptr;
    if (!src) return;
    const int slot = i % PKB_SLOTS;
    const uint32_t bar = smem_u32(&bars[slot]);
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(bar), "r"(row_bytes) : "memory");
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(
                     smem_u32(ring + (size_t)slot * row_bytes)),
                 "l"(src), "r"(row_bytes), "r"(bar)
                 : "memory");
    ++uses[slot];
  };
  for (int i = 0; i < PKB_SLOTS - 1 && i < n; ++i) issue(i);
  bool ok = true;
  for (int i = 0; i < n; ++i) {
    const int slot = i % PKB_SLOTS;
    if (issued[i] && ok) {
      if (!pk_wait(smem_u32(&bars[slot]), (uses[slot] - 1) & 1u)) {
        atomicOr(&g_err_pack, RIFT_EBIT_TIMEOUT);
        ok = false;
      } else {
        asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;\n" ::"l"(
                         packed + (size_t)(base + r0 + i) * d),
                     "r"(smem_u32(ring + (size_t)slot * row_bytes)), "r"(row_bytes)
                     : "memory");
      }
    }
    asm volatile("cp.async.bulk.commit_group;\n" ::: "memory");
    const int next = i + PKB_SLOTS - 1;  // reuses the slot of row i - 1
    if (next < n && ok) {
      asm volatile("cp.async.bulk.wait_group.read 1;\n" ::: "memory");
      issue(next);
    }
  }
  asm volatile("cp.async.bulk.wait_group 0;\n" ::: "memory");
  if (!ok) {  // a load never completed: wait (bounded) for the others issued before leaving
    for (int q = 0; q < PKB_SLOTS; ++q)
      if (uses[q]) pk_wait(smem_u32(&bars[q]), (uses[q] - 1) & 1u);
  }
}

void launch_pack(const void* X, rift_dtype xdt, int N, int n_v, int d, const int* kept,
                 const int* n_kept, const int* sel, const int* sel_off, const int* sys_ids, int S,
                 const int* query_ids, int Q, const void* embed, int vocab, const void* ctx, const int* ctx_off,
                 void* packed, int max_T, int* cu_seqlens, int* positions, int* T, int row_base,
                 cudaStream_t st) {
  const uint16_t* cx = static_cast<const uint16_t*>(ctx);
  const int max_L = S + n_v + Q;
  dim3 grid(N, (max_L + PK_ROWS - 1) / PK_ROWS);
  if (xdt == RIFT_BF16) {
    const size_t smem = (size_t)PKB_SLOTS * d * 2;
    static std::atomic<unsigned long long> smem_raised{0};
    if (raise_smem_limit(smem_raised, pack_bulk_kernel, PKB_SLOTS * 8192 * 2) != cudaSuccess)
      return;  // the error stays pending for the caller's launch check
    dim3 gb(N, (max_L + PKB_ROWS - 1) / PKB_ROWS);
    launch_ex(pack_bulk_kernel, gb, dim3(64), smem, st, true, static_cast<const uint16_t*>(X), N, n_v, d, kept,
              n_kept, sel, sel_off, sys_ids, S, query_ids, Q, static_cast<const uint16_t*>(embed), vocab, cx, ctx_off,
              static_cast<uint16_t*>(packed), max_T, positions, row_base, cu_seqlens, T);
  } else
    launch_ex(pack_kernel<float>, grid, dim3(PK_THREADS), 0, st, true, static_cast<const float*>(X), N, n_v, d, kept,
              n_kept, sel, sel_off, sys_ids, S, query_ids, Q, static_cast<const uint16_t*>(embed), vocab, cx, ctx_off,
              static_cast<uint16_t*>(packed), max_T, positions, row_base, cu_seqlens, T);
}

}  // namespace rift
