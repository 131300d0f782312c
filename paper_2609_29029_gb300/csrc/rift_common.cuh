// Shared device helpers of the Rift CUDA library (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "rift.h"

// Device error bits, OR-ed into a per-translation-unit flag and collected by rift_sync_status.
#define RIFT_EBIT_NONFINITE 1u
#define RIFT_EBIT_CAPACITY 2u
#define RIFT_EBIT_TIMEOUT 4u
#define RIFT_EBIT_BADID 8u

// Upper bound on the spin iterations of any device-side wait (mbarrier, flag).  Waits that
// reach it set RIFT_EBIT_TIMEOUT and give up instead of hanging the GPU.
#define RIFT_SPIN_LIMIT (1u << 26)

#define RIFT_CUDA_TRY(expr)                          \
  do {                                               \
    cudaError_t _e = (expr);                         \
    if (_e != cudaSuccess) return RIFT_ERR_CUDA;     \
  } while (0)

#define RIFT_LAUNCH_CHECK() RIFT_CUDA_TRY(cudaGetLastError())

namespace rift {

// The unique id of the calling thread's current CUDA context (cuCtxGetId: ids are never reused
// within a process, unlike context handles), or 0 if it cannot be read.  (rift_abi.cu)
unsigned long long current_context_id();

// Raises `kernel`'s dynamic shared-memory limit to `bytes` in the current CUDA context.  A
// function's attributes belong to a context (every device's primary context, and any context a
// host creates with the driver API has its own), so `done`, the call site's record, holds the id
// of the context last raised; a call from another context (or with an unreadable id) raises again.
template <typename K>
inline cudaError_t raise_smem_limit(std::atomic<unsigned long long>& done, K* kernel, int bytes) {
  const unsigned long long ctx = current_context_id();
  if (ctx != 0 && done.load(std::memory_order_acquire) == ctx) return cudaSuccess;
  const cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess && ctx != 0) done.store(ctx, std::memory_order_release);
  return e;
}

// Programmatic dependent launch.  A kernel launched with `pdl` set (launch_ex) may begin while
// the kernel before it in the stream is still running: each of its threads calls pdl_wait()
// before its first access to memory that earlier kernels write or read (constant weights
// excepted), and pdl_trigger() lets the kernel after it begin launching.  Both are no-ops in a
// kernel launched without the attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory"); }

template <typename... KArgs, typename... Args>
static inline cudaError_t launch_ex(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                                    bool pdl, Args... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

static inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float warp_min(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Inclusive prefix sum over the 32 lanes of a warp.
__device__ __forceinline__ int warp_incl_scan(int v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int n = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += n;
  }
  return v;
}

// Block-wide sum; every thread gets the result.  `red` holds >= 32 floats.
__device__ __forceinline__ float block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) red[wid] = v;
  __syncthreads();
  float r = 0.f;
  for (int w = 0; w < nw; ++w) r += red[w];  // fixed order: same result in every thread
  return r;
}

// Block-wide exclusive prefix sum of one int per thread (in thread order); *total gets the
// sum.  `sh` holds >= 33 ints.
__device__ __forceinline__ int block_excl_scan(int v, int* sh, int* total) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  int inc = warp_incl_scan(v);
  __syncthreads();
  if (lane == 31) sh[wid] = inc;
  __syncthreads();
  if (wid == 0) {
    int x = (lane < nw) ? sh[lane] : 0;
    int xi = warp_incl_scan(x);
    if (lane < nw) sh[lane] = xi - x;
    if (lane == nw - 1) sh[32] = xi;
  }
  __syncthreads();
  int res = sh[wid] + inc - v;
  *total = sh[32];
  return res;
}

__device__ __forceinline__ float bf16_bits_to_float(uint16_t b) {
  return __uint_as_float(static_cast<uint32_t>(b) << 16);
}

// Unpack 8 bf16 values held in a uint4.
__device__ __forceinline__ void unpack_bf16x8(const uint4& v, float* f) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}

__device__ __forceinline__ uint32_t pack_half2(float lo, float hi) {
  __half2 h = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

}  // namespace rift
