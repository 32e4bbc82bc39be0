// Device helpers shared by the LoopGuard kernels: dtype access, sticky device status,
// bounded mbarrier waits, 1-D bulk (TMA) copies between global and shared memory and 16-byte
// asynchronous copies into shared memory.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "lg.h"

namespace lg {

// A bounded wait gives up after this many nanoseconds of %globaltimer.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

// Programmatic dependent launch (sm_90 and later).  Every kernel of the library is launched
// with programmatic stream serialization (launch_pdl below), so it may be scheduled while the
// kernel before it in the stream is still running.  Each kernel therefore starts with
// pdl_enter(): griddepcontrol.wait returns once the kernels it depends on have completed and
// their memory is visible (at once when there is no such kernel), so nothing of the kernel
// touches global memory before its predecessor is done; launch_dependents then lets the
// next kernel be scheduled early in turn, and it waits the same way.  Completion is
// transitive: the predecessor itself passed its wait only after its own predecessor was done.
__device__ __forceinline__ void pdl_enter() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Returns the error of a launch or call from the enclosing cudaError_t function.
#define LG_TRY(x)                                   \
  do {                                              \
    const cudaError_t lg_try_e_ = (x);              \
    if (lg_try_e_ != cudaSuccess) return lg_try_e_; \
  } while (0)

// Launch with programmatic stream serialization (see pdl_enter).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

__device__ __forceinline__ void set_status(int32_t *status, int code) {
  if (status) atomicCAS(status, 0, code);
}

__device__ __forceinline__ bool status_bad(const int32_t *status) {
  return status && *(volatile const int32_t *)status != 0;
}

// The device status as one decision for the whole CTA: thread 0 reads it and a barrier hands it
// to every thread, so that a status another CTA sets meanwhile cannot split the CTA between an
// early return and a later barrier.  Every thread of the CTA calls it.
__device__ __forceinline__ bool cta_status_bad(const int32_t *status) {
  __shared__ int s_status_bad;
  if (threadIdx.x == 0) s_status_bad = status_bad(status);
  __syncthreads();
  return s_status_bad != 0;
}

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

// ------------------------------------------------------------------ mbarrier

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits for the phase with the given parity to complete; false after kWaitLimitNs.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  while (true) {
    for (int i = 0; i < 64; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (global_ns() - t0 > kWaitLimitNs) return false;
  }
}

// ------------------------------------------------------------------ bulk copies

// 1-D bulk copy global -> shared, completion counted in bytes on `bar`.  Both addresses
// 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_load(void *smem_dst, const void *gmem_src, uint32_t bytes,
                                          uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(smem_addr(smem_dst)), "l"(gmem_src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

// 16-byte asynchronous copy global -> shared (L2 only, no registers), tracked per thread in
// commit groups; both addresses 16-byte aligned.
__device__ __forceinline__ void cp_async16(void *smem_dst, const void *gmem_src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(smem_dst)),
               "l"(gmem_src)
               : "memory");
}

__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}

// returns once at most N of this thread's most recent commit groups are still pending
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// makes this thread's completed shared-memory writes visible to the async proxy (a bulk store)
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// 1-D bulk copy shared -> global; both addresses 16-byte aligned, bytes a multiple of 16
__device__ __forceinline__ void bulk_store(void *gmem_dst, const void *smem_src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(gmem_dst),
               "r"(smem_addr(smem_src)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

// this thread's bulk stores have finished reading their shared-memory sources
__device__ __forceinline__ void bulk_wait_read_all() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}

// this thread's bulk stores are complete (written to global memory)
__device__ __forceinline__ void bulk_wait_all() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// ------------------------------------------------------------------ element access

// bf16 pair packed in a 32-bit word -> two floats (exact widening)
__device__ __forceinline__ float2 bf16x2_to_float2(uint32_t w) {
  return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}

template <typename T>
struct Elem;

template <>
struct Elem<__nv_bfloat16> {
  static constexpr int kSize = 2;
  static constexpr int kDtype = LG_BF16;
  __device__ __forceinline__ static float load(const void *p, int64_t i) {
    return __bfloat162float(((const __nv_bfloat16 *)p)[i]);
  }
  __device__ __forceinline__ static void store(void *p, int64_t i, float v) {
    ((__nv_bfloat16 *)p)[i] = __float2bfloat16_rn(v);
  }
  __device__ __forceinline__ static uint32_t sign(const void *p, int64_t i) {
    return ((const uint16_t *)p)[i] >> 15;
  }
  // 16 bytes -> 8 floats as 4 float2 pairs (element 2j in .x, 2j+1 in .y)
  __device__ __forceinline__ static void unpack(const uint4 &u, float2 *f) {
    f[0] = bf16x2_to_float2(u.x);
    f[1] = bf16x2_to_float2(u.y);
    f[2] = bf16x2_to_float2(u.z);
    f[3] = bf16x2_to_float2(u.w);
  }
};

template <>
struct Elem<float> {
  static constexpr int kSize = 4;
  static constexpr int kDtype = LG_F32;
  __device__ __forceinline__ static float load(const void *p, int64_t i) {
    return ((const float *)p)[i];
  }
  __device__ __forceinline__ static void store(void *p, int64_t i, float v) {
    ((float *)p)[i] = v;
  }
  __device__ __forceinline__ static uint32_t sign(const void *p, int64_t i) {
    return ((const uint32_t *)p)[i] >> 31;
  }
  // 16 bytes -> 4 floats as 2 float2 pairs
  __device__ __forceinline__ static void unpack(const uint4 &u, float2 *f) {
    f[0] = make_float2(__uint_as_float(u.x), __uint_as_float(u.y));
    f[1] = make_float2(__uint_as_float(u.z), __uint_as_float(u.w));
  }
};

__host__ __device__ constexpr int ilog2(int x) { return x <= 1 ? 0 : 1 + ilog2(x / 2); }
__host__ __device__ constexpr int pow2_ceil(int x) { return x <= 1 ? 1 : 2 * pow2_ceil((x + 1) / 2); }

}  // namespace lg
