// Device-side helpers shared by the HeadKV kernels: element unpacking,
// the error word, bounded mbarrier waits, 1D TMA bulk copies and block scans.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "hkv.h"

namespace hkv {

// the limit of any device wait (a test build may shorten it)
#ifndef HKV_WAIT_TIMEOUT_NS
#define HKV_WAIT_TIMEOUT_NS 2000000000ull
#endif
constexpr uint64_t kWaitTimeoutNs = HKV_WAIT_TIMEOUT_NS;  // 2 s by default

// ---------------------------------------------------------------------------
// elements: a 16-byte piece holds 4 fp32 or 8 bf16 values
// ---------------------------------------------------------------------------
template <typename T>
struct Elem;

template <>
struct Elem<float> {
  static constexpr int kPerPiece = 4;
  __device__ static __forceinline__ void unpack(const uint4 &u, float *f) {
    f[0] = __uint_as_float(u.x);
    f[1] = __uint_as_float(u.y);
    f[2] = __uint_as_float(u.z);
    f[3] = __uint_as_float(u.w);
  }
  __device__ static __forceinline__ float load1(const void *base, size_t i) {
    return reinterpret_cast<const float *>(base)[i];
  }
};

template <>
struct Elem<__nv_bfloat16> {
  static constexpr int kPerPiece = 8;
  // a bf16 value is the top half of the fp32 with the same bits: exact
  __device__ static __forceinline__ void unpack(const uint4 &u, float *f) {
    f[0] = __uint_as_float(u.x << 16);
    f[1] = __uint_as_float(u.x & 0xFFFF0000u);
    f[2] = __uint_as_float(u.y << 16);
    f[3] = __uint_as_float(u.y & 0xFFFF0000u);
    f[4] = __uint_as_float(u.z << 16);
    f[5] = __uint_as_float(u.z & 0xFFFF0000u);
    f[6] = __uint_as_float(u.w << 16);
    f[7] = __uint_as_float(u.w & 0xFFFF0000u);
  }
  __device__ static __forceinline__ float load1(const void *base, size_t i) {
    const uint16_t b = reinterpret_cast<const uint16_t *>(base)[i];
    return __uint_as_float(((uint32_t)b) << 16);
  }
};

// ---------------------------------------------------------------------------
// error word: the first failure wins
// ---------------------------------------------------------------------------
__device__ __forceinline__ void set_err(uint32_t *err, uint32_t code) {
  if (err) atomicCAS(err, 0u, code);
}

// ---------------------------------------------------------------------------
// mbarrier + 1D bulk copy (TMA engine), single-CTA use
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

// adds to the bytes the current phase waits for, without arriving
__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Non-blocking: whether the phase with the given parity has completed
// (try_wait above may suspend the thread for a while before it answers).
__device__ __forceinline__ bool mbar_test_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// 2^x with the hardware base-2 exponential (PTX ex2.approx.ftz.f32): a few
// ulp; a subnormal result flushes to zero, which in a softmax only drops
// weights below 2^-126 of the row's maximum
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Waits for the phase with the given parity; false if it did not complete
// within kWaitTimeoutNs.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 63u) == 0 && globaltimer() - t0 > kWaitTimeoutNs) return false;
  }
}

// global -> shared bulk copy of `bytes` (multiple of 16, both ends 16-byte
// aligned), completion counted on `bar`
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes,
                                         uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// An L2 policy that evicts the lines it is applied to first, and the bulk
// copy above under such a policy: for data streamed once (the K/V arena in
// decode attention), so that it does not push small, soon re-read data (the
// kernels' records, partial results and counters) out of L2.
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ void bulk_g2s_hint(void *dst, const void *src, uint32_t bytes,
                                              uint64_t *bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

// 16-byte asynchronous global -> shared copy (both ends 16-byte aligned) and
// the wait for all of the thread's outstanding ones
__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
}

// ---------------------------------------------------------------------------
// block-wide scans (all threads must call; `scratch` holds >= 33 entries)
// ---------------------------------------------------------------------------
template <typename V>
__device__ __forceinline__ V warp_incl_scan(V x) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    V y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  return x;
}

// exclusive scan over the block; returns this thread's exclusive prefix and
// writes the block total to *total
template <typename V>
__device__ __forceinline__ V block_excl_scan(V x, V *scratch, V *total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nwarps = (blockDim.x + 31) >> 5;
  V incl = warp_incl_scan(x);
  if (lane == 31) scratch[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    V wv = lane < nwarps ? scratch[lane] : V(0);
    V wi = warp_incl_scan(wv);
    if (lane < nwarps) scratch[lane] = wi - wv;
    if (lane == nwarps - 1) scratch[32] = wi;
  }
  __syncthreads();
  V res = scratch[warp] + incl - x;
  *total = scratch[32];
  __syncthreads();
  return res;
}

}  // namespace hkv
