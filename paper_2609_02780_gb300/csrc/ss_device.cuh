// Inline-PTX building blocks shared by the library's kernels: the bf16 m16n8k16 tensor
// core MMA, streaming loads, mbarriers and bulk (TMA) copies into shared memory.
#pragma once

#include "ss_internal.cuh"

namespace ss {

// D += A (16x16 bf16, row) * B (16x8 bf16, col), fp32 accumulate. Lane (g, t) holds
// A rows g and g + 8 and B column g; the k index of each register pair is free to be
// permuted as long as A and B use the same permutation.
__device__ __forceinline__ void mma_16816(float (&d)[4], uint32_t a0, uint32_t a1,
                                          uint32_t a2, uint32_t a3, uint32_t b0,
                                          uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 r;
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}

// ---- TMA bulk copies and mbarriers (inline PTX) ----
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Non-blocking test of a phase (never suspends the thread, unlike try_wait).
__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Global -> shared bulk copy of `bytes` (multiple of 16, 16-byte aligned ends) that
// completes the transaction count of `bar`.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes,
                                          uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(dst), "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Bounded wait for a phase of an mbarrier: gives up after `polls` polls or ~1 s,
// whichever comes first (0 polls: gives up at once, without looking).
static __device__ bool mbar_wait_limit(uint32_t bar, uint32_t parity, uint32_t polls) {
  if (polls == 0u) return false;
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t i = 1; i < polls; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 1023u) == 0u && global_ns() - t0 > 1000000000ull) break;
  }
  return false;
}
// The default limit: 2^26 polls or ~1 s.
static __device__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity) {
  return mbar_wait_limit(bar, parity, kDefaultWaitPolls);
}

// ---- fixed-order block reductions (deterministic) ----
// Block reduction of (max, sum 2^(s - max)) pairs in a fixed order; result to all.
static __device__ void block_ml(float& m, float& l, float* sm, float* sl) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = blockDim.x >> 5;
  for (int off = 16; off > 0; off >>= 1) {
    const float mo = __shfl_down_sync(0xffffffffu, m, off);
    const float lo = __shfl_down_sync(0xffffffffu, l, off);
    ml_combine(m, l, mo, lo);
  }
  if (lane == 0) {
    sm[warp] = m;
    sl[warp] = l;
  }
  __syncthreads();
  if (warp == 0) {
    m = lane < nw ? sm[lane] : -INFINITY;
    l = lane < nw ? sl[lane] : 0.f;
    for (int off = 16; off > 0; off >>= 1) {
      const float mo = __shfl_down_sync(0xffffffffu, m, off);
      const float lo = __shfl_down_sync(0xffffffffu, l, off);
      ml_combine(m, l, mo, lo);
    }
    if (lane == 0) {
      sm[0] = m;
      sl[0] = l;
    }
  }
  __syncthreads();
  m = sm[0];
  l = sl[0];
  __syncthreads();
}

// Fixed-order block sum; result to all threads.
static __device__ float block_sum(float v, float* sm) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = blockDim.x >> 5;
  for (int off = 16; off > 0; off >>= 1) v += __shfl_down_sync(0xffffffffu, v, off);
  if (lane == 0) sm[warp] = v;
  __syncthreads();
  if (warp == 0) {
    v = lane < nw ? sm[lane] : 0.f;
    for (int off = 16; off > 0; off >>= 1) v += __shfl_down_sync(0xffffffffu, v, off);
    if (lane == 0) sm[0] = v;
  }
  __syncthreads();
  v = sm[0];
  __syncthreads();
  return v;
}

static __device__ float block_min(float v, float* sm) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = blockDim.x >> 5;
  for (int off = 16; off > 0; off >>= 1) v = fminf(v, __shfl_down_sync(0xffffffffu, v, off));
  if (lane == 0) sm[warp] = v;
  __syncthreads();
  if (warp == 0) {
    v = lane < nw ? sm[lane] : INFINITY;
    for (int off = 16; off > 0; off >>= 1) v = fminf(v, __shfl_down_sync(0xffffffffu, v, off));
    if (lane == 0) sm[0] = v;
  }
  __syncthreads();
  v = sm[0];
  __syncthreads();
  return v;
}


// Exclusive prefix sum over the block (thread order); all threads get their prefix.
static __device__ int block_excl_scan(int v, int* sw) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = blockDim.x >> 5;
  int x = v;
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) sw[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nw ? sw[lane] : 0;
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, off);
      if (lane >= off) w += y;
    }
    sw[lane] = w;
  }
  __syncthreads();
  const int prefix = warp > 0 ? sw[warp - 1] : 0;
  return prefix + x - v;
}

}  // namespace ss
