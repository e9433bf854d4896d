// Index construction kernels (Sec. 4.1): appending shallow keys to the full-history
// cache (Eq. 2) and the unit descriptor (Eq. 3).
#include "ss_internal.cuh"

namespace ss {

// Copies n_tokens rows of every slab from src [slab][src_stride][d] into the index
// slabs [slab][ncap][d] starting at token tok0 (16-byte vector copies).
__global__ void k_append(__nv_bfloat16* __restrict__ keys, int64_t ncap, int64_t tok0,
                         const __nv_bfloat16* __restrict__ src, int64_t src_stride,
                         int n_slabs, int64_t n_tokens) {
  constexpr int kVec = kHeadDim * 2 / 16;  // 16-byte vectors per key row
  const int64_t total = (int64_t)n_slabs * n_tokens * kVec;
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < total;
       x += (int64_t)gridDim.x * blockDim.x) {
    const int64_t row = x / kVec;
    const int v = (int)(x - row * kVec);
    const int64_t slab = row / n_tokens;
    const int64_t t = row - slab * n_tokens;
    const uint4* s = reinterpret_cast<const uint4*>(src + (slab * src_stride + t) * kHeadDim) + v;
    uint4* d = reinterpret_cast<uint4*>(keys + (slab * ncap + tok0 + t) * kHeadDim) + v;
    *d = *s;
  }
}

cudaError_t launch_append(__nv_bfloat16* keys, int64_t ncap, int64_t tok0,
                          const __nv_bfloat16* src, int64_t src_stride_tokens,
                          int n_slabs, int64_t n_tokens, cudaStream_t s) {
  if (n_tokens <= 0) return cudaSuccess;
  const int64_t total = (int64_t)n_slabs * n_tokens * (kHeadDim * 2 / 16);
  const int threads = 256;
  const int64_t want = (total + threads - 1) / threads;
  const int blocks = (int)(want < 65536 ? want : 65536);
  k_append<<<blocks, threads, 0, s>>>(keys, ncap, tok0, src, src_stride_tokens, n_slabs, n_tokens);
  return cudaGetLastError();
}

// Eq. 3: k_u = Norm(mean over the unit's tokens of vec over key heads of K^{P-1}).
// One CTA per unit, one thread per vec element (key head g, channel j); the mean is an
// fp32 sum in token order divided by T_u; Norm(0) = 0.
__global__ void k_descriptors(const __nv_bfloat16* __restrict__ keys, int64_t ncap, int P,
                              int Hkv, int Tu, int64_t u_begin, float* __restrict__ desc) {
  __shared__ float red[32];
  const int64_t u = u_begin + blockIdx.x;
  const int tid = threadIdx.x;
  const int g = tid / kHeadDim, j = tid - g * kHeadDim;
  const __nv_bfloat16* base =
      keys + ((int64_t)((P - 1) * Hkv + g) * ncap + u * Tu) * kHeadDim + j;
  float acc = 0.f;
  for (int t = 0; t < Tu; ++t) acc += __bfloat162float(base[(int64_t)t * kHeadDim]);
  const float mean = acc / (float)Tu;
  float sq = mean * mean;
  for (int off = 16; off > 0; off >>= 1) sq += __shfl_down_sync(0xffffffffu, sq, off);
  const int lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
  if (lane == 0) red[warp] = sq;
  __syncthreads();
  if (warp == 0) {
    sq = lane < nw ? red[lane] : 0.f;
    for (int off = 16; off > 0; off >>= 1) sq += __shfl_down_sync(0xffffffffu, sq, off);
    if (lane == 0) red[0] = sq;
  }
  __syncthreads();
  const float nrm = sqrtf(red[0]);
  desc[u * (int64_t)(Hkv * kHeadDim) + tid] = nrm > 0.f ? mean / nrm : 0.f;
}

cudaError_t launch_descriptors(const __nv_bfloat16* keys, int64_t ncap, int P, int Hkv,
                               int Tu, int64_t u_begin, int64_t u_end, float* desc,
                               cudaStream_t s) {
  if (u_end <= u_begin) return cudaSuccess;
  const int64_t n = u_end - u_begin;
  for (int64_t off = 0; off < n; off += 65535) {
    const int blocks = (int)((n - off) < 65535 ? (n - off) : 65535);
    k_descriptors<<<blocks, Hkv * kHeadDim, 0, s>>>(keys, ncap, P, Hkv, Tu, u_begin + off, desc);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace ss
