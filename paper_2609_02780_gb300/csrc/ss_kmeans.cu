// k-means compression of the shallow index (the cluster-compressed index variant).
//
// The paper bounds memory by replacing older history with cluster representatives
// (Sec. 4.1, Eq. 5-7: units merged online into temporally adjacent clusters whose
// representative KVs are running means). The token-level reading implemented here:
// for every window of W consecutive frames and every (layer i, key head g), the
// window's keys X are clustered by Lloyd's algorithm,
//   C^0 = X[0 : n_c]  (the window's first n_c tokens, in token order)
//   repeat `iters` times:
//     assign  a(x) = argmin_c ||x - c||^2   (lowest centroid id among equal distances)
//     update  c = mean of the keys assigned to c; a centroid with no keys keeps its value
// and the index stores the last update's centroids (bf16, nearest-even), the last
// assignment, and per (centroid, unit of the window) member counts for retrieval.
#include "ss_internal.cuh"
#include "ss_device.cuh"

namespace ss {

constexpr int kKmWarps = 8;
constexpr int kKmThreads = kKmWarps * 32;
constexpr int kKmChunk = 64;  // keys staged in shared memory per step of the update

struct KmJob {
  const __nv_bfloat16* keys;  // [n_slabs][ncap][d]
  int64_t ncap;
  __nv_bfloat16* cent;        // [n_slabs][wcap * n_c][d]
  uint8_t* assign;            // [n_slabs][ncap]
  int32_t* mcnt;              // [n_slabs][wcap][n_c][wu] members per (centroid, unit)
  int32_t* msize;             // [n_slabs][wcap][n_c] members per centroid
  int64_t tok_first;          // first token of this call's first window
  int Wt;                     // tokens per window
  int Tu;                     // tokens per unit
  int wu;                     // units per window
  int w_begin;                // index of this call's first window
  int wcap;
  int n_c, n_c8;              // centroids; rounded up to a multiple of 8
  int iters;
};

size_t kmeans_smem_bytes(int n_c, int Wt) {
  const int n_c8 = (n_c + 7) & ~7;
  return (size_t)n_c8 * 512 * 2 + (size_t)kKmChunk * kHeadDim * 2 + (size_t)n_c8 * 8 +
         (size_t)((Wt + 15) & ~15);
}

// Tensor-core operands of the centroids for the distance step: each fp32 centroid is
// split into c_hi = bf16(c) and c_lo = bf16(c - c_hi), and x . c is accumulated as
// x . c_hi + x . c_lo (the keys x are exact bf16 values), which carries ~16 significant
// bits of c. Layout: [group of 8 centroids][hi, lo][v = 0..3][lane]; lane (g, t) holds
// dims 8 (4 v + t) .. + 7 of centroid 8 * group + g, the B-fragment order of the MMA
// below (the same k permutation as the keys' A fragments). ||c||^2 comes from fp32 c.
__device__ void km_build_operands(const float* Cf, uint4* Bf, float* cn2, int n_c, int n_c8) {
  const int n_ent = n_c8 * 32;  // (n_c8 / 8) groups x 2 x 4 x 32
  for (int e = threadIdx.x; e < n_ent; e += blockDim.x) {
    const int lane = e & 31, v = (e >> 5) & 3, hl = (e >> 7) & 1, grp = e >> 8;
    const int c = grp * 8 + (lane >> 2);
    const int d0 = 8 * (4 * v + (lane & 3));
    uint32_t w[4];
#pragma unroll
    for (int h = 0; h < 4; ++h) {
      float x0 = 0.f, x1 = 0.f;
      if (c < n_c) {
        x0 = Cf[c * kHeadDim + d0 + 2 * h];
        x1 = Cf[c * kHeadDim + d0 + 2 * h + 1];
      }
      __nv_bfloat16 b0 = __float2bfloat16_rn(x0), b1 = __float2bfloat16_rn(x1);
      if (hl) {
        b0 = __float2bfloat16_rn(x0 - __bfloat162float(b0));
        b1 = __float2bfloat16_rn(x1 - __bfloat162float(b1));
      }
      w[h] = (uint32_t)__bfloat16_as_ushort(b0) | ((uint32_t)__bfloat16_as_ushort(b1) << 16);
    }
    Bf[e] = make_uint4(w[0], w[1], w[2], w[3]);
  }
  for (int c = threadIdx.x; c < n_c8; c += blockDim.x) {
    float s = 0.f;
    if (c < n_c) {
      for (int d = 0; d < kHeadDim; ++d) s = fmaf(Cf[c * kHeadDim + d], Cf[c * kHeadDim + d], s);
    } else {
      s = INFINITY;  // padding centroids are never nearest
    }
    cn2[c] = s;
  }
}

// One CTA per (window, slab).
__global__ void __launch_bounds__(kKmThreads) k_kmeans(const KmJob J) {
  extern __shared__ __align__(16) unsigned char sm[];
  const int n_c = J.n_c, n_c8 = J.n_c8, Wt = J.Wt;
  float* Cf = reinterpret_cast<float*>(sm);
  uint4* Bf = reinterpret_cast<uint4*>(sm + (size_t)n_c8 * 512);
  float* S = reinterpret_cast<float*>(Bf);  // sums of the update, over the operands
  __nv_bfloat16* chunk = reinterpret_cast<__nv_bfloat16*>(sm + (size_t)n_c8 * 1024);
  float* cn2 = reinterpret_cast<float*>(chunk + kKmChunk * kHeadDim);
  int* cnt = reinterpret_cast<int*>(cn2 + n_c8);
  uint8_t* a = reinterpret_cast<uint8_t*>(cnt + n_c8);

  const int wl = blockIdx.x, slab = blockIdx.y;
  const int wg = J.w_begin + wl;
  const int64_t tok0 = J.tok_first + (int64_t)wl * Wt;
  const __nv_bfloat16* X = J.keys + ((int64_t)slab * J.ncap + tok0) * kHeadDim;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = lane >> 2, t4 = lane & 3;

  for (int x = tid; x < n_c8 * kHeadDim; x += blockDim.x)
    Cf[x] = (x >> 7) < n_c ? __bfloat162float(X[x]) : 0.f;
  __syncthreads();
  km_build_operands(Cf, Bf, cn2, n_c, n_c8);
  __syncthreads();

  const int ntile = (Wt + 15) / 16;
  const int ngrp = n_c8 / 8;
  for (int it = 0; it < J.iters; ++it) {
    // ---- assign: nearest centroid of every key (tensor cores) ----
    // a warp walks its tiles with the next tile's key fragments already in flight
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    auto load_tile = [&](int tile, uint4 (&fa)[4], uint4 (&fb)[4]) {
      const int q0 = tile * 16 + g, q1 = q0 + 8;
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        fa[v] = tile < ntile && q0 < Wt ? ld_stream(X + (int64_t)q0 * kHeadDim + 8 * (4 * v + t4)) : z;
        fb[v] = tile < ntile && q1 < Wt ? ld_stream(X + (int64_t)q1 * kHeadDim + 8 * (4 * v + t4)) : z;
      }
    };
    uint4 ra[4], rb[4];
    load_tile(warp, ra, rb);
    for (int tile = warp; tile < ntile; tile += kKmWarps) {
      const int r0 = tile * 16 + g, r1 = r0 + 8;
      uint4 na[4], nb[4];
      load_tile(tile + kKmWarps, na, nb);
      float bd0 = INFINITY, bd1 = INFINITY;
      int bc0 = 0, bc1 = 0;
      for (int grp = 0; grp < ngrp; ++grp) {
        const uint4* bh = Bf + (size_t)grp * 256;
        const uint4* bl = bh + 128;
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          const uint4 h = bh[v * 32 + lane], l = bl[v * 32 + lane];
          mma_16816(acc, ra[v].x, rb[v].x, ra[v].y, rb[v].y, h.x, h.y);
          mma_16816(acc, ra[v].z, rb[v].z, ra[v].w, rb[v].w, h.z, h.w);
          mma_16816(acc, ra[v].x, rb[v].x, ra[v].y, rb[v].y, l.x, l.y);
          mma_16816(acc, ra[v].z, rb[v].z, ra[v].w, rb[v].w, l.z, l.w);
        }
        // ||x - c||^2 - ||x||^2 = ||c||^2 - 2 x . c; scanned in increasing centroid id
        const int c0 = grp * 8 + 2 * t4;
        const float n0 = cn2[c0], n1 = cn2[c0 + 1];
        const float d00 = fmaf(-2.f, acc[0], n0), d01 = fmaf(-2.f, acc[1], n1);
        const float d10 = fmaf(-2.f, acc[2], n0), d11 = fmaf(-2.f, acc[3], n1);
        if (d00 < bd0) { bd0 = d00; bc0 = c0; }
        if (d01 < bd0) { bd0 = d01; bc0 = c0 + 1; }
        if (d10 < bd1) { bd1 = d10; bc1 = c0; }
        if (d11 < bd1) { bd1 = d11; bc1 = c0 + 1; }
      }
      // the 4 lanes of a row hold interleaved centroids: smallest (distance, id)
#pragma unroll
      for (int off = 1; off < 4; off <<= 1) {
        const float od0 = __shfl_xor_sync(0xffffffffu, bd0, off);
        const int oc0 = __shfl_xor_sync(0xffffffffu, bc0, off);
        const float od1 = __shfl_xor_sync(0xffffffffu, bd1, off);
        const int oc1 = __shfl_xor_sync(0xffffffffu, bc1, off);
        if (od0 < bd0 || (od0 == bd0 && oc0 < bc0)) { bd0 = od0; bc0 = oc0; }
        if (od1 < bd1 || (od1 == bd1 && oc1 < bc1)) { bd1 = od1; bc1 = oc1; }
      }
      if (t4 == 0) {
        if (r0 < Wt) a[r0] = (uint8_t)bc0;
        if (r1 < Wt) a[r1] = (uint8_t)bc1;
      }
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        ra[v] = na[v];
        rb[v] = nb[v];
      }
    }
    __syncthreads();
    // ---- update: fp32 sums in token order; warp w owns centroids w, w + 8, ... ----
    for (int x = tid; x < n_c8 * kHeadDim; x += blockDim.x) S[x] = 0.f;
    for (int c = tid; c < n_c8; c += blockDim.x) cnt[c] = 0;
    __syncthreads();
    // the chunks pass through shared memory in token order; each thread's share of the
    // next chunk is loaded into registers while the current one is summed
    constexpr int kPer = kKmChunk * 16 / kKmThreads;
    uint4 nxt[kPer];
    auto load_chunk = [&](int q0) {
      const int nr = min(kKmChunk, Wt - q0);
#pragma unroll
      for (int e = 0; e < kPer; ++e) {
        const int x = e * kKmThreads + tid;
        if (q0 < Wt && x < nr * 16) nxt[e] = ld_stream(X + (int64_t)q0 * kHeadDim + 8 * x);
      }
    };
    auto store_chunk = [&](int q0) {
      const int nr = min(kKmChunk, Wt - q0);
#pragma unroll
      for (int e = 0; e < kPer; ++e) {
        const int x = e * kKmThreads + tid;
        if (q0 < Wt && x < nr * 16) reinterpret_cast<uint4*>(chunk)[x] = nxt[e];
      }
    };
    load_chunk(0);
    store_chunk(0);
    for (int p0 = 0; p0 < Wt; p0 += kKmChunk) {
      const int nrow = min(kKmChunk, Wt - p0);
      load_chunk(p0 + kKmChunk);
      __syncthreads();
      for (int c = warp; c < n_c; c += kKmWarps) {
        float4 acc = *reinterpret_cast<const float4*>(S + c * kHeadDim + 4 * lane);
        int n = 0;
        for (int h = 0; h < nrow; h += 32) {
          const bool mine = h + lane < nrow && a[p0 + h + lane] == c;
          unsigned m = __ballot_sync(0xffffffffu, mine);
          while (m) {
            const int j = __ffs(m) - 1;
            m &= m - 1;
            const uint2 kv = *reinterpret_cast<const uint2*>(chunk + (h + j) * kHeadDim + 4 * lane);
            acc.x += __bfloat162float(__ushort_as_bfloat16((unsigned short)(kv.x & 0xffffu)));
            acc.y += __bfloat162float(__ushort_as_bfloat16((unsigned short)(kv.x >> 16)));
            acc.z += __bfloat162float(__ushort_as_bfloat16((unsigned short)(kv.y & 0xffffu)));
            acc.w += __bfloat162float(__ushort_as_bfloat16((unsigned short)(kv.y >> 16)));
            ++n;
          }
        }
        *reinterpret_cast<float4*>(S + c * kHeadDim + 4 * lane) = acc;
        if (lane == 0) cnt[c] += n;
      }
      __syncthreads();
      store_chunk(p0 + kKmChunk);
    }
    for (int x = tid; x < n_c * kHeadDim; x += blockDim.x) {
      const int c = x >> 7;
      if (cnt[c] > 0) Cf[x] = S[x] / (float)cnt[c];
    }
    __syncthreads();
    if (it + 1 < J.iters) {
      km_build_operands(Cf, Bf, cn2, n_c, n_c8);
      __syncthreads();
    }
  }

  // ---- outputs: centroids (bf16), assignment, member counts ----
  __nv_bfloat16* co = J.cent + ((int64_t)slab * J.wcap * n_c + (int64_t)wg * n_c) * kHeadDim;
  for (int x = tid; x < n_c * kHeadDim; x += blockDim.x) co[x] = __float2bfloat16_rn(Cf[x]);
  uint8_t* ao = J.assign + (int64_t)slab * J.ncap + tok0;
  int32_t* mc = J.mcnt + ((int64_t)slab * J.wcap + wg) * n_c * J.wu;
  for (int p = tid; p < Wt; p += blockDim.x) {
    const int c = a[p];
    ao[p] = (uint8_t)c;
    atomicAdd(mc + c * J.wu + p / J.Tu, 1);
  }
  int32_t* ms = J.msize + ((int64_t)slab * J.wcap + wg) * n_c;
  for (int c = tid; c < n_c; c += blockDim.x) ms[c] = cnt[c];
}

// Window metadata: first unit of each new window and the window of each window slot
// (slot = first unit / units per window; windows start on window boundaries).
__global__ void k_window_meta(int32_t* win_u0, int32_t* win_slot, int w_begin, int n_new,
                              int64_t first_unit, int wu) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= n_new) return;
  const int64_t u0 = first_unit + (int64_t)j * wu;
  win_u0[w_begin + j] = (int32_t)u0;
  win_slot[u0 / wu] = w_begin + j;
}

cudaError_t launch_kmeans(const __nv_bfloat16* keys, int64_t ncap, int n_slabs,
                          __nv_bfloat16* cent, uint8_t* assign, int32_t* mcnt, int32_t* msize,
                          int32_t* win_u0, int32_t* win_slot, int wcap, int w_begin, int n_new,
                          int64_t first_frame, int window_frames, int tokens_per_frame,
                          int frames_per_unit, int n_c, int iters, cudaStream_t s) {
  if (n_new <= 0) return cudaSuccess;
  const int wu = window_frames / frames_per_unit;
  const int Tu = tokens_per_frame * frames_per_unit;
  KmJob J;
  J.keys = keys;
  J.ncap = ncap;
  J.cent = cent;
  J.assign = assign;
  J.mcnt = mcnt;
  J.msize = msize;
  J.tok_first = first_frame * tokens_per_frame;
  J.Wt = window_frames * tokens_per_frame;
  J.Tu = Tu;
  J.wu = wu;
  J.w_begin = w_begin;
  J.wcap = wcap;
  J.n_c = n_c;
  J.n_c8 = (n_c + 7) & ~7;
  J.iters = iters;
  cudaError_t e = cudaMemset2DAsync(mcnt + (int64_t)w_begin * n_c * wu,
                                    (size_t)wcap * n_c * wu * sizeof(int32_t), 0,
                                    (size_t)n_new * n_c * wu * sizeof(int32_t), n_slabs, s);
  if (e != cudaSuccess) return e;
  k_window_meta<<<(n_new + 255) / 256, 256, 0, s>>>(win_u0, win_slot, w_begin, n_new,
                                                     first_frame / frames_per_unit, wu);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const size_t smem = kmeans_smem_bytes(n_c, J.Wt);
  e = ensure_smem((const void*)k_kmeans, (int)smem);
  if (e != cudaSuccess) return e;
  k_kmeans<<<dim3(n_new, n_slabs), kKmThreads, smem, s>>>(J);
  return cudaGetLastError();
}

}  // namespace ss
