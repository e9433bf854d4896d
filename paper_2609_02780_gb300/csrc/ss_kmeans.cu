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
//
// Two kernels: k_kmeans_tc (tcgen05 MMAs, TMA-staged keys, one key read per round) for
// n_c <= 64 and windows of <= 16384 tokens, and k_kmeans (mma.sync) for the rest.
#include "ss_internal.cuh"
#include "ss_device.cuh"
#include "ss_tc.cuh"

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

// ---------------------------------------------------------------------------
// Lloyd rounds on the 5th-generation tensor cores (n_c <= 64, windows of <= 16384
// tokens). One CTA per (window, slab), sized so that two CTAs share an SM: a CTA's rounds
// are a chain of dependent steps per tile, and the second CTA's tiles fill its gaps.
// Every round streams the window's keys once, in tiles of 128 tokens, through two
// shared-memory stages filled by tiled TMA copies (128-byte swizzle; a 4-D tensor map
// [slab][window][token][dim] whose token extent is the window, so a ragged last tile
// reads zeros). Per tile:
//   MMA1  D1[token][c] = x . c_hi + x . c_lo, the lo products accumulated onto the hi ones
//         (M = 128 tokens, N = n16, K = 2 x 128 dims; c_hi = bf16(c), c_lo = bf16(c - c_hi),
//         so x . c carries ~16 significant bits of c; fp32 accumulation in TMEM)
//   assign a(x) = argmin_c ||c||^2 - 2 x . c, lowest id on ties; the epilogue writes the
//         one-hot row of a(x) (bf16 1.0) into shared memory
//   MMA2  D2[dim][c] += sum_x x[dim] * onehot[x][c]
//         (M = 128 dims, N = 64, K = 128 tokens: the key tile read MN-major, the same
//         bytes as MMA1's K-major operand, so each key is loaded once per round)
// At the end of a round the member sums D2 and the counts give the new centroids
// (c = sum * (1 / count); an empty centroid keeps its value), from which the epilogue
// builds the next round's split operands. Every sum has a fixed order (the tensor core's
// accumulation order over the window's tiles), so results repeat bit for bit. The last
// round's assignments and member counts per (centroid, unit) go straight to global memory.
//
// Warp roles: warp 0 issues the TMA copies, warp 1 allocates tensor memory and issues
// the MMAs (one thread), warps 2-5 are the epilogue (thread e owns TMEM lane e: token e
// of a tile for MMA1, dim e for MMA2 and the update). All waits are bounded; a wait that
// gives up raises a shared abort flag that ends every role's loop, then the copies and
// MMAs in flight are drained and the tensor memory is freed. Every epilogue thread runs
// the same sequence of named barriers whatever happens.
// ---------------------------------------------------------------------------
constexpr int kTcStages = 2;
constexpr int kTcTile = 128;                            // tokens per tile
constexpr int kTcStageBytes = kTcTile * kHeadDim * 2;   // 32 KB
constexpr int kTcEpiThreads = 128;                      // one per TMEM lane
constexpr int kTcThreads = 64 + kTcEpiThreads;          // + TMA warp + MMA warp
constexpr int kTcMaxCentroids = 64;
constexpr int kTcMaxWindowTokens = 16384;
constexpr int kTcD1Bufs = 2;
constexpr int kTcB1Bytes = 128 * 256;                   // hi and lo rows, two 64-dim halves
constexpr int kTcOneHotBytes = kTcTile * 128;           // 128 tokens x 64 centroids (bf16)
// tensor memory (256 columns, half an SM's): D1 in two buffers at 0 and 64 (n16 columns
// used), D2 at 128 (64 columns), the fp32 centroids at 192 (lane = dim, column = centroid)
constexpr uint32_t kTcTmemCols = 256;
constexpr uint32_t kTcD2Col = 128;
constexpr uint32_t kTcCfCol = 192;

struct TcJob {
  __nv_bfloat16* cent;        // [n_slabs][wcap * n_c][d]
  uint8_t* assign;            // [n_slabs][ncap]
  int32_t* mcnt;              // [n_slabs][wcap][n_c][wu] (zeroed by the launcher)
  int32_t* msize;             // [n_slabs][wcap][n_c]
  const __nv_bfloat16* keys;  // [n_slabs][ncap][d] (initial centroids)
  int64_t ncap;
  int64_t tok_first;
  int Wt, Tu, wu, w_begin, wcap, n_c, n16, iters;
  uint32_t* status;           // device word: kStatusTimeout on a wait that gave up
};

// Barriers and per-round tallies, at the end of the dynamic shared memory (the CTA has no
// static shared memory, so the dynamic region starts on the 1024-byte boundary the
// swizzled tiles need).
struct TcBars {
  unsigned long long full[kTcStages], empty[kTcStages];
  unsigned long long d1_full[kTcD1Bufs], epi_done[kTcD1Bufs], mma2_done;
  unsigned long long d2_full, b1_ready, final_mma;
  uint32_t taddr;
  int abort;
  int cnt[kTcMaxCentroids];
  float cn2[kTcMaxCentroids];
};

// ring, B1 operand, one-hot rows, barriers
size_t kmeans_tc_smem_bytes(int Wt) {
  (void)Wt;
  return (size_t)kTcStages * kTcStageBytes + kTcB1Bytes + kTcOneHotBytes + sizeof(TcBars);
}

bool kmeans_tc_supported(int n_c, int Wt) {
  return n_c <= kTcMaxCentroids && Wt <= kTcMaxWindowTokens && Wt >= 1;
}

// Bounded wait that also gives up when another role raised the abort flag; a wait that
// runs out raises it.
__device__ __forceinline__ bool tc_wait(uint32_t bar, uint32_t parity, volatile int* abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t i = 1; i < kDefaultWaitPolls; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 255u) == 0u) {
      if (*abort) return false;
      if (global_ns() - t0 > 1000000000ull) break;
    }
  }
  *abort = 1;
  return false;
}

// Writes centroid c's split operand rows (c_hi in row c, c_lo in row n16 + c) at dim e of
// the 128-byte swizzled K-major tile B1 (two halves of 64 dims, each N1 rows x 128 B).
__device__ __forceinline__ void tc_put_split(unsigned char* B1, int N1, int row, int e, float x) {
  const __nv_bfloat16 hi = __float2bfloat16_rn(x);
  const __nv_bfloat16 lo = __float2bfloat16_rn(x - __bfloat162float(hi));
  const int half = e >> 6, b = (e & 63) * 2;
  const int r2 = row + (N1 >> 1);
  unsigned char* h0 = B1 + half * (N1 * 128);
  *reinterpret_cast<__nv_bfloat16*>(h0 + row * 128 + ((((b >> 4) ^ (row & 7))) << 4) + (b & 15)) = hi;
  *reinterpret_cast<__nv_bfloat16*>(h0 + r2 * 128 + ((((b >> 4) ^ (r2 & 7))) << 4) + (b & 15)) = lo;
}

// Byte offset of centroid c in row r of the one-hot tile (MN-major, 128-byte swizzle).
__device__ __forceinline__ int onehot_off(int r, int c) {
  return r * 128 + ((((c >> 3) ^ (r & 7))) << 4) + (c & 7) * 2;
}

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// One round's operands from 32 fp32 centroids cf[0..31] = centroids c0 .. c0 + 31 at this
// thread's dim e: the centroids to tensor memory, their split rows of B1 (when `b1`), and
// their squares summed over the warp's 32 dims by a shuffle tree into part[quarter][c].
__device__ __forceinline__ void tc_put_centroids(const float (&cf)[32], int c0, int e, int q,
                                                 int lane, int n16, unsigned char* B1,
                                                 uint32_t cf_taddr, bool b1, float* part) {
  tmem_st32(cf_taddr + (uint32_t)c0, cf);
  if (b1)
#pragma unroll
    for (int c = 0; c < 32; ++c)
      if (c0 + c < n16) tc_put_split(B1, 2 * n16, c0 + c, e, cf[c]);
#pragma unroll
  for (int c = 0; c < 32; ++c) {
    float v = cf[c] * cf[c];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    if (lane == 0) part[q * kTcMaxCentroids + c0 + c] = v;
  }
}

// ||c||^2 of every centroid from the four lane quarters' partial sums (in quarter order:
// a fixed order); padding centroids get +inf, so they are never nearest.
__device__ __forceinline__ void tc_norms(TcBars& S, const float* part, int e, int n_c, int n16) {
  if (e < n16)
    S.cn2[e] = e < n_c ? ((part[e] + part[kTcMaxCentroids + e]) + part[2 * kTcMaxCentroids + e]) +
                             part[3 * kTcMaxCentroids + e]
                       : INFINITY;
}

__global__ void __launch_bounds__(256, 2)
    k_kmeans_tc(const __grid_constant__ CUtensorMap kmap, const TcJob J) {
  extern __shared__ __align__(1024) unsigned char sm[];
  unsigned char* ring = sm;
  unsigned char* B1 = ring + kTcStages * kTcStageBytes;
  unsigned char* onehot = B1 + kTcB1Bytes;
  TcBars& S = *reinterpret_cast<TcBars*>(onehot + kTcOneHotBytes);
  float* part = reinterpret_cast<float*>(onehot);    // the one-hot space between rounds

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if ((smem_u32(sm) & 1023u) != 0u) {                // the swizzled tiles need the boundary
    if (tid == 0) atomicOr(J.status, kStatusInternal);
    return;
  }
  const int wl = blockIdx.x, slab = blockIdx.y;
  const int n_c = J.n_c, n16 = J.n16, N1 = 2 * n16, Wt = J.Wt;
  const int ntile = (Wt + kTcTile - 1) / kTcTile;
  const int J_tiles = J.iters * ntile;
  volatile int* abort = &S.abort;

  if (tid == 0) {
    for (int s = 0; s < kTcStages; ++s) {
      mbar_init(smem_u32(&S.full[s]), 1);
      mbar_init(smem_u32(&S.empty[s]), 1);
    }
    for (int b = 0; b < kTcD1Bufs; ++b) {
      mbar_init(smem_u32(&S.d1_full[b]), 1);
      mbar_init(smem_u32(&S.epi_done[b]), kTcEpiThreads);
    }
    mbar_init(smem_u32(&S.mma2_done), 1);
    mbar_init(smem_u32(&S.d2_full), 1);
    mbar_init(smem_u32(&S.b1_ready), 1);
    mbar_init(smem_u32(&S.final_mma), 1);
    S.abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (tid < kTcMaxCentroids) S.cnt[tid] = 0;
  if (warp == 1) {
    tmem_alloc(smem_u32(&S.taddr), kTcTmemCols);
    tmem_relinquish();
  }
  if (warp == 0 && lane == 0) tma_prefetch_map(&kmap);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = S.taddr;

  if (warp == 0) {
    // ---- TMA producer ----
    if (lane == 0) {
      int issued_last[kTcStages];
      for (int s = 0; s < kTcStages; ++s) issued_last[s] = -1;
      for (int j = 0; j < J_tiles && !*abort; ++j) {
        const int st = j % kTcStages;
        if (j >= kTcStages && !tc_wait(smem_u32(&S.empty[st]), ((j / kTcStages) - 1) & 1, abort))
          break;
        const uint32_t bar = smem_u32(&S.full[st]);
        const uint32_t dst = smem_u32(ring + st * kTcStageBytes);
        const int y = (j % ntile) * kTcTile;
        mbar_expect_tx(bar, kTcStageBytes);
        tma_load_4d(dst, &kmap, bar, 0, y, wl, slab);
        tma_load_4d(dst + kTcStageBytes / 2, &kmap, bar, 64, y, wl, slab);
        issued_last[st] = j;
      }
      // let every issued copy land before the CTA can exit
      for (int s = 0; s < kTcStages; ++s)
        if (issued_last[s] >= 0)
          mbar_wait_bounded(smem_u32(&S.full[s]), (issued_last[s] / kTcStages) & 1);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---- MMA issuer: MMA1 of a tile as soon as its keys, a free D1 buffer and (at a
    // round's first tile) the round's operands are ready; MMA2 of the oldest tile whose
    // one-hot rows are written ----
    if (lane == 0) {
      const uint32_t id1 = idesc_bf16_f32(128, n16, false, false);
      const uint32_t id2 = idesc_bf16_f32(128, 64, true, true);
      const uint32_t b1s = smem_u32(B1);
      const uint32_t os = smem_u32(onehot);
      int n1 = 0, n2 = 0;                       // next tile for MMA1, for MMA2
      uint64_t t_idle = 0;
      uint32_t idle = 0;
      while (n2 < J_tiles) {
        bool did = false;
        if (n1 < J_tiles && n1 - n2 < kTcD1Bufs) {
          const int tile = n1 % ntile, st = n1 % kTcStages, buf = n1 % kTcD1Bufs;
          // (non-blocking tests: a suspended try_wait here would hold back the other queue)
          bool ready = tile != 0 || (n2 == n1 && mbar_test_wait(smem_u32(&S.b1_ready), (n1 / ntile) & 1));
          ready = ready && mbar_test_wait(smem_u32(&S.full[st]), (n1 / kTcStages) & 1);
          if (ready) {
            tc_fence_after();
            const uint32_t as = smem_u32(ring + st * kTcStageBytes);
            const uint32_t d1 = tbase + (uint32_t)buf * 64u;
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              const int kk = k & 7;
              const uint32_t ka = (kk >> 2) * (kTcStageBytes / 2) + (kk & 3) * 32;
              const uint32_t kb = (kk >> 2) * (N1 * 128) + (kk & 3) * 32 + (k >> 3) * (n16 * 128);
              umma_bf16(d1, sdesc_sw128(as + ka, 16, 1024), sdesc_sw128(b1s + kb, 16, 1024), id1,
                        k > 0 ? 1u : 0u);
            }
            umma_commit(smem_u32(&S.d1_full[buf]));
            ++n1;
            did = true;
          }
        }
        if (n2 < n1 && mbar_test_wait(smem_u32(&S.epi_done[n2 % kTcD1Bufs]), (n2 / kTcD1Bufs) & 1)) {
          tc_fence_after();
          const uint32_t xs = smem_u32(ring + (n2 % kTcStages) * kTcStageBytes);
          const bool first = (n2 % ntile) == 0;
#pragma unroll
          for (int k = 0; k < 8; ++k)
            umma_bf16(tbase + kTcD2Col, sdesc_sw128(xs + k * 2048, kTcStageBytes / 2, 1024),
                      sdesc_sw128(os + k * 2048, kTcStageBytes / 2, 1024), id2,
                      (first && k == 0) ? 0u : 1u);
          umma_commit(smem_u32(&S.mma2_done));
          umma_commit(smem_u32(&S.empty[n2 % kTcStages]));
          if ((n2 % ntile) == ntile - 1) umma_commit(smem_u32(&S.d2_full));
          ++n2;
          did = true;
        }
        if (did) {
          idle = 0;
        } else if (__nanosleep(32), (++idle & 255u) == 0u) {
          // bounded: give up after ~1 s without progress, or when another role did
          const uint64_t now = global_ns();
          if (idle == 256u) t_idle = now;
          if (*abort || now - t_idle > 1000000000ull || idle >= kDefaultWaitPolls) {
            *abort = 1;
            break;
          }
        }
      }
      // every MMA issued has completed before the tensor memory is freed
      umma_commit(smem_u32(&S.final_mma));
      mbar_wait_bounded(smem_u32(&S.final_mma), 0);
    }
    __syncwarp();
  } else {
    // ---- epilogue: warps 2-5. Thread e: TMEM lane e (token e of a tile for MMA1, dim e
    // for MMA2 and the update) ----
    const int q = warp & 3;                      // the lane quarter this warp may access
    const int e = q * 32 + lane;
    const uint32_t lane_addr = tbase + ((uint32_t)(q * 32) << 16);
    const __nv_bfloat16* X0 =
        J.keys + ((int64_t)slab * J.ncap + J.tok_first + (int64_t)wl * Wt) * kHeadDim;
    const int64_t tok0 = J.tok_first + (int64_t)wl * Wt;
    uint8_t* ao = J.assign + (int64_t)slab * J.ncap + tok0;
    int32_t* mc = J.mcnt + ((int64_t)slab * J.wcap + J.w_begin + wl) * n_c * J.wu;
    int prev = -1;                               // the 1.0 the one-hot tile holds in row e
    bool ok = true;
    {
      // C0 = the window's first n_c keys; the round-0 operands (the one-hot space holds
      // the norms' partial sums first, then is cleared)
#pragma unroll 1
      for (int c0 = 0; c0 < 64; c0 += 32) {
        float cf[32];
#pragma unroll
        for (int c = 0; c < 32; ++c)
          cf[c] = c0 + c < n_c ? __bfloat162float(X0[(int64_t)(c0 + c) * kHeadDim + e]) : 0.f;
        tc_put_centroids(cf, c0, e, q, lane, n16, B1, lane_addr + kTcCfCol, true, part);
      }
      epi_bar();
      tc_norms(S, part, e, n_c, n16);
      epi_bar();
#pragma unroll
      for (int x = 0; x < kTcOneHotBytes / 16 / kTcEpiThreads; ++x)
        reinterpret_cast<uint4*>(onehot)[x * kTcEpiThreads + e] = make_uint4(0u, 0u, 0u, 0u);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    epi_bar();
    if (e == 0) mbar_arrive(smem_u32(&S.b1_ready));

    for (int j = 0; j < J_tiles; ++j) {
      const int tile = j % ntile, round = j / ntile, buf = j % kTcD1Bufs;
      const bool last = round + 1 == J.iters;
      ok = ok && tc_wait(smem_u32(&S.d1_full[buf]), (j / kTcD1Bufs) & 1, abort);
      tc_fence_after();
      // nearest centroid of token tile * 128 + e (chunks of 32 columns)
      float best = INFINITY;
      int bc = 0;
      if (ok && n16 == 64) {
        // all 64 columns in one load and one wait
        const uint32_t d1 = lane_addr + (uint32_t)buf * 64u;
        float xa[32], xb[32];
        tmem_ld32x2(d1, d1 + 32u, xa, xb);
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          const float dist = fmaf(-2.f, xa[c], S.cn2[c]);
          if (dist < best) {
            best = dist;
            bc = c;
          }
        }
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          const float dist = fmaf(-2.f, xb[c], S.cn2[32 + c]);
          if (dist < best) {
            best = dist;
            bc = 32 + c;
          }
        }
      } else if (ok) {
        const uint32_t d1 = lane_addr + (uint32_t)buf * 64u;
#pragma unroll 1
        for (int c0 = 0; c0 < n16; c0 += 32) {
          if (n16 - c0 >= 32) {
            float xc[32];
            tmem_ld32(d1 + (uint32_t)c0, xc);
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              const float dist = fmaf(-2.f, xc[c], S.cn2[c0 + c]);
              if (dist < best) {
                best = dist;
                bc = c0 + c;
              }
            }
          } else {
            float xc[16];
            tmem_ld16(d1 + (uint32_t)c0, xc);
#pragma unroll
            for (int c = 0; c < 16; ++c) {
              const float dist = fmaf(-2.f, xc[c], S.cn2[c0 + c]);
              if (dist < best) {
                best = dist;
                bc = c0 + c;
              }
            }
          }
        }
      }
      const int tok = tile * kTcTile + e;
      const bool valid = tok < Wt;
      // the one-hot tile is free once MMA2 of the previous tile has completed
      ok = ok && (j == 0 || tc_wait(smem_u32(&S.mma2_done), (j - 1) & 1, abort));
      if (ok) {
        // one 2-byte store clears the row's previous 1.0, one sets the new
        if (prev >= 0) *reinterpret_cast<uint16_t*>(onehot + onehot_off(e, prev)) = 0;
        prev = valid ? bc : -1;
        if (valid) {
          *reinterpret_cast<uint16_t*>(onehot + onehot_off(e, bc)) = 0x3F80;   // bf16 1.0
          atomicAdd(&S.cnt[bc], 1);
          if (last) {
            ao[tok] = (uint8_t)bc;
            atomicAdd(mc + bc * J.wu + tok / J.Tu, 1);
          }
        }
      }
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(smem_u32(&S.epi_done[buf]));

      if (tile == ntile - 1) {
        // ---- end of a round: new centroids from the member sums ----
        epi_bar();                                            // every count is in
        ok = ok && tc_wait(smem_u32(&S.d2_full), round & 1, abort);
        tc_fence_after();
        // (every MMA of the round has completed: the one-hot space is free)
        const bool write = !*abort;
        __nv_bfloat16* co = J.cent + ((int64_t)slab * J.wcap * n_c +
                                      (int64_t)(J.w_begin + wl) * n_c) * kHeadDim;
#pragma unroll 1
        for (int c0 = 0; c0 < 64; c0 += 32) {
          float cf[32];
#pragma unroll
          for (int c = 0; c < 32; ++c) cf[c] = 0.f;
          if (ok) {
            float sum[32];
            tmem_ld32x2(lane_addr + kTcD2Col + (uint32_t)c0, lane_addr + kTcCfCol + (uint32_t)c0,
                        sum, cf);
            // mean = sum * (1 / n): the reciprocal rounded once, then one rounded product
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              const int n = c0 + c < n_c ? S.cnt[c0 + c] : 0;
              if (n > 0) cf[c] = __fmul_rn(sum[c], __frcp_rn((float)n));
            }
          }
          if (last) {
#pragma unroll
            for (int c = 0; c < 32; ++c)
              if (write && c0 + c < n_c) co[(int64_t)(c0 + c) * kHeadDim + e] = __float2bfloat16_rn(cf[c]);
          } else {
            tc_put_centroids(cf, c0, e, q, lane, n16, B1, lane_addr + kTcCfCol, ok, part);
          }
        }
        if (!last) {
          epi_bar();
          tc_norms(S, part, e, n_c, n16);
          if (e < kTcMaxCentroids) S.cnt[e] = 0;
          epi_bar();
          // the one-hot space back to zeros (the row's previous 1.0 is gone with it)
#pragma unroll
          for (int x = 0; x < kTcOneHotBytes / 16 / kTcEpiThreads; ++x)
            reinterpret_cast<uint4*>(onehot)[x * kTcEpiThreads + e] = make_uint4(0u, 0u, 0u, 0u);
          prev = -1;
          fence_proxy_async_smem();
          tc_fence_before();
          epi_bar();
          if (e == 0 && ok) mbar_arrive(smem_u32(&S.b1_ready));
        } else {
          epi_bar();
          int32_t* ms = J.msize + ((int64_t)slab * J.wcap + J.w_begin + wl) * n_c;
          if (write && e < n_c) ms[e] = S.cnt[e];
        }
      }
    }
    epi_bar();
  }
  tc_fence_before();
  __syncthreads();
  if (tid == 0 && *abort) atomicOr(J.status, kStatusTimeout);
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tbase, kTcTmemCols);
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
                          int frames_per_unit, int n_c, int iters, uint32_t* status,
                          cudaStream_t s) {
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
  if (kmeans_tc_supported(n_c, J.Wt)) {
    // keys of this call's windows as [slab][window][token][dim]: the token extent is the
    // window, so a tile past the window's end reads zeros
    const uint64_t dims[4] = {(uint64_t)kHeadDim, (uint64_t)J.Wt, (uint64_t)n_new, (uint64_t)n_slabs};
    const uint64_t strides[3] = {(uint64_t)kHeadDim * 2, (uint64_t)J.Wt * kHeadDim * 2,
                                 (uint64_t)ncap * kHeadDim * 2};
    const uint32_t box[4] = {64, kTcTile, 1, 1};
    CUtensorMap map;
    e = encode_bf16_map(&map, keys + J.tok_first * kHeadDim, 4, dims, strides, box);
    if (e != cudaSuccess) return e;
    TcJob T;
    T.cent = cent;
    T.assign = assign;
    T.mcnt = mcnt;
    T.msize = msize;
    T.keys = keys;
    T.ncap = ncap;
    T.tok_first = J.tok_first;
    T.Wt = J.Wt;
    T.Tu = Tu;
    T.wu = wu;
    T.w_begin = w_begin;
    T.wcap = wcap;
    T.n_c = n_c;
    T.n16 = (n_c + 15) & ~15;
    T.iters = iters;
    T.status = status;
    const size_t smem = kmeans_tc_smem_bytes(J.Wt);
    e = ensure_smem((const void*)k_kmeans_tc, (int)smem);
    if (e != cudaSuccess) return e;
    k_kmeans_tc<<<dim3(n_new, n_slabs), kTcThreads, smem, s>>>(map, T);
    return cudaGetLastError();
  }
  const size_t smem = kmeans_smem_bytes(n_c, J.Wt);
  e = ensure_smem((const void*)k_kmeans, (int)smem);
  if (e != cudaSuccess) return e;
  k_kmeans<<<dim3(n_new, n_slabs), kKmThreads, smem, s>>>(J);
  return cudaGetLastError();
}

}  // namespace ss
