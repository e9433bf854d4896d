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
// tokens). One CTA per (window, slab); every round streams the window's keys once, in
// tiles of 128 tokens, through a ring of shared-memory stages filled by tiled TMA
// copies (128-byte swizzle; a 4-D tensor map [slab][window][token][dim] whose token
// extent is the window, so a ragged last tile reads zeros). Per tile:
//   MMA1  D1[token][c]      = x . c_hi,  D1[token][n16 + c] = x . c_lo
//         (M = 128 tokens, N = 2 n16, K = 128 dims; c_hi = bf16(c), c_lo = bf16(c - c_hi),
//         so x . c carries ~16 significant bits of c; fp32 accumulation in TMEM)
//   assign a(x) = argmin_c ||c||^2 - 2 (x . c_hi + x . c_lo), lowest id on ties; the
//         epilogue writes the one-hot row of a(x) (bf16 1.0) into shared memory
//   MMA2  D2[dim][c] += sum_x x[dim] * onehot[x][c]
//         (M = 128 dims, N = 64, K = 128 tokens: the key tile read MN-major, the same
//         bytes as MMA1's K-major operand, so each key is loaded once per round)
// At the end of a round the member sums D2 and the counts give the new centroids
// (c = sum / count; an empty centroid keeps its value), from which the epilogue builds
// the next round's split operands. Every sum has a fixed order (the tensor core's
// accumulation order over the window's tiles), so results repeat bit for bit.
//
// Warp roles: warp 0 issues the TMA copies, warp 1 allocates tensor memory and issues
// the MMAs (one thread), warps 2-5 are the epilogue (thread e owns TMEM lane e: token e
// of a tile for MMA1, dim e for MMA2). All waits are bounded; a wait that gives up
// raises a shared abort flag that ends every role's loop, then the copies and MMAs in
// flight are drained and the tensor memory is freed.
// ---------------------------------------------------------------------------
constexpr int kTcStages = 4;
constexpr int kTcTile = 128;                            // tokens per tile
constexpr int kTcStageBytes = kTcTile * kHeadDim * 2;   // 32 KB
constexpr int kTcEpiWarps = 8;                          // two per TMEM lane quarter
constexpr int kTcEpiThreads = kTcEpiWarps * 32;
constexpr int kTcThreads = 64 + kTcEpiThreads;          // + TMA warp + MMA warp
constexpr int kTcMaxCentroids = 64;
constexpr int kTcMaxWindowTokens = 16384;
constexpr int kTcD1Bufs = 3;
// tensor memory: D1 in three buffers of 128 columns, D2 (64 columns), the fp32
// centroids (lane = dim, column = centroid; 64 columns)
constexpr uint32_t kTcTmemCols = 512;
constexpr uint32_t kTcD2Col = 384;
constexpr uint32_t kTcCfCol = 448;

struct TcJob {
  __nv_bfloat16* cent;        // [n_slabs][wcap * n_c][d]
  uint8_t* assign;            // [n_slabs][ncap]
  int32_t* mcnt;              // [n_slabs][wcap][n_c][wu]
  int32_t* msize;             // [n_slabs][wcap][n_c]
  const __nv_bfloat16* keys;  // [n_slabs][ncap][d] (initial centroids)
  int64_t ncap;
  int64_t tok_first;
  int Wt, Tu, wu, w_begin, wcap, n_c, n16, iters;
  uint32_t* status;           // device word: kStatusTimeout on a wait that gave up
};

struct TcBars {
  unsigned long long full[kTcStages], empty[kTcStages];
  unsigned long long d1_full[kTcD1Bufs], epi_done[kTcD1Bufs], mma2_done[2];
  unsigned long long d2_full, b1_ready, final_mma;
  uint32_t taddr;
  int abort;
  int cnt[kTcMaxCentroids];
  float cn2[kTcMaxCentroids];
  float part[4][kTcMaxCentroids];  // ||c||^2 partial sums of each lane quarter
  float xbest[2][2][kTcTile];      // [tile parity][centroid half][row]: nearest distance
  int xbc[2][2][kTcTile];          // and its centroid
};

// ring, B1 operand (128 rows x 256 B), one-hot rows (2 x 128 x 128 B), assignment bytes
size_t kmeans_tc_smem_bytes(int Wt) {
  return 1024 + (size_t)kTcStages * kTcStageBytes + 128 * 256 + 2 * kTcTile * 128 +
         (size_t)((Wt + 15) & ~15);
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

// Byte offset of centroid c in row r of a one-hot tile (MN-major, 128-byte swizzle).
__device__ __forceinline__ int onehot_off(int r, int c) {
  return r * 128 + ((((c >> 3) ^ (r & 7))) << 4) + (c & 7) * 2;
}

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 256;" ::: "memory"); }
// The two warps of one TMEM lane quarter (barriers 2-5).
__device__ __forceinline__ void pair_bar(int q) {
  asm volatile("bar.sync %0, 64;" ::"r"(2 + q) : "memory");
}

// New round operands from the fp32 centroids cf[0..31] = centroids 32 h .. 32 h + 31 at
// this thread's dim er: the centroids to tensor memory, the split rows of B1 and
// ||c||^2 of every centroid (squares summed over each warp's 32 dims by a shuffle tree,
// then over the four lane quarters in order: a fixed order). On return this thread holds
// the squared norms of its own 32 centroids in cn2r.
__device__ __forceinline__ void tc_round_operands(const float* cf, int h, int q, int lane, int er,
                                                  int ei, int n_c, int n16, unsigned char* B1,
                                                  TcBars& S, uint32_t cf_taddr, bool build_b1,
                                                  float (&cn2r)[32]) {
  float w[32];
#pragma unroll
  for (int c = 0; c < 32; ++c) w[c] = cf[c];
  tmem_st32(cf_taddr + 32 * h, w);
  if (build_b1)
#pragma unroll
    for (int c = 0; c < 32; ++c)
      if (32 * h + c < n16) tc_put_split(B1, 2 * n16, 32 * h + c, er, cf[c]);
#pragma unroll
  for (int c = 0; c < 32; ++c) {
    float v = cf[c] * cf[c];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    if (lane == 0) S.part[q][32 * h + c] = v;
  }
  epi_bar();
  if (ei < n16) {
    float s2 = INFINITY;   // padding centroids are never nearest
    if (ei < n_c) s2 = ((S.part[0][ei] + S.part[1][ei]) + S.part[2][ei]) + S.part[3][ei];
    S.cn2[ei] = s2;
  }
  epi_bar();
#pragma unroll
  for (int c = 0; c < 32; ++c) cn2r[c] = 32 * h + c < n16 ? S.cn2[32 * h + c] : INFINITY;
}

__global__ void __launch_bounds__(kTcThreads, 1)
    k_kmeans_tc(const __grid_constant__ CUtensorMap kmap, const TcJob J) {
  extern __shared__ unsigned char sm_raw[];
  __shared__ TcBars S;
  unsigned char* sm = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  unsigned char* ring = sm;
  unsigned char* B1 = ring + kTcStages * kTcStageBytes;
  unsigned char* onehot = B1 + 128 * 256;
  uint8_t* a_s = onehot + 2 * kTcTile * 128;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
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
    for (int b = 0; b < 2; ++b) mbar_init(smem_u32(&S.mma2_done[b]), 1);
    mbar_init(smem_u32(&S.d2_full), 1);
    mbar_init(smem_u32(&S.b1_ready), 1);
    mbar_init(smem_u32(&S.final_mma), 1);
    S.abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (tid < kTcMaxCentroids) S.cnt[tid] = 0;
  // the one-hot tiles start at zero; afterwards only the single 1.0 of a row changes
  for (int x = tid; x < 2 * kTcTile * 128 / 16; x += kTcThreads)
    reinterpret_cast<uint4*>(onehot)[x] = make_uint4(0u, 0u, 0u, 0u);
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
    // ---- MMA issuer: issues MMA1 of a tile as soon as its keys, a free D1 buffer and
    // (at a round's first tile) the round's operands are ready, and MMA2 of the oldest
    // tile whose one-hot rows are written, whichever comes first ----
    if (lane == 0) {
      const uint32_t id1 = idesc_bf16_f32(128, N1, false, false);
      const uint32_t id2 = idesc_bf16_f32(128, 64, true, true);
      const uint32_t b1s = smem_u32(B1);
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
            const uint32_t d1 = tbase + (uint32_t)buf * 128u;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const uint32_t ka = (k >> 2) * (kTcStageBytes / 2) + (k & 3) * 32;
              const uint32_t kb = (k >> 2) * (N1 * 128) + (k & 3) * 32;
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
          const uint32_t os = smem_u32(onehot + (n2 & 1) * (kTcTile * 128));
          const bool first = (n2 % ntile) == 0;
#pragma unroll
          for (int k = 0; k < 8; ++k)
            umma_bf16(tbase + kTcD2Col, sdesc_sw128(xs + k * 2048, kTcStageBytes / 2, 1024),
                      sdesc_sw128(os + k * 2048, kTcStageBytes / 2, 1024), id2,
                      (first && k == 0) ? 0u : 1u);
          umma_commit(smem_u32(&S.mma2_done[n2 & 1]));
          umma_commit(smem_u32(&S.empty[n2 % kTcStages]));
          if ((n2 % ntile) == ntile - 1) umma_commit(smem_u32(&S.d2_full));
          ++n2;
          did = true;
        }
        if (did) {
          idle = 0;
        } else if (__nanosleep(32), (++idle & 255u) == 0u) {
          // (the short sleep keeps this polling loop from taking the issue slots of the
          // epilogue warps that share its scheduler)
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
    // ---- epilogue: warps 2-9. Thread (h, er): TMEM lane er (token er of a tile for
    // MMA1, dim er for MMA2) and centroids 32 h .. 32 h + 31 ----
    // Every epilogue thread runs the same sequence of named barriers whatever happens
    // (a wait that gives up clears `ok` and the work is skipped, never the barriers).
    const int q = warp & 3;                      // the lane quarter this warp may access
    const int h = (warp - 2) >> 2;               // centroid half
    const int er = q * 32 + lane;
    const int ei = h * 128 + er;                 // 0 .. 255
    const uint32_t lane_addr = tbase + ((uint32_t)(q * 32) << 16);
    const __nv_bfloat16* X0 =
        J.keys + ((int64_t)slab * J.ncap + J.tok_first + (int64_t)wl * Wt) * kHeadDim;
    const int c_lo = 32 * h;                     // this thread's first centroid
    const int n_mine = max(0, min(32, n16 - c_lo));
    float cn2r[32];                              // ||c||^2 of this thread's centroids
    int prev[2] = {-1, -1};                      // the 1.0 each one-hot tile holds in row er
    bool ok = true;
    {
      // C0 = the window's first n_c keys; the round-0 operands
      float cf[32];
#pragma unroll
      for (int c = 0; c < 32; ++c)
        cf[c] = c_lo + c < n_c ? __bfloat162float(X0[(int64_t)(c_lo + c) * kHeadDim + er]) : 0.f;
      tc_round_operands(cf, h, q, lane, er, ei, n_c, n16, B1, S, lane_addr + kTcCfCol, true, cn2r);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    epi_bar();
    if (ei == 0) mbar_arrive(smem_u32(&S.b1_ready));

    for (int j = 0; j < J_tiles; ++j) {
      const int tile = j % ntile, round = j / ntile, buf = j % kTcD1Bufs, x = j & 1;
      ok = ok && tc_wait(smem_u32(&S.d1_full[buf]), (j / kTcD1Bufs) & 1, abort);
      tc_fence_after();
      // nearest of this half's centroids to token tile * 128 + er
      float best = INFINITY;
      int bc = c_lo;
      if (ok && n_mine > 0) {
        const uint32_t d1 = lane_addr + (uint32_t)buf * 128u;
        if (n_mine == 32) {
          float hi[32], lo[32];
          tmem_ld32x2(d1 + c_lo, d1 + n16 + c_lo, hi, lo);
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            const float dist = fmaf(-2.f, hi[c] + lo[c], cn2r[c]);
            if (dist < best) {
              best = dist;
              bc = c_lo + c;
            }
          }
        } else {
#pragma unroll
          for (int c0 = 0; c0 < 32; c0 += 16) {
            if (c0 < n_mine) {
              float hi[16], lo[16];
              tmem_ld16(d1 + c_lo + c0, hi);
              tmem_ld16(d1 + n16 + c_lo + c0, lo);
#pragma unroll
              for (int t = 0; t < 16; ++t) {
                const float dist = fmaf(-2.f, hi[t] + lo[t], cn2r[c0 + t]);
                if (dist < best) {
                  best = dist;
                  bc = c_lo + c0 + t;
                }
              }
            }
          }
        }
      }
      // the two halves' candidates (double-buffered by tile parity): the nearest, the
      // lower half on a tie (lower ids), is the row's centroid
      if (h == 1) {
        S.xbest[x][1][er] = best;
        S.xbc[x][1][er] = bc;
      }
      pair_bar(q);
      const int tok = tile * kTcTile + er;
      const bool valid = tok < Wt;
      if (h == 0) {
        if (S.xbest[x][1][er] < best) bc = S.xbc[x][1][er];
        ok = ok && (j < 2 || tc_wait(smem_u32(&S.mma2_done[x]), ((j >> 1) - 1) & 1, abort));
        if (ok) {
          // one 2-byte store clears the row's previous 1.0 in this tile, one sets the new
          unsigned char* t1 = onehot + x * (kTcTile * 128);
          if (prev[x] >= 0) *reinterpret_cast<uint16_t*>(t1 + onehot_off(er, prev[x])) = 0;
          prev[x] = valid ? bc : -1;
          if (valid) {
            *reinterpret_cast<uint16_t*>(t1 + onehot_off(er, bc)) = 0x3F80;   // bf16 1.0
            a_s[tok] = (uint8_t)bc;
            atomicAdd(&S.cnt[bc], 1);
          }
        }
        fence_proxy_async_smem();
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&S.epi_done[buf]));

      if (tile == ntile - 1) {
        // ---- end of a round: new centroids from the member sums ----
        epi_bar();                                            // every count is in
        ok = ok && tc_wait(smem_u32(&S.d2_full), round & 1, abort);
        tc_fence_after();
        float cf[32];
#pragma unroll
        for (int c = 0; c < 32; ++c) cf[c] = 0.f;
        if (ok) {
          float sum[32];
          tmem_ld32x2(lane_addr + kTcD2Col + c_lo, lane_addr + kTcCfCol + c_lo, sum, cf);
          // mean = sum * (1 / n): the reciprocal rounded once, then one rounded product
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            const int n = c_lo + c < n_c ? S.cnt[c_lo + c] : 0;
            if (n > 0) cf[c] = __fmul_rn(sum[c], __frcp_rn((float)n));
          }
        }
        const bool more = round + 1 < J.iters;
        tc_round_operands(cf, h, q, lane, er, ei, n_c, n16, B1, S, lane_addr + kTcCfCol,
                          ok && more, cn2r);
        if (more) {
          if (ei < kTcMaxCentroids) S.cnt[ei] = 0;
          fence_proxy_async_smem();
          tc_fence_before();
          epi_bar();
          if (ei == 0 && ok) mbar_arrive(smem_u32(&S.b1_ready));
        } else {
          // (the barriers below run whatever `write` says: abort may be raised between the
          // threads' reads of it)
          const bool write = !*abort;
          // ---- outputs: centroids (bf16), assignment, member counts ----
          __nv_bfloat16* co = J.cent + ((int64_t)slab * J.wcap * n_c +
                                        (int64_t)(J.w_begin + wl) * n_c) * kHeadDim;
#pragma unroll
          for (int c = 0; c < 32; ++c)
            if (write && c_lo + c < n_c)
              co[(int64_t)(c_lo + c) * kHeadDim + er] = __float2bfloat16_rn(cf[c]);
          // member counts per (centroid, unit of the window) tallied in shared memory (the
          // one-hot tiles' space: every MMA has completed), then written out
          const int64_t tok0 = J.tok_first + (int64_t)wl * Wt;
          uint8_t* ao = J.assign + (int64_t)slab * J.ncap + tok0;
          int32_t* mc = J.mcnt + ((int64_t)slab * J.wcap + J.w_begin + wl) * n_c * J.wu;
          int* tally = reinterpret_cast<int*>(onehot);
          const int n_tally = n_c * J.wu;
          const bool in_smem = n_tally <= 2 * kTcTile * 128 / 4;
          if (write && in_smem)
            for (int x = ei; x < n_tally; x += kTcEpiThreads) tally[x] = 0;
          epi_bar();
          for (int p = ei; write && p < Wt; p += kTcEpiThreads) {
            const int c = a_s[p];
            ao[p] = (uint8_t)c;
            if (in_smem) atomicAdd(&tally[c * J.wu + p / J.Tu], 1);
            else atomicAdd(mc + c * J.wu + p / J.Tu, 1);
          }
          epi_bar();
          if (write && in_smem)
            for (int x = ei; x < n_tally; x += kTcEpiThreads) mc[x] = tally[x];
          int32_t* ms = J.msize + ((int64_t)slab * J.wcap + J.w_begin + wl) * n_c;
          if (write && ei < n_c) ms[ei] = S.cnt[ei];
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
