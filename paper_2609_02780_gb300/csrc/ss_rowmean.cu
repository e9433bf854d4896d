// Lists ranked by the mean over the question rows of the rows' softmax weights.
//
// Sec. 4.2 scores the candidates against the final prompt token. With every question row
// attending on its own, token p's weight in list (layer i, query head h) is
//   alpha(p) = (1/R) sum_r 2^(s_r(p) - M_r) / L_r,   s_r(p) = q_r . k_p * log2(e) / sqrt(d),
// where (M_r, L_r) are row r's softmax statistics over the history tokens. Every row's
// statistics must be known before any alpha, so the keys are read twice:
//   pass 1  k_rm_stats: S^T = Q . K^T on the tcgen05 tensor cores, the question rows of a
//           key head's G query heads on the TMEM lanes (M = 128 rows per MMA, N = 128
//           tokens, K = 128 dims), each epilogue thread keeping its row's online
//           (max, sum) over the tokens; partial statistics per CTA, combined in a fixed
//           order by k_rm_combine;
//   pass 2  k_rm_alpha: S = K . Q^T, the tokens on the TMEM lanes (M = 128 tokens,
//           N = the G * R rows), each epilogue thread summing its token's weights over a
//           head's rows; alpha goes to the list's dense row, ranked by the general top-k
//           (ids = positions) and summed per unit by the general mass kernel.
// Keys reach shared memory through tiled TMA copies (128-byte swizzle), the question
// rows once per CTA. The rows of head h occupy positions h * Rp .. h * Rp + R - 1
// (Rp = R rounded up to 16; the padding rows are zero and ignored).
#include "ss_internal.cuh"
#include "ss_device.cuh"
#include "ss_tc.cuh"
#include "ss_pack.cuh"

namespace ss {

constexpr int kRmTile = 128;                           // tokens per tile
constexpr int kRmStageBytes = kRmTile * kHeadDim * 2;  // 32 KB

struct RmJob {
  int prob;            // problem index in the batch
  int Rp;              // rows per head, padded to 16
  int GRp;             // G * Rp
  int chunks;          // CTAs per slab
  int nbuf;            // TMEM accumulator buffers
  int stages;          // key stages
  float2* part;        // [slabs][GRp][chunks] partial (m, l) of pass 1
  float2* stat;        // [slabs][GRp] (M, 1 / L) of every row
};

__device__ __forceinline__ void rm_bar(int nthreads) {
  asm volatile("bar.sync 1, %0;" ::"r"(nthreads) : "memory");
}

// Copies the question rows of slab (i, g) into a 128-byte swizzled K-major operand:
// row rho = h * Rp + r (h < G, r < R) from q[i][r][g * G + h][:], zero elsewhere, in
// blocks of `rows_per_block` rows (each block: two halves of rows_per_block x 128 B).
__device__ void rm_load_q(const Prob& P, int slab, int Rp, int n_rows, int rows_per_block,
                          unsigned char* dst, int t0, int nt) {
  const int i = slab / P.Hkv, g = slab - i * P.Hkv;
  const int64_t row_stride = (int64_t)P.Hq * kHeadDim;
  // eight 16-byte chunks per thread loaded together, then stored (one memory latency
  // per eight)
  for (int e0 = t0; e0 < n_rows * 16; e0 += 8 * nt) {
    uint4 v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int e = e0 + u * nt;
      const int rho = e >> 4, c = e & 15;
      const int h = rho / Rp, r = rho - h * Rp;
      v[u] = make_uint4(0u, 0u, 0u, 0u);
      if (e < n_rows * 16 && h < P.G && r < P.R)
        v[u] = *reinterpret_cast<const uint4*>(P.q + (int64_t)i * P.R * row_stride +
                                               (int64_t)r * row_stride +
                                               (int64_t)(g * P.G + h) * kHeadDim + 8 * c);
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int e = e0 + u * nt;
      if (e >= n_rows * 16) break;
      const int rho = e >> 4, c = e & 15;
      const int b = rho / rows_per_block, n = rho - b * rows_per_block;
      unsigned char* blk = dst + (size_t)b * rows_per_block * 256;
      *reinterpret_cast<uint4*>(blk + (c >> 3) * (rows_per_block * 128) + n * 128 +
                                ((((c & 7) ^ (n & 7))) << 4)) = v[u];
    }
  }
}

// Bounded wait that gives up when another role raised the abort flag.
__device__ __forceinline__ bool rm_wait(uint32_t bar, uint32_t parity, volatile int* abort) {
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

struct RmBars {
  unsigned long long full[4], empty[4], d_full[2], epi_done[2], q_ready, final_mma;
  uint32_t taddr;
  int abort;
};

// Producer / MMA / drain shared by both passes. The MMA thread calls `mma(j, stage, buf)`
// for each tile j once its keys and a free accumulator buffer are there.
template <typename MmaFn>
__device__ void rm_pipeline(const CUtensorMap* kmap, RmBars& S, unsigned char* ring, int stages,
                            int nbuf, int n_epi, int n_tiles, int64_t row0, MmaFn&& mma) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &S.abort;
  if (warp == 0 && lane == 0) {
    int issued_last[4] = {-1, -1, -1, -1};
    for (int j = 0; j < n_tiles && !*abort; ++j) {
      const int st = j % stages;
      if (j >= stages && !rm_wait(smem_u32(&S.empty[st]), ((j / stages) - 1) & 1, abort)) break;
      const uint32_t bar = smem_u32(&S.full[st]);
      const uint32_t dst = smem_u32(ring + st * kRmStageBytes);
      const int y = (int)(row0 + (int64_t)j * kRmTile);
      mbar_expect_tx(bar, kRmStageBytes);
      tma_load_2d(dst, kmap, bar, 0, y);
      tma_load_2d(dst + kRmStageBytes / 2, kmap, bar, 64, y);
      issued_last[st] = j;
    }
    for (int s = 0; s < stages; ++s)
      if (issued_last[s] >= 0) mbar_wait_bounded(smem_u32(&S.full[s]), (issued_last[s] / stages) & 1);
  } else if (warp == 1 && lane == 0) {
    if (rm_wait(smem_u32(&S.q_ready), 0, abort)) {
      for (int j = 0; j < n_tiles; ++j) {
        const int st = j % stages, buf = j % nbuf;
        if (j >= nbuf && !rm_wait(smem_u32(&S.epi_done[buf]), ((j / nbuf) - 1) & 1, abort)) break;
        if (!rm_wait(smem_u32(&S.full[st]), (j / stages) & 1, abort)) break;
        tc_fence_after();
        mma(j, smem_u32(ring + st * kRmStageBytes), buf);
        umma_commit(smem_u32(&S.d_full[buf]));
        umma_commit(smem_u32(&S.empty[st]));
      }
    }
    umma_commit(smem_u32(&S.final_mma));
    mbar_wait_bounded(smem_u32(&S.final_mma), 0);
  }
  (void)n_epi;
}

__device__ __forceinline__ void rm_init(RmBars& S, int stages, int nbuf, int n_epi, uint32_t cols) {
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(smem_u32(&S.full[s]), 1);
      mbar_init(smem_u32(&S.empty[s]), 1);
    }
    for (int b = 0; b < nbuf; ++b) {
      mbar_init(smem_u32(&S.d_full[b]), 1);
      mbar_init(smem_u32(&S.epi_done[b]), n_epi);
    }
    mbar_init(smem_u32(&S.q_ready), 1);
    mbar_init(smem_u32(&S.final_mma), 1);
    S.abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&S.taddr), cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
}

// The tiles [t0, t1) of history tokens of chunk `c` of a slab.
__device__ __forceinline__ void rm_chunk(const Prob& P, int chunks, int c, int& t0, int& t1) {
  const int n_tok = P.Uh * P.Tu;
  const int T = (n_tok + kRmTile - 1) / kRmTile;
  t0 = (int)((int64_t)T * c / chunks);
  t1 = (int)((int64_t)T * (c + 1) / chunks);
}

// ---------------------------------------------------------------------------
// Pass 1: per-row (max, sum) of the log2-scaled scores over the chunk's tokens.
// Warps: 0 TMA, 1 MMA (+ TMEM), then 4 per (128-row block, column part): NMB blocks,
// each tile's 128 token columns split in CS parts, every part keeping its own (max, sum)
// per row, combined in part order at the end.
// ---------------------------------------------------------------------------
// Launch bound: the block's threads rounded up to whole groups of four warps (the unit
// in which a block's registers are allocated).
constexpr int rm_bound(int threads) { return (threads + 127) / 128 * 128; }

template <int NMB, int CS>
__global__ void __launch_bounds__(rm_bound(64 + 128 * NMB * CS), 1)
    k_rm_stats(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ Batch B,
               const RmJob J) {
  extern __shared__ unsigned char sm_raw[];
  __shared__ RmBars S;
  __shared__ float2 part_s[(CS > 1 ? CS - 1 : 1) * NMB * 128];
  unsigned char* sm = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  unsigned char* qs = sm;                                // NMB x 32 KB
  unsigned char* ring = qs + NMB * 32768;
  constexpr int n_epi = 128 * NMB * CS;
  constexpr int CW = kRmTile / CS;                       // columns of a part
  constexpr int PW = CW >= 64 ? 64 : 32;                 // columns per TMEM load
  const int nbuf = J.nbuf, stages = J.stages;
  const uint32_t cols = nbuf * NMB * 128 <= 256 ? 256u : 512u;
  rm_init(S, stages, nbuf, n_epi, cols);
  const uint32_t tbase = S.taddr;
  const Prob& P = B.p[J.prob];
  const int slab = blockIdx.y, chunk = blockIdx.x;
  int t0, t1;
  rm_chunk(P, J.chunks, chunk, t0, t1);
  const int n_tiles = t1 - t0;
  const int n_tok = P.Uh * P.Tu;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &S.abort;
  if (warp < 2) {
    rm_pipeline(&kmap, S, ring, stages, nbuf, n_epi, n_tiles,
                (int64_t)slab * P.ncap + (int64_t)t0 * kRmTile,
                [&](int j, uint32_t ks, int buf) {
                  const uint32_t id = idesc_bf16_f32(128, 128, false, false);
#pragma unroll
                  for (int b = 0; b < NMB; ++b) {
                    const uint32_t d = tbase + (uint32_t)(buf * NMB + b) * 128u;
                    const uint32_t as = smem_u32(qs + b * 32768);
#pragma unroll
                    for (int k = 0; k < 8; ++k) {
                      const uint32_t ko = (k >> 2) * 16384 + (k & 3) * 32;
                      umma_bf16(d, sdesc_sw128(as + ko, 16, 1024), sdesc_sw128(ks + ko, 16, 1024),
                                id, k > 0 ? 1u : 0u);
                    }
                  }
                  (void)j;
                });
  } else {
    pdl_release();
    const int e = threadIdx.x - 64;
    const int grp = e >> 7, b = grp % NMB, cp = grp / NMB, q = warp & 3;
    const int rho = b * 128 + q * 32 + lane;            // this thread's row
    const int c0 = cp * CW;                             // its first token column
    const int h = rho / J.Rp, r = rho - h * J.Rp;
    const bool row_ok = h < P.G && r < P.R;
    // a warp whose 32 rows are all padding only keeps the pipeline's count
    const bool live = __any_sync(0xffffffffu, row_ok);
    // the slab's question rows (written before the wait: inputs only)
    rm_load_q(P, slab, J.Rp, NMB * 128, 128, qs, e, n_epi);
    fence_proxy_async_smem();
    rm_bar(n_epi);
    if (e == 0) mbar_arrive(smem_u32(&S.q_ready));
    const uint32_t lane_addr = tbase + ((uint32_t)(q * 32) << 16);
    const unsigned long long sc2 = f2pack(kScoreScale, kScoreScale);
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < n_tiles; ++j) {
      const int buf = j % nbuf;
      ok = ok && rm_wait(smem_u32(&S.d_full[buf]), (j / nbuf) & 1, abort);
      tc_fence_after();
      if (ok && live) {
        const uint32_t d = lane_addr + (uint32_t)(buf * NMB + b) * 128u + (uint32_t)c0;
        const int nv = min(kRmTile, n_tok - (t0 + j) * kRmTile) - c0;   // valid columns
        // the part's columns PW at a time (online update per load); pairs (a[c], b[c])
        // of the loaded columns go through the packed fp32x2 path
#pragma unroll
        for (int pc = 0; pc < CW; pc += PW) {
          float v0[32], v1[32];
          if constexpr (PW == 64) tmem_ld32x2(d + pc, d + pc + 32, v0, v1);
          else tmem_ld32(d + pc, v0);
          constexpr int NP = PW / 2;                    // packed pairs
          auto A = [&](int c) -> float { return v0[c]; };
          auto Bv = [&](int c) -> float {
            if constexpr (PW == 64) return v1[c];
            else return v0[16 + c];
          };
          float mt = -INFINITY;
          if (nv >= pc + PW) {
            // (a full load needs no per-column test; the max is taken on the raw dot
            // products and scaled once; packed pairs are adjacent columns of one load,
            // which sit in adjacent registers)
            auto W = [&](int i) -> float {
              if constexpr (PW == 64) return i < 32 ? v0[i] : v1[i - 32];
              else return v0[i];
            };
            float a0 = -INFINITY, a1 = -INFINITY;
#pragma unroll
            for (int c = 0; c < PW; c += 4) {
              a0 = fmax3(a0, W(c), W(c + 1));
              a1 = fmax3(a1, W(c + 2), W(c + 3));
            }
            mt = fmaxf(a0, a1) * kScoreScale;
            if (mt > m) {
              l = (m == -INFINITY) ? 0.f : l * fast_exp2(m - mt);
              m = mt;
            }
            const unsigned long long nm2 = f2pack(-m, -m);
            unsigned long long p0 = 0ull, p1 = 0ull;
#pragma unroll
            for (int c = 0; c < NP; ++c) {
              const unsigned long long x = ffma2(f2pack(W(2 * c), W(2 * c + 1)), sc2, nm2);
              const unsigned long long ex = f2pack(fast_exp2(f2lo(x)), fast_exp2(f2hi(x)));
              if (c & 1) p1 = fadd2(p1, ex);
              else p0 = fadd2(p0, ex);
            }
            l += (f2lo(p0) + f2lo(p1)) + (f2hi(p0) + f2hi(p1));
          } else if (nv > pc) {
            // the ragged last tile: column pc + c of A, pc + NP + c of Bv
#pragma unroll
            for (int c = 0; c < NP; ++c) {
              if (pc + c < nv) mt = fmaxf(mt, A(c));
              if (pc + NP + c < nv) mt = fmaxf(mt, Bv(c));
            }
            mt *= kScoreScale;
            if (mt > m) {
              l = (m == -INFINITY) ? 0.f : l * fast_exp2(m - mt);
              m = mt;
            }
            float acc = 0.f;
#pragma unroll
            for (int c = 0; c < NP; ++c) {
              if (pc + c < nv) acc += fast_exp2(fmaf(A(c), kScoreScale, -m));
              if (pc + NP + c < nv) acc += fast_exp2(fmaf(Bv(c), kScoreScale, -m));
            }
            l += acc;
          }
        }
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&S.epi_done[buf]));
    }
    // the column parts of a row, combined in part order
    if constexpr (CS > 1) {
      if (cp > 0) part_s[(cp - 1) * (NMB * 128) + rho] = make_float2(m, l);
      rm_bar(n_epi);
      if (cp == 0)
        for (int c = 1; c < CS; ++c) {
          const float2 v = part_s[(c - 1) * (NMB * 128) + rho];
          if (v.y > 0.f) ml_combine(m, l, v.x, v.y);
        }
    }
    pdl_wait();   // the previous kernel of the call (its resets) has completed
    if (cp == 0 && ok && !*abort && row_ok)
      J.part[((int64_t)slab * J.GRp + rho) * J.chunks + chunk] = make_float2(m, l);
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) pdl_wait();
  if (threadIdx.x == 0 && S.abort) atomicOr(P.status, kStatusTimeout);
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tbase, cols);
}

// The exponent offset M + log2(L) (and 1 / L) of every row from the chunks' partials,
// combined in chunk order.
__global__ void __launch_bounds__(256) k_rm_combine(const __grid_constant__ Batch B, const RmJob J) {
  pdl_wait();
  pdl_release();
  const Prob& P = B.p[J.prob];
  const int x = blockIdx.x * blockDim.x + threadIdx.x;
  const int n_slabs = P.P * P.Hkv;
  if (x >= n_slabs * J.GRp) return;
  const int rho = x % J.GRp;
  const int h = rho / J.Rp, r = rho - h * J.Rp;
  if (h >= P.G || r >= P.R) return;
  float m = -INFINITY, l = 0.f;
  for (int c = 0; c < J.chunks; ++c) {
    const float2 v = J.part[(int64_t)x * J.chunks + c];
    if (v.y > 0.f) ml_combine(m, l, v.x, v.y);
  }
  // 2^(s - M) / L = 2^(s - (M + log2 L)): the weight needs one exponent offset per row
  J.stat[x] = make_float2(l > 0.f ? m + __log2f(l) : INFINITY, l > 0.f ? 1.0f / l : 0.f);
}

// ---------------------------------------------------------------------------
// Pass 2: alpha of every history token of the chunk for the slab's G lists.
// Warps: 0 TMA, 1 MMA (+ TMEM), 2-17 epilogue (four groups of four, heads split).
// Each row's exponent offset enters the accumulator through one more MMA K step: A' (the
// tokens, MN-major) is 1 in K columns 0-2, B' (the rows, MN-major) holds minus the row's
// offset / scale split into three bf16 parts, so D = s - offset / scale and the epilogue
// needs no per-row constants (no shared-memory loads next to the tensor cores' reads).
// ---------------------------------------------------------------------------
constexpr int kRmEpi2 = 512;
constexpr int kRmGroups2 = kRmEpi2 / 128;
constexpr int kRmXaBytes = 2 * 2048;                   // A': 2 blocks of 64 tokens x 16 K

// Bytes of B' for one operand tile of `ne` rows: blocks of 64 rows x 16 K (2 KB each).
__host__ __device__ constexpr int rm_xb_bytes(int ne) { return (ne + 63) / 64 * 2048; }

// Element (k, n) of a 128-byte swizzled MN-major operand whose 64-element blocks are
// 2048 bytes apart (16 K rows of 128 bytes each).
__device__ __forceinline__ int rm_mn_offset(int k, int n) {
  return (n >> 6) * 2048 + (k >> 3) * 1024 + (k & 7) * 128 + ((((n >> 3) & 7) ^ (k & 7)) << 4) +
         (n & 7) * 2;
}

__global__ void __launch_bounds__(rm_bound(64 + kRmEpi2), 1)
    k_rm_alpha(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ Batch B,
               const RmJob J) {
  extern __shared__ unsigned char sm_raw[];
  __shared__ RmBars S;
  unsigned char* sm = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int GRp = J.GRp;
  // question rows as the B operand: one tile of GRp rows, or two of NE rows each
  const int two = GRp > 256;
  const int NE = two ? ((GRp / 2 + 15) & ~15) : GRp;
  unsigned char* qs = sm;
  const int q_bytes = (two ? 2 : 1) * NE * 256;
  unsigned char* xa = qs + ((q_bytes + 1023) & ~1023);   // A' (kRmXaBytes)
  unsigned char* xb = xa + kRmXaBytes;                     // B' of each operand tile
  const int xb_tile = rm_xb_bytes(NE);
  unsigned char* ring = xb + (((two ? 2 : 1) * xb_tile + 1023) & ~1023);
  const int nbuf = J.nbuf, stages = J.stages;
  const uint32_t cols = nbuf * (two ? 2 * NE : NE) <= 256 ? 256u : 512u;
  rm_init(S, stages, nbuf, kRmEpi2, cols);
  const uint32_t tbase = S.taddr;
  const Prob& P = B.p[J.prob];
  const int slab = blockIdx.y, chunk = blockIdx.x;
  int t0, t1;
  rm_chunk(P, J.chunks, chunk, t0, t1);
  const int n_tiles = t1 - t0;
  const int n_tok = P.Uh * P.Tu;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t buf_cols = two ? 2 * NE : NE;
  volatile int* abort = &S.abort;
  if (warp < 2) {
    rm_pipeline(&kmap, S, ring, stages, nbuf, kRmEpi2, n_tiles,
                (int64_t)slab * P.ncap + (int64_t)t0 * kRmTile,
                [&](int j, uint32_t ks, int buf) {
                  const uint32_t id = idesc_bf16_f32(128, NE, false, false);
                  const uint32_t idx = idesc_bf16_f32(128, NE, true, true);
                  for (int t = 0; t < 1 + two; ++t) {
                    const uint32_t d = tbase + (uint32_t)buf * buf_cols + (uint32_t)(t * NE);
                    const uint32_t bs = smem_u32(qs + t * NE * 256);
#pragma unroll
                    for (int k = 0; k < 8; ++k) {
                      const uint32_t ka = (k >> 2) * 16384 + (k & 3) * 32;
                      const uint32_t kb = (k >> 2) * (NE * 128) + (k & 3) * 32;
                      umma_bf16(d, sdesc_sw128(ks + ka, 16, 1024), sdesc_sw128(bs + kb, 16, 1024),
                                id, k > 0 ? 1u : 0u);
                    }
                    // the offsets: D += A' B'^T
                    umma_bf16(d, sdesc_sw128(smem_u32(xa), 2048, 1024),
                              sdesc_sw128(smem_u32(xb + t * xb_tile), 2048, 1024), idx, 1u);
                  }
                  (void)j;
                });
  } else {
    const int e = threadIdx.x - 64;
    const int grp = e >> 7, q = warp & 3;
    const int tl = q * 32 + lane;                        // token lane
    rm_load_q(P, slab, J.Rp, (two ? 2 : 1) * NE, NE, qs, e, kRmEpi2);
    // A': ones in K columns 0-2 for all 128 tokens, zeros elsewhere; B' zeroed
    for (int x = e; x < 128 * 16; x += kRmEpi2) {
      const int k = x >> 7, m = x & 127;
      *reinterpret_cast<__nv_bfloat16*>(xa + rm_mn_offset(k, m)) =
          __float2bfloat16_rn(k < 3 ? 1.f : 0.f);
    }
    for (int x = e; x < (two ? 2 : 1) * xb_tile / 16; x += kRmEpi2)
      reinterpret_cast<uint4*>(xb)[x] = make_uint4(0u, 0u, 0u, 0u);
    rm_bar(kRmEpi2);
    pdl_wait();                                          // the rows' statistics (pass 1)
    for (int x = e; x < (two ? 2 : 1) * NE; x += kRmEpi2) {
      const int t = x / NE, n = x - t * NE;              // operand tile, its row
      const int hr = x / J.Rp, rr = x - hr * J.Rp;
      // offset / scale in three bf16 parts (24 significant bits); rows past R (or past
      // the G heads) get one that takes their terms to 0
      float v = 1e30f;
      if (x < GRp && hr < P.G && rr < P.R) {
        const float o = J.stat[(int64_t)slab * GRp + x].x;
        if (o < INFINITY) v = o / kScoreScale;
      }
      const __nv_bfloat16 b1 = __float2bfloat16_rn(v);
      const float r1 = v - __bfloat162float(b1);
      const __nv_bfloat16 b2 = __float2bfloat16_rn(r1);
      const __nv_bfloat16 b3 = __float2bfloat16_rn(r1 - __bfloat162float(b2));
      unsigned char* tb = xb + t * xb_tile;
      *reinterpret_cast<__nv_bfloat16*>(tb + rm_mn_offset(0, n)) = __hneg(b1);
      *reinterpret_cast<__nv_bfloat16*>(tb + rm_mn_offset(1, n)) = __hneg(b2);
      *reinterpret_cast<__nv_bfloat16*>(tb + rm_mn_offset(2, n)) = __hneg(b3);
    }
    fence_proxy_async_smem();
    rm_bar(kRmEpi2);
    if (e == 0) mbar_arrive(smem_u32(&S.q_ready));
    pdl_release();
    const int G = P.G, Rp = J.Rp;
    const int h_begin = G * grp / kRmGroups2, h_end = G * (grp + 1) / kRmGroups2;
    const int i = slab / P.Hkv, g = slab - i * P.Hkv;
    const float invR = 1.0f / (float)P.R;
    const uint32_t lane_addr = tbase + ((uint32_t)(q * 32) << 16);
    bool ok = true;
    for (int j = 0; j < n_tiles; ++j) {
      const int buf = j % nbuf;
      ok = ok && rm_wait(smem_u32(&S.d_full[buf]), (j / nbuf) & 1, abort);
      tc_fence_after();
      const int tok = (t0 + j) * kRmTile + tl;
      if (ok) {
        for (int h = h_begin; h < h_end; ++h) {
          const uint32_t col = lane_addr + (uint32_t)buf * buf_cols + (uint32_t)(h * Rp);
          float a = 0.f, a2 = 0.f;
          // a head's rows in one load and one wait where they fit 32 or 64 columns (the
          // accumulator already holds s - offset / scale: one packed multiply per pair)
          const unsigned long long sc2 = f2pack(kScoreScale, kScoreScale);
          auto add = [&](const float (&v)[32], int r0) {
            unsigned long long p0 = 0ull, p1 = 0ull;
#pragma unroll
            for (int t = 0; t < 32; t += 4) {
              const unsigned long long x0 = fmul2(f2pack(v[t], v[t + 1]), sc2);
              const unsigned long long x1 = fmul2(f2pack(v[t + 2], v[t + 3]), sc2);
              p0 = fadd2(p0, f2pack(fast_exp2(f2lo(x0)), fast_exp2(f2hi(x0))));
              p1 = fadd2(p1, f2pack(fast_exp2(f2lo(x1)), fast_exp2(f2hi(x1))));
            }
            a += f2lo(p0) + f2lo(p1);
            a2 += f2hi(p0) + f2hi(p1);
            (void)r0;
          };
          if (Rp == 32) {
            float v[32];
            tmem_ld32(col, v);
            add(v, 0);
          } else if (Rp == 64) {
            float v0[32], v1[32];
            tmem_ld32x2(col, col + 32, v0, v1);
            add(v0, 0);
            add(v1, 32);
          } else {
            for (int r0 = 0; r0 < Rp; r0 += 16) {
              float v[16];
              tmem_ld16(col + (uint32_t)r0, v);
#pragma unroll
              for (int t = 0; t < 16; ++t) a += fast_exp2(v[t] * kScoreScale);
            }
          }
          if (tok < n_tok)
            P.cand_s[(int64_t)(i * P.Hq + g * G + h) * P.cand_cap + tok] = (a + a2) * invR;
        }
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&S.epi_done[buf]));
    }
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) pdl_wait();
  if (threadIdx.x == 0 && S.abort) atomicOr(P.status, kStatusTimeout);
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tbase, cols);
}

// Host: both passes for problem `pi` of the batch (its own key tensor map).
bool rowmean_supported(int R, int G) {
  const int Rp = (R + 15) & ~15;
  return R >= 1 && Rp <= 64 && G * Rp <= 512;
}

size_t rowmean_workspace_bytes(int n_slabs, int R, int G, int max_chunks) {
  const int GRp = G * ((R + 15) & ~15);
  return (size_t)n_slabs * GRp * (max_chunks + 1) * sizeof(float2);
}

// CTAs per slab: as many as fit in one wave (one CTA per SM), at least one.
int rowmean_chunks(int n_slabs, int hist_tokens, int sm_count) {
  const int T = (hist_tokens + kRmTile - 1) / kRmTile;
  int c = sm_count / n_slabs;
  c = c < 1 ? 1 : c;
  return T < c ? (T < 1 ? 1 : T) : c;
}

cudaError_t launch_rowmean(const Batch& B, int pi, float2* scratch, int chunks, cudaStream_t s) {
  const Prob& P = B.p[pi];
  const int n_slabs = P.P * P.Hkv;
  const int Rp = (P.R + 15) & ~15, GRp = P.G * Rp;
  if (P.Uh <= 0) return cudaSuccess;
  RmJob J;
  J.prob = pi;
  J.Rp = Rp;
  J.GRp = GRp;
  J.chunks = chunks;
  J.part = scratch;
  J.stat = scratch + (size_t)n_slabs * GRp * chunks;
  // keys of every slab: rows [slab * ncap + token], 128 dims
  const uint64_t dims[2] = {(uint64_t)kHeadDim, (uint64_t)n_slabs * (uint64_t)P.ncap};
  const uint64_t strides[1] = {(uint64_t)kHeadDim * 2};
  const uint32_t box[2] = {64, kRmTile};
  CUtensorMap map;
  cudaError_t e = encode_bf16_map(&map, P.keys, 2, dims, strides, box);
  if (e != cudaSuccess) return e;
  const int nmb = (GRp + 127) / 128;
  {
    J.nbuf = nmb <= 2 ? 2 : 1;
    J.stages = nmb <= 2 ? 4 : 2;
    const size_t smem = 1024 + (size_t)nmb * 32768 + (size_t)J.stages * kRmStageBytes;
    // column parts: up to 16 epilogue warps per CTA
    const int cs = nmb == 1 ? 4 : nmb == 2 ? 2 : 1;
    auto kern = nmb == 1 ? k_rm_stats<1, 4> : nmb == 2 ? k_rm_stats<2, 2>
              : nmb == 3 ? k_rm_stats<3, 1> : k_rm_stats<4, 1>;
    e = ensure_smem((const void*)kern, (int)smem);
    if (e != cudaSuccess) return e;
    e = launch_pdl(kern, dim3(chunks, n_slabs), dim3(64 + 128 * nmb * cs), smem, s, map, B, J);
    if (e != cudaSuccess) return e;
  }
  e = launch_pdl(k_rm_combine, dim3((n_slabs * GRp + 255) / 256), dim3(256), 0, s, B, J);
  if (e != cudaSuccess) return e;
  {
    const bool two = GRp > 256;
    const int NE = two ? ((GRp / 2 + 15) & ~15) : GRp;
    const int qb = ((two ? 2 : 1) * NE * 256 + 1023) & ~1023;
    const int xb = ((two ? 2 : 1) * rm_xb_bytes(NE) + 1023) & ~1023;
    const int pre = 1024 + qb + kRmXaBytes + xb;        // before the key stages
    J.nbuf = (two ? 2 * NE : NE) <= 256 ? 2 : 1;
    // key stages: what the 227 KB of shared memory leave (less the static part), at most 4
    const int st = (232448 - 256 - pre) / kRmStageBytes;
    J.stages = st < 4 ? st : 4;
    if (J.stages < 2) return cudaErrorInvalidConfiguration;
    const size_t smem = (size_t)pre + (size_t)J.stages * kRmStageBytes;
    e = ensure_smem((const void*)k_rm_alpha, (int)smem);
    if (e != cudaSuccess) return e;
    e = launch_pdl(k_rm_alpha, dim3(chunks, n_slabs), dim3(64 + kRmEpi2), smem, s, map, B, J);
  }
  return e;
}

}  // namespace ss
