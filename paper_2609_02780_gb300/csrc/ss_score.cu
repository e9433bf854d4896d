// Query preparation and the key-scoring kernel of query-time evidence retrieval.
//
// Sec. 4.2: for each shallow layer i and query head h the question's query state
// attends to every candidate history token; Eq. 11 keeps the top tokens of each list.
// This file computes, in one pass over the stored keys:
//   * s = q_eff[i][h] . K[i][h / G][p] * log2(e) / sqrt(d) for every history token p
//     (bf16 products, fp32 accumulation on the tensor cores);
//   * for every (list, unit) the pair (max s, sum 2^(s - max)) over the unit's tokens,
//     from which the softmax statistics of each list and the attention mass of each
//     unit follow exactly;
//   * a superset of every list's top-k tokens: each token whose score reaches a
//     running lower bound of the list's k-th best score is appended to the list's
//     candidate array.
#include "ss_internal.cuh"

namespace ss {

// ---------------------------------------------------------------------------
// Query representation and per-call resets.
// q_eff[i][h] is the last question row ("final prompt token", Sec. 4.2 / Table 4) or
// the rows' mean (fp32 sum in row order, divided by R, rounded to bf16 nearest-even).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kHeadDim) k_prep(const __grid_constant__ Batch B) {
  const int pi = blockIdx.y;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  const int n_lists = P.P * P.Hq;
  const int L = blockIdx.x;
  if (L >= n_lists) return;
  const int i = L / P.Hq, h = L % P.Hq;
  const int d = threadIdx.x;
  const int64_t row_stride = (int64_t)P.Hq * kHeadDim;
  const __nv_bfloat16* q0 = P.q + (int64_t)i * P.R * row_stride + (int64_t)h * kHeadDim + d;
  float v;
  if (B.q_agg == 0) {
    v = __bfloat162float(q0[(int64_t)(P.R - 1) * row_stride]);
  } else {
    float acc = 0.f;
    for (int r = 0; r < P.R; ++r) acc = __fadd_rn(acc, __bfloat162float(q0[(int64_t)r * row_stride]));
    v = __fdiv_rn(acc, (float)P.R);
  }
  P.qeff[(int64_t)L * kHeadDim + d] = __float2bfloat16_rn(v);
  if (d == 0) {
    P.cand_cnt[L] = 0;
    P.gthr[L] = float_to_ordered(-INFINITY);
  }
  for (int u = L * kHeadDim + d; u < P.ucap; u += n_lists * kHeadDim) P.votes[u] = 0;
  if (L == 0 && d < 4) P.counts[d] = 0;
  if (L == 0 && d == 0) *P.status = 0u;
}

cudaError_t launch_prep(const Batch& B, cudaStream_t s) {
  int max_lists = 0;
  for (int j = 0; j < B.n; ++j) max_lists = max(max_lists, B.p[j].P * B.p[j].Hq);
  dim3 grid(max_lists, B.n);
  k_prep<<<grid, kHeadDim, 0, s>>>(B);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Scoring kernel.
//
// Grid: one CTA per (problem, slab = (layer i, key head g), chunk of history units).
// Block: kScoreWarps compute warps + 1 threshold warp.
//
// Compute warps take the chunk's units round-robin and walk each unit in tiles of 16
// tokens. A tile's scores for the G query heads of the group come from 8
// m16n8k16 bf16 MMAs: A = 16 keys x 16 dims, B = 16 dims x 8 heads (G used).
// The contraction order over d is free, so lane (row g, column group t) loads the
// 64 contiguous bytes {32 v + 8 t .. 32 v + 8 t + 7 : v = 0..3} of rows g and g + 8 with
// 16-byte loads straight from HBM into the A-fragment registers, and the query
// fragments use the same permutation. The accumulator gives lane (g, t) the scores
// of keys g and g + 8 for heads 2t and 2t + 1.
//
// Candidate filter: a token is appended to its list when s >= thr[h], where thr[h] is
// always a lower bound of the list's k-th best score, so every top-k token is
// appended. The threshold warp maintains thr from a per-head histogram of the
// appended scores (bins of 1/8 log2 unit anchored at the first units' maximum: the
// lower edge of the bin below the one where the count from the top reaches k is a
// valid bound whatever the rounding of the bin computation) and
// shares it with the other CTAs of the list through a global atomicMax.
// ---------------------------------------------------------------------------
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

struct ScoreShared {
  int hist[kMaxGroup][kHistBins];
  float thr[kMaxGroup];
  float base[kMaxGroup];
  uint32_t max0[kMaxGroup];
  int first_done;
  int all_done;
  int base_valid;
};

// One column (query head) of a tile: online (max, sum 2^(s - max)) over valid rows.
__device__ __forceinline__ void stats_update(float& m, float& l, float x0, bool v0,
                                             float x1, bool v1) {
  if (v0 | v1) {
    const float mt = fmaxf(v0 ? x0 : -INFINITY, v1 ? x1 : -INFINITY);
    if (mt > m) {
      l *= fast_exp2(m - mt);
      m = mt;
    }
    l += (v0 ? fast_exp2(x0 - m) : 0.f) + (v1 ? fast_exp2(x1 - m) : 0.f);
  }
}

__device__ __forceinline__ void hist_add(ScoreShared& S, int c, float s, float base,
                                         bool base_ok) {
  if (!base_ok) return;
  const int bin = __float2int_rd((s - base) * kBinsPerUnit);
  if (bin >= 0) atomicAdd(&S.hist[c][min(bin, kHistBins - 1)], 1);
}

__device__ void threshold_warp(ScoreShared& S, const Prob& P, int list0, int k) {
  const int lane = threadIdx.x & 31;
  const int G = P.G;
  bool base_ok = false;
  volatile int* vfirst = &S.first_done;
  volatile int* vdone = &S.all_done;
  volatile float* vthr = S.thr;
  for (int iter = 0; iter < (1 << 21); ++iter) {
    const int done = *vdone;
    if (!base_ok) {
      if (*vfirst >= kScoreWarps) {
        __threadfence_block();
        if (lane < G) {
          const float mx = ordered_to_float(((volatile uint32_t*)S.max0)[lane]);
          S.base[lane] = (mx == -INFINITY) ? 0.f : mx - kHistBelowMax;
        }
        __syncwarp();
        __threadfence_block();
        if (lane == 0) *(volatile int*)&S.base_valid = 1;
        base_ok = true;
      }
    } else {
      for (int c = 0; c < G; ++c) {
        const volatile int* hc = S.hist[c];
        int cnts[16];
        int sum = 0;
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          cnts[q] = hc[kHistBins - 1 - (16 * lane + q)];
          sum += cnts[q];
        }
        int cum = sum;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
          const int y = __shfl_up_sync(0xffffffffu, cum, off);
          if (lane >= off) cum += y;
        }
        const unsigned hit = __ballot_sync(0xffffffffu, cum >= k);
        float t_new = -INFINITY;
        if (hit) {
          const int f = __ffs(hit) - 1;
          if (lane == f) {
            int run = cum - sum;
            int q = 0;
            for (; q < 15; ++q) {
              run += cnts[q];
              if (run >= k) break;
            }
            // One bin of margin: a score counted in bin b satisfies s >= base + b / 8
            // only up to the rounding of (s - base), far below a bin width.
            const int bin = kHistBins - 1 - (16 * lane + q);
            t_new = S.base[c] + (float)(bin - 1) / kBinsPerUnit;
          }
          t_new = __shfl_sync(0xffffffffu, t_new, f);
        }
        if (lane == 0) {
          float t;
          if (hit) {
            const uint32_t old = atomicMax(P.gthr + list0 + c, float_to_ordered(t_new));
            t = fmaxf(t_new, ordered_to_float(old));
          } else {
            t = ordered_to_float(*(volatile uint32_t*)(P.gthr + list0 + c));
          }
          if (t > vthr[c]) vthr[c] = t;
        }
        __syncwarp();
      }
    }
    if (done >= kScoreWarps) break;
    __nanosleep(400);
  }
}

__global__ void __launch_bounds__(kScoreThreads, kScoreCtasPerSm)
    k_score(const __grid_constant__ Batch B) {
  __shared__ ScoreShared S;
  const int b = blockIdx.x;
  const int pi = problem_of_block(B, b);
  const Prob& P = B.p[pi];
  const int local = b - P.cta_begin;
  const int n_slabs = P.P * P.Hkv;
  if (P.chunks <= 0) return;
  const int slab = local / P.chunks, chunk = local - slab * P.chunks;
  if (slab >= n_slabs) return;
  const int u0 = (int)(((int64_t)P.Uh * chunk) / P.chunks);
  const int u1 = (int)(((int64_t)P.Uh * (chunk + 1)) / P.chunks);

  for (int x = threadIdx.x; x < kMaxGroup * kHistBins; x += blockDim.x)
    (&S.hist[0][0])[x] = 0;
  if (threadIdx.x < kMaxGroup) {
    S.thr[threadIdx.x] = -INFINITY;
    S.base[threadIdx.x] = 0.f;
    S.max0[threadIdx.x] = float_to_ordered(-INFINITY);
  }
  if (threadIdx.x == 0) {
    S.first_done = 0;
    S.all_done = 0;
    S.base_valid = 0;
  }
  __syncthreads();

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = slab / P.Hkv, kvh = slab - i * P.Hkv;
  const int G = P.G;
  const int list0 = i * P.Hq + kvh * G;
  const int k = B.k;
  if (warp == kScoreWarps) {
    threshold_warp(S, P, list0, k);
    return;
  }

  const int g = lane >> 2, t4 = lane & 3;
  // Query fragments (B operand), permuted like the key loads.
  uint32_t qf[8][2];
  {
    const uint32_t* qw = reinterpret_cast<const uint32_t*>(P.qeff);
    const int64_t qoff = (int64_t)(list0 + g) * (kHeadDim / 2);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int e = 8 * (4 * (j >> 1) + t4) + 4 * (j & 1);
      if (g < G) {
        qf[j][0] = qw[qoff + (e >> 1)];
        qf[j][1] = qw[qoff + (e >> 1) + 1];
      } else {
        qf[j][0] = 0u;
        qf[j][1] = 0u;
      }
    }
  }
  const int c0 = 2 * t4, c1 = 2 * t4 + 1;
  const bool hv0 = c0 < G, hv1 = c1 < G;
  const int L0 = list0 + c0, L1 = list0 + c1;
  const int Tu = P.Tu;
  const int tpu = (Tu + 15) >> 4;
  const int n_chunk_units = u1 - u0;
  const int n_my = n_chunk_units > warp
                       ? (n_chunk_units - warp + kScoreWarps - 1) / kScoreWarps
                       : 0;
  const int ntiles = n_my * tpu;
  const __nv_bfloat16* slab_keys = P.keys + (int64_t)slab * P.ncap * kHeadDim;
  float* cs0 = P.cand_s + (int64_t)(hv0 ? L0 : list0) * P.cand_cap;
  int32_t* ci0 = P.cand_id + (int64_t)(hv0 ? L0 : list0) * P.cand_cap;
  float* cs1 = P.cand_s + (int64_t)(hv1 ? L1 : list0) * P.cand_cap;
  int32_t* ci1 = P.cand_id + (int64_t)(hv1 ? L1 : list0) * P.cand_cap;
  float2* us0 = P.ustats + (int64_t)(hv0 ? L0 : list0) * P.ucap;
  float2* us1 = P.ustats + (int64_t)(hv1 ? L1 : list0) * P.ucap;
  const unsigned gmask = 0x11111111u << t4;
  const unsigned lt_mask = (1u << lane) - 1u;

  float m0 = -INFINITY, l0 = 0.f, m1 = -INFINITY, l1 = 0.f;
  float thr0 = INFINITY, thr1 = INFINITY, bs0 = 0.f, bs1 = 0.f;
  bool base_ok = false, first_unit = true;

  auto tile_pos = [&](int t, int& u, int& j) {
    const int m = t / tpu;
    j = t - m * tpu;
    u = u0 + warp + m * kScoreWarps;
  };
  auto load_tile = [&](uint4 (&buf)[8], int t) {
    int u, j;
    tile_pos(t, u, j);
    const int r0 = 16 * j + g;
    const __nv_bfloat16* p0 = slab_keys + ((int64_t)u * Tu + r0) * kHeadDim + 8 * t4;
    const bool ok0 = r0 < Tu, ok1 = r0 + 8 < Tu;
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      buf[v] = ok0 ? ld_stream(p0 + 32 * v) : make_uint4(0u, 0u, 0u, 0u);
      buf[4 + v] = ok1 ? ld_stream(p0 + 8 * kHeadDim + 32 * v) : make_uint4(0u, 0u, 0u, 0u);
    }
  };
  auto process = [&](const uint4 (&buf)[8], int t) {
    int u, j;
    tile_pos(t, u, j);
    if (j == 0) {
      const volatile float* vthr = S.thr;
      thr0 = hv0 ? vthr[c0] : INFINITY;
      thr1 = hv1 ? vthr[c1] : INFINITY;
      base_ok = *(volatile int*)&S.base_valid != 0;
      if (base_ok) {
        const volatile float* vbase = S.base;
        bs0 = vbase[c0];
        bs1 = vbase[c1];
      }
      m0 = m1 = -INFINITY;
      l0 = l1 = 0.f;
    }
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
      const int v = jj >> 1;
      const uint32_t a0 = (jj & 1) ? buf[v].z : buf[v].x;
      const uint32_t a1 = (jj & 1) ? buf[4 + v].z : buf[4 + v].x;
      const uint32_t a2 = (jj & 1) ? buf[v].w : buf[v].y;
      const uint32_t a3 = (jj & 1) ? buf[4 + v].w : buf[4 + v].y;
      mma_16816(acc, a0, a1, a2, a3, qf[jj][0], qf[jj][1]);
    }
    const int r0 = 16 * j + g;
    const bool v0 = r0 < Tu, v1 = r0 + 8 < Tu;
    const float s00 = acc[0] * kScoreScale, s01 = acc[1] * kScoreScale;
    const float s10 = acc[2] * kScoreScale, s11 = acc[3] * kScoreScale;
    stats_update(m0, l0, s00, v0, s10, v1);
    stats_update(m1, l1, s01, v0, s11, v1);

    const bool p00 = hv0 && v0 && s00 >= thr0, p10 = hv0 && v1 && s10 >= thr0;
    const bool p01 = hv1 && v0 && s01 >= thr1, p11 = hv1 && v1 && s11 >= thr1;
    if (__any_sync(0xffffffffu, p00 | p01 | p10 | p11)) {
      const int tok0 = u * Tu + r0, tok1 = tok0 + 8;
      const unsigned b00 = __ballot_sync(0xffffffffu, p00) & gmask;
      const unsigned b10 = __ballot_sync(0xffffffffu, p10) & gmask;
      const unsigned b01 = __ballot_sync(0xffffffffu, p01) & gmask;
      const unsigned b11 = __ballot_sync(0xffffffffu, p11) & gmask;
      {
        const int n = __popc(b00) + __popc(b10);
        int base = 0;
        if (g == 0 && n > 0) base = atomicAdd(P.cand_cnt + L0, n);
        base = __shfl_sync(0xffffffffu, base, t4);
        if (p00) {
          const int pos = base + __popc(b00 & lt_mask);
          cs0[pos] = s00;
          ci0[pos] = tok0;
          hist_add(S, c0, s00, bs0, base_ok);
        }
        if (p10) {
          const int pos = base + __popc(b00) + __popc(b10 & lt_mask);
          cs0[pos] = s10;
          ci0[pos] = tok1;
          hist_add(S, c0, s10, bs0, base_ok);
        }
      }
      {
        const int n = __popc(b01) + __popc(b11);
        int base = 0;
        if (g == 0 && n > 0) base = atomicAdd(P.cand_cnt + L1, n);
        base = __shfl_sync(0xffffffffu, base, t4);
        if (p01) {
          const int pos = base + __popc(b01 & lt_mask);
          cs1[pos] = s01;
          ci1[pos] = tok0;
          hist_add(S, c1, s01, bs1, base_ok);
        }
        if (p11) {
          const int pos = base + __popc(b01) + __popc(b11 & lt_mask);
          cs1[pos] = s11;
          ci1[pos] = tok1;
          hist_add(S, c1, s11, bs1, base_ok);
        }
      }
    }
    if (j == tpu - 1) {
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        const float mo0 = __shfl_xor_sync(0xffffffffu, m0, off);
        const float lo0 = __shfl_xor_sync(0xffffffffu, l0, off);
        const float mo1 = __shfl_xor_sync(0xffffffffu, m1, off);
        const float lo1 = __shfl_xor_sync(0xffffffffu, l1, off);
        ml_combine(m0, l0, mo0, lo0);
        ml_combine(m1, l1, mo1, lo1);
      }
      if (g == 0) {
        if (hv0) us0[u] = make_float2(m0, l0);
        if (hv1) us1[u] = make_float2(m1, l1);
        if (first_unit) {
          if (hv0) atomicMax(&S.max0[c0], float_to_ordered(m0));
          if (hv1) atomicMax(&S.max0[c1], float_to_ordered(m1));
        }
      }
      if (first_unit) {
        __syncwarp();
        __threadfence_block();
        if (lane == 0) atomicAdd(&S.first_done, 1);
        first_unit = false;
      }
    }
  };

  uint4 bufA[8], bufB[8];
  if (ntiles > 0) load_tile(bufA, 0);
  if (ntiles > 1) load_tile(bufB, 1);
  for (int t = 0; t < ntiles; t += 2) {
    process(bufA, t);
    if (t + 2 < ntiles) load_tile(bufA, t + 2);
    if (t + 1 < ntiles) {
      process(bufB, t + 1);
      if (t + 3 < ntiles) load_tile(bufB, t + 3);
    }
  }
  if (lane == 0) {
    if (first_unit) atomicAdd(&S.first_done, 1);
    atomicAdd(&S.all_done, 1);
  }
}

int score_chunks_per_slab(int n_slabs_total, int hist_units, int sm_count) {
  // Pick the chunk length (in units) that minimises waves x chunk length over the
  // resident CTA slots; ties go to fewer CTAs.
  if (hist_units <= 0 || n_slabs_total <= 0) return 0;
  const int64_t slots = (int64_t)sm_count * kScoreCtasPerSm;
  int best_c = 1;
  int64_t best_cost = INT64_MAX;
  for (int c = 1; c <= hist_units && c <= 4096; ++c) {
    const int64_t ctas = (int64_t)n_slabs_total * c;
    const int64_t waves = (ctas + slots - 1) / slots;
    const int64_t len = (hist_units + c - 1) / c;
    const int64_t cost = waves * len;
    if (cost < best_cost) {
      best_cost = cost;
      best_c = c;
    }
  }
  return best_c;
}

cudaError_t launch_score(const Batch& B, cudaStream_t s) {
  if (B.score_ctas <= 0) return cudaSuccess;
  k_score<<<B.score_ctas, kScoreThreads, 0, s>>>(B);
  return cudaGetLastError();
}

}  // namespace ss
