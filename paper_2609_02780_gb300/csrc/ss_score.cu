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
#include "ss_device.cuh"

namespace ss {

// ---------------------------------------------------------------------------
// Query representation and per-call resets.
// q_eff[i][h] is the last question row ("final prompt token", Sec. 4.2 / Table 4) or
// the rows' mean (fp32 sum in row order, divided by R, rounded to bf16 nearest-even).
// ---------------------------------------------------------------------------
// k_sample: grid (slab, problem, sample z), 256 threads. Computes q_eff of the slab's G
// query heads (block z = 0 stores it and resets the per-call state), then scores the G
// heads against every token of the history unit z * Uh / Z on the tensor cores (keys
// staged in shared memory, the scoring kernel's fragment layout). The largest sampled
// score of each list anchors its threshold ladder.
constexpr int kSampleRows = 128;  // key rows staged per pass of k_sample (8 MMA tiles)

int sample_units(int k, int tokens_per_unit, int hist_units) {
  (void)k;
  (void)tokens_per_unit;
  return hist_units < kSampleUnits ? hist_units : kSampleUnits;
}

__global__ void __launch_bounds__(256) k_sample(const __grid_constant__ Batch B) {
  __shared__ __align__(16) __nv_bfloat16 qsb[kMaxGroup][kHeadDim];
  __shared__ float wmax[8][kMaxGroup];
  __shared__ __align__(16) unsigned char kt[kSampleRows * kHeadDim * 2];
  // Before the wait for the previous kernel: only reads of the inputs (query rows and
  // the first pass of the sampled unit's keys), which no kernel of the chain writes.
  const int pi = blockIdx.y;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  const int slab = blockIdx.x, z = blockIdx.z;
  const int n_slabs = P.P * P.Hkv;
  if (slab >= n_slabs) return;
  const int i = slab / P.Hkv, gk = slab - i * P.Hkv, G = P.G;
  const int list0 = i * P.Hq + gk * G;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t row_stride = (int64_t)P.Hq * kHeadDim;
  const bool sampling = z < P.n_sample;
  const int64_t u = sampling ? ((int64_t)z * P.Uh) / P.n_sample : 0;
  const __nv_bfloat16* sk = P.keys + ((int64_t)slab * P.ncap + u * P.Tu) * kHeadDim;
  // a pass's rows as 16-byte vectors, all of a thread's loads in flight at once; the
  // first two passes are loaded before the wait
  constexpr int kPerThread = kSampleRows * (kHeadDim / 8) / 256;
  uint4 vbuf[kPerThread], vbuf2[kPerThread];
  auto load_pass = [&](uint4 (&vb)[kPerThread], int rb, int nr) {
    const uint4* src = reinterpret_cast<const uint4*>(sk + (int64_t)rb * kHeadDim);
#pragma unroll
    for (int q = 0; q < kPerThread; ++q) {
      const int x = q * 256 + tid;
      if (x < nr * (kHeadDim / 8)) vb[q] = src[x];
    }
  };
  if (sampling) {
    load_pass(vbuf, 0, min(kSampleRows, P.Tu));
    if (P.Tu > kSampleRows) load_pass(vbuf2, kSampleRows, min(kSampleRows, P.Tu - kSampleRows));
  }
  for (int x = tid; x < kMaxGroup * kHeadDim; x += blockDim.x) {
    const int hh = x / kHeadDim, d = x - hh * kHeadDim;
    __nv_bfloat16 qe = __float2bfloat16_rn(0.f);
    if (hh < G) {
      const __nv_bfloat16* q0 = P.q + (int64_t)i * P.R * row_stride + (int64_t)(gk * G + hh) * kHeadDim + d;
      float v;
      if (B.q_agg == 0) {
        v = __bfloat162float(q0[(int64_t)(P.R - 1) * row_stride]);
      } else {
        float acc = 0.f;
        for (int r = 0; r < P.R; ++r) acc = __fadd_rn(acc, __bfloat162float(q0[(int64_t)r * row_stride]));
        v = __fdiv_rn(acc, (float)P.R);
      }
      qe = __float2bfloat16_rn(v);
    }
    qsb[hh][d] = qe;
  }
  pdl_wait();     // the previous call's use of the workspace
  pdl_release();
  if (z == 0) {
    for (int x = tid; x < G * kHeadDim; x += blockDim.x)  // each thread's own qsb entries
      P.qeff[(int64_t)list0 * kHeadDim + x] = qsb[x / kHeadDim][x % kHeadDim];
    if (tid < G) {
      P.cand_cnt[list0 + tid] = 0;
      P.gthr[list0 + tid] = float_to_ordered(-INFINITY);
    }
    for (int x = tid; x < G * kLadderLevels; x += blockDim.x)
      P.ladder[(int64_t)list0 * kLadderLevels + x] = 0;
    if (tid == 0) P.next_unit[slab * kUnitCounterStride] = P.chunks * kScoreWarps;  // past the fixed first units
    for (int v = slab * blockDim.x + tid; v < P.ucap; v += n_slabs * blockDim.x) P.votes[v] = 0;
    if (slab == 0 && tid < 4) P.counts[tid] = 0;
    // a compression whose wait gave up is reported by every later retrieval
    if (slab == 0 && tid == 0) *P.status = P.index_status ? (*P.index_status & kStatusTimeout) : 0u;
  }
  __syncthreads();
  if (!sampling) return;
  // query fragments, permuted like the key fragments (as in the scoring kernel)
  const int g = lane >> 2, t4 = lane & 3;
  uint32_t qf[8][2];
  {
    const uint32_t* qw = reinterpret_cast<const uint32_t*>(&qsb[g][0]);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int e = 8 * (4 * (j >> 1) + t4) + 4 * (j & 1);
      qf[j][0] = qw[e >> 1];
      qf[j][1] = qw[(e >> 1) + 1];
    }
  }
  const int c0 = 2 * t4, c1 = c0 + 1;
  const bool hv0 = c0 < G, hv1 = c1 < G;
  float mx0 = -INFINITY, mx1 = -INFINITY;
  for (int rb = 0; rb < P.Tu; rb += kSampleRows) {
    const int nr = min(kSampleRows, P.Tu - rb);
    __syncthreads();
    uint4* dst = reinterpret_cast<uint4*>(kt);
    if (rb == kSampleRows) {
#pragma unroll
      for (int q = 0; q < kPerThread; ++q) vbuf[q] = vbuf2[q];
    } else if (rb > kSampleRows) {
      load_pass(vbuf, rb, nr);  // the first two passes were loaded before the wait
    }
#pragma unroll
    for (int q = 0; q < kPerThread; ++q) {
      const int x = q * 256 + tid;
      if (x < nr * (kHeadDim / 8)) dst[x] = vbuf[q];
    }
    __syncthreads();
    // warp w scores rows [16 w, 16 w + 16) of this pass
    const int tr = kTileRows * warp;
    if (tr < nr) {
      const unsigned char* tb = kt + (size_t)tr * kHeadDim * 2;
      uint4 ra[4], rbv[4];
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        ra[v] = *reinterpret_cast<const uint4*>(tb + g * 256 + 16 * (4 * v + t4));
        rbv[v] = *reinterpret_cast<const uint4*>(tb + (g + 8) * 256 + 16 * (4 * v + t4));
      }
      float acc[4] = {0.f, 0.f, 0.f, 0.f}, acd[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        mma_16816(acc, ra[v].x, rbv[v].x, ra[v].y, rbv[v].y, qf[2 * v][0], qf[2 * v][1]);
        mma_16816(acd, ra[v].z, rbv[v].z, ra[v].w, rbv[v].w, qf[2 * v + 1][0], qf[2 * v + 1][1]);
      }
      const int r0 = tr + g;
      const bool v0 = r0 < nr, v1 = r0 + 8 < nr;
      const float s00 = (acc[0] + acd[0]) * kScoreScale, s01 = (acc[1] + acd[1]) * kScoreScale;
      const float s10 = (acc[2] + acd[2]) * kScoreScale, s11 = (acc[3] + acd[3]) * kScoreScale;
      if (hv0) {
        if (v0) mx0 = fmaxf(mx0, s00);
        if (v1) mx0 = fmaxf(mx0, s10);
      }
      if (hv1) {
        if (v0) mx1 = fmaxf(mx1, s01);
        if (v1) mx1 = fmaxf(mx1, s11);
      }
    }
  }
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
  }
  if (g == 0) {
    wmax[warp][c0] = mx0;
    if (c1 < kMaxGroup) wmax[warp][c1] = mx1;
  }
  __syncthreads();
  if (tid < G) {
    float m = -INFINITY;
    for (int w = 0; w < 8; ++w) m = fmaxf(m, wmax[w][tid]);
    P.samp_max[(list0 + tid) * kSampleUnits + z] = m;
  }
}

cudaError_t launch_prep(const Batch& B, cudaStream_t s) {
  int max_slabs = 0, max_z = 1;
  for (int j = 0; j < B.n; ++j) {
    max_slabs = max(max_slabs, B.p[j].P * B.p[j].Hkv);
    max_z = max(max_z, B.p[j].n_sample);
  }
  return launch_pdl(k_sample, dim3(max_slabs, B.n, max_z), dim3(256), 0, s, B);
}

// ---------------------------------------------------------------------------
// Scoring kernel.
//
// Grid: P.chunks CTAs per (problem, slab = (layer i, key head g)), one wave.
// Block: kScoreWarps compute warps + 2 threshold warps.
//
// All compute warps of a slab's CTAs take history units from the slab's shared unit
// counter, so SMs that run faster score more units, and walk each unit in tiles of 16
// tokens. Each warp streams its tiles through its own ring of kScoreStages shared
// memory buffers with TMA bulk copies (cp.async.bulk + mbarrier transaction counts),
// so the data in flight costs no registers. A tile's scores for the G query heads
// of the group come from 8 m16n8k16 bf16 MMAs: A = 16 keys x 16 dims, B = 16 dims x 8
// heads (G used). The contraction order over d is free, so lane (row g, column
// group t) reads the 16-byte chunks {4 v + t : v = 0..3} of rows g and g + 8, and the
// query fragments use the same permutation. The accumulator gives lane (g, t) the
// scores of keys g and g + 8 for heads 2t and 2t + 1.
//
// Candidate filter: a token is appended to its list when s >= thr[h], where thr[h] is
// always a lower bound of the list's k-th best score, so every top-k token is
// appended. Every appended score also counts in the CTA's ladder for its list (256
// levels 1/16 apart in log2 units, anchored at the list's best sampled unit); a
// threshold warp merges the CTA's counts into the list's global ladder and scans it
// from the top: the level where the count first reaches k bounds the k-th best score
// from below, because at least k appended tokens (of any CTA) score that much. The
// bound, shared through gthr, tracks the k-th best of everything scored so far.
// Each unit's softmax statistics (max, sum 2^(s - max)) are written per list; the
// list totals are combined later in unit order, whichever warp scored a unit.
// ---------------------------------------------------------------------------
constexpr int kUnitQueue = 8;    // > units a warp's issue cursor can run ahead
constexpr int kStagePairs = 64;  // staged candidates per (warp, list) before a write-out
static_assert(kStagePairs <= kReserve, "a write-out overflows into one new slot block");
static_assert(kStagePairs < 256, "staged counts are packed in 8 bits");

struct ScoreShared {
  int lad[kMaxGroup][kLadderLevels];  // this CTA's appended-score counts not yet merged
  float thr[kMaxGroup];
  float anchor[kMaxGroup];
  int all_done;
  unsigned long long bar[kScoreWarps][kScoreStages];  // one mbarrier per warp stage
  int uq[kScoreWarps][kUnitQueue];      // per warp: units taken, in order
  // per warp and list: appended (score, id) pairs waiting to be written out together
  float2 stage[kScoreWarps][kMaxGroup][kStagePairs];
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

// Appended score: count it at its ladder level in this CTA's shared counts.
__device__ __forceinline__ void ladder_add(ScoreShared& S, int c, float s, float a) {
  const int lv = __float2int_rd((s - a) * kLadderPerUnit) + kLadderZero;
  if (lv >= 0) atomicAdd(&S.lad[c][min(lv, kLadderLevels - 1)], 1);
}

constexpr int kThrLists = kMaxGroup / kThresholdWarps;  // lists per threshold warp

// The threshold warp merges this CTA's ladder counts into the lists' global counts and
// derives from those the lower bound thr of each list's k-th best score: if the
// levels >= i hold at least k appended tokens (of any CTA), the k-th best score is at
// least level i's lower edge. One level of margin covers the rounding of the level
// computation. Lane l handles the levels 255 - (32 q + l), q = 0..7, so that a warp's
// accesses to one block of 32 levels are consecutive words (no shared-memory bank
// conflicts, one 128-byte global transaction).
__device__ __noinline__ void threshold_warp(ScoreShared& S, const Prob& P, int list0, int k,
                                           int c0) {
  constexpr int per = kLadderLevels / 32;  // blocks of 32 levels; block 0 the top ones
  const int lane = threadIdx.x & 31;
  const int G = P.G;
  if (c0 >= G) return;  // no list of this warp's half
  volatile int* vdone = &S.all_done;
  volatile float* vthr = S.thr;
  auto level = [&](int q) { return kLadderLevels - 1 - (32 * q + lane); };
  for (int iter = 0; iter < (1 << 21); ++iter) {
    const int done = *vdone;
    // the bounds other CTAs published (lane c holds list c's)
    const float pub = lane < G ? ordered_to_float(*(volatile uint32_t*)(P.gthr + list0 + lane))
                               : -INFINITY;
    // the global counts of this warp's lists, all in flight at once (one round trip per
    // pass); they predate this pass's merge, whose counts are added to them here
    int cnt[kThrLists][per];
#pragma unroll
    for (int j = 0; j < kThrLists; ++j) {
      const int c = c0 + j;
      const volatile int* gl = P.ladder + (int64_t)(list0 + (c < G ? c : 0)) * kLadderLevels;
#pragma unroll
      for (int q = 0; q < per; ++q) cnt[j][q] = c < G ? gl[level(q)] : 0;
    }
#pragma unroll
    for (int j = 0; j < kThrLists; ++j) {
      const int c = c0 + j;
      if (c >= G) break;
      // merge this CTA's new counts of list c into the global ladder (not waited for)
      int* gl = P.ladder + (int64_t)(list0 + c) * kLadderLevels;
#pragma unroll
      for (int q = 0; q < per; ++q) {
        const int dv = atomicExch(&S.lad[c][level(q)], 0);
        if (dv) atomicAdd(gl + level(q), dv);
        cnt[j][q] += dv;
      }
      // the first block of 32 levels where the count from the top reaches k, then the
      // first level inside it
      int above = 0, qf = -1;
#pragma unroll
      for (int q = 0; q < per; ++q) {
        const int tq = __reduce_add_sync(0xffffffffu, (unsigned)cnt[j][q]);
        if (qf < 0 && above + tq >= k) qf = q;
        if (qf < 0) above += tq;
      }
      float t = -INFINITY;
      if (qf >= 0) {
        int mine = 0;
#pragma unroll
        for (int q = 0; q < per; ++q)
          if (q == qf) mine = cnt[j][q];
        int cum = mine;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
          const int y = __shfl_up_sync(0xffffffffu, cum, off);
          if (lane >= off) cum += y;
        }
        const unsigned hit = __ballot_sync(0xffffffffu, above + cum >= k);
        const int f = __ffs(hit) - 1;
        const int lv = kLadderLevels - 1 - (32 * qf + f);
        t = S.anchor[c] + (float)(lv - kLadderZero - 1) / kLadderPerUnit;
      }
      // published only when it raises the bound seen in gthr (the lists' words share a
      // few cache lines, which every CTA of the grid polls)
      const float other = __shfl_sync(0xffffffffu, pub, c);
      if (lane == 0 && t > other) atomicMax(P.gthr + list0 + c, float_to_ordered(t));  // not waited for
      t = fmaxf(t, other);
      if (lane == 0 && t > vthr[c]) vthr[c] = t;
    }
    __syncwarp();
    if (done >= kScoreWarps) break;
    __nanosleep(iter < 32 ? 128 : 1024);
  }
}

__global__ void __launch_bounds__(kScoreThreads, kScoreCtasPerSm)
    k_score(const __grid_constant__ Batch B) {
  __shared__ ScoreShared S;
  extern __shared__ __align__(128) unsigned char tiles[];  // [warp][stage][kTileBytes]
  const int b = blockIdx.x;
  const int pi = problem_of_block(B, b);
  const Prob& P = B.p[pi];
  const int local = b - P.cta_begin;
  const int n_slabs = P.P * P.Hkv;
  if (P.chunks <= 0) return;
  // In a one-wave grid consecutive CTAs go to different slabs, so each slab's CTAs
  // spread over the SMs; a grid of several waves keeps a slab's CTAs together.
  if (local >= n_slabs * P.chunks) return;
  const int slab = B.score_spread ? local % n_slabs : local / P.chunks;

  const int i = slab / P.Hkv, kvh = slab - i * P.Hkv;
  const int G = P.G;
  const int list0 = i * P.Hq + kvh * G;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int x = threadIdx.x; x < kMaxGroup * kLadderLevels; x += blockDim.x)
    (&S.lad[0][0])[x] = 0;
  if (threadIdx.x == 0) S.all_done = 0;
  if (threadIdx.x < kScoreWarps * kScoreStages)
    mbar_init(smem_u32(&S.bar[0][0] + threadIdx.x), 1u);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  __syncthreads();

  const int Tu = P.Tu;
  const int tpu = (Tu + kTileRows - 1) / kTileRows;
  const int Uh = P.Uh;
  const __nv_bfloat16* slab_keys = P.keys + (int64_t)slab * P.ncap * kHeadDim;
  unsigned char* my_tiles = tiles + (size_t)(warp < kScoreWarps ? warp : 0) * kScoreStages * kTileBytes;
  const uint32_t my_tiles_s = smem_u32(my_tiles);
  const uint32_t my_bars = smem_u32(&S.bar[warp < kScoreWarps ? warp : 0][0]);
  // Lane 0 starts the bulk copy of tile t (unit uu, tile jj of the unit) into its
  // stage once the warp's reads of that stage are ordered before the async write.
  auto issue = [&](int t, int uu, int jj) {
    if (uu >= Uh) return;
    const int r0 = kTileRows * jj;
    const int nrows = min(kTileRows, Tu - r0);
    const int st = t % kScoreStages;
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      const uint32_t bar = my_bars + 8u * st;
      const uint32_t bytes = (uint32_t)nrows * kHeadDim * 2u;
      mbar_expect_tx(bar, bytes);
      bulk_load(my_tiles_s + (uint32_t)st * kTileBytes,
                slab_keys + ((int64_t)uu * Tu + r0) * kHeadDim, bytes, bar);
    }
  };
  // Each compute warp's first unit is fixed (a slab's CTAs take units idx * kScoreWarps
  // + warp; the slab's counter, reset by the prep kernel, hands out the rest), so its
  // first tiles are requested before the wait for the prep kernel: they read only the
  // keys, which no kernel of the chain writes.
  int iu = Uh;
  int n_pre = 0;
  if (warp < kScoreWarps) {
    const int idx = B.score_spread ? local / n_slabs : local - slab * P.chunks;
    const int first = idx * kScoreWarps + warp;
    iu = first < Uh ? first : Uh;
    n_pre = min(kScoreStages, tpu);
    for (int t = 0; t < n_pre; ++t) issue(t, iu, t);
  }
  pdl_wait();     // q_eff, anchors and resets of the prep kernel
  pdl_release();
  if (threadIdx.x < kMaxGroup) {
    // a CTA that starts late begins with the bound published by the earlier ones
    S.thr[threadIdx.x] = threadIdx.x < G ? ordered_to_float(P.gthr[list0 + threadIdx.x]) : -INFINITY;
    S.anchor[threadIdx.x] = threadIdx.x < G ? list_anchor(P, list0 + threadIdx.x) : 0.f;
  }
  __syncthreads();

  const int k = B.k;
  if (warp >= kScoreWarps) {
    threshold_warp(S, P, list0, k, (warp - kScoreWarps) * kThrLists);
    return;
  }

  const int g = lane >> 2, t4 = lane & 3;
  // Query fragments (B operand), permuted like the key fragment reads below.
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
  int* next_unit = P.next_unit + slab * kUnitCounterStride;
  const int64_t cbase0 = (int64_t)(hv0 ? L0 : list0) * P.cand_cap;
  const int64_t cbase1 = (int64_t)(hv1 ? L1 : list0) * P.cand_cap;
  const volatile float* vthr = S.thr;
  const unsigned gmask = 0x11111111u << t4;
  const unsigned lt_mask = (1u << lane) - 1u;
  const float an0 = S.anchor[c0], an1 = S.anchor[c1 < kMaxGroup ? c1 : 0];
  // Candidate slots reserved for this lane group's two lists (identical in its 8 lanes).
  int rp0 = 0, rl0 = 0, rp1 = 0, rl1 = 0;

  // Appends the scores of keys tok0 (row g) and tok0 + 8 (row g + 8) that reach the
  // current thresholds, and counts them in the CTA's ladder.
  // Staged pairs of this lane group's two lists (counts identical in its 8 lanes),
  // packed as sc0 | sc1 << 8.
  int scp = 0;
  // Writes the staged pairs of every lane group to their lists' reserved slots (8 lanes
  // store 64 contiguous bytes at a time), reserving a new slot block when one runs out.
  // The whole warp calls it.
  auto flush = [&]() {
    __syncwarp();
    const int sc0 = scp & 0xff, sc1 = scp >> 8;
    const bool need0 = sc0 > rl0, need1 = sc1 > rl1;
    int nb0 = 0, nb1 = 0;
    if (g == 0 && need0) nb0 = atomicAdd(P.cand_cnt + L0, kReserve);
    if (g == 0 && need1) nb1 = atomicAdd(P.cand_cnt + L1, kReserve);
    nb0 = __shfl_sync(0xffffffffu, nb0, t4);
    nb1 = __shfl_sync(0xffffffffu, nb1, t4);
    for (int r = g; r < sc0; r += 8)
      P.cand_pair[cbase0 + (r < rl0 ? rp0 + r : nb0 + (r - rl0))] = S.stage[warp][c0][r];
    for (int r = g; r < sc1; r += 8)
      P.cand_pair[cbase1 + (r < rl1 ? rp1 + r : nb1 + (r - rl1))] = S.stage[warp][c1][r];
    if (need0) {
      rp0 = nb0 + (sc0 - rl0);
      rl0 = kReserve - (sc0 - rl0);
    } else {
      rp0 += sc0;
      rl0 -= sc0;
    }
    if (need1) {
      rp1 = nb1 + (sc1 - rl1);
      rl1 = kReserve - (sc1 - rl1);
    } else {
      rp1 += sc1;
      rl1 -= sc1;
    }
    scp = 0;
    __syncwarp();
  };
  auto append = [&](float s00, float s01, float s10, float s11, int tok0, bool v0, bool v1,
                    float thr0, float thr1) {
    const bool p00 = hv0 && v0 && s00 >= thr0, p10 = hv0 && v1 && s10 >= thr0;
    const bool p01 = hv1 && v0 && s01 >= thr1, p11 = hv1 && v1 && s11 >= thr1;
    const int tok1 = tok0 + 8;
    const unsigned b00 = __ballot_sync(0xffffffffu, p00) & gmask;
    const unsigned b10 = __ballot_sync(0xffffffffu, p10) & gmask;
    const unsigned b01 = __ballot_sync(0xffffffffu, p01) & gmask;
    const unsigned b11 = __ballot_sync(0xffffffffu, p11) & gmask;
    const int n0 = __popc(b00) + __popc(b10), n1 = __popc(b01) + __popc(b11);
    if (__any_sync(0xffffffffu, (scp & 0xff) + n0 > kStagePairs || (scp >> 8) + n1 > kStagePairs))
      flush();
    const int sc0 = scp & 0xff, sc1 = scp >> 8;
    if (p00) {
      S.stage[warp][c0][sc0 + __popc(b00 & lt_mask)] = make_float2(s00, __int_as_float(tok0));
      ladder_add(S, c0, s00, an0);
    }
    if (p10) {
      S.stage[warp][c0][sc0 + __popc(b00) + __popc(b10 & lt_mask)] =
          make_float2(s10, __int_as_float(tok1));
      ladder_add(S, c0, s10, an0);
    }
    if (p01) {
      S.stage[warp][c1][sc1 + __popc(b01 & lt_mask)] = make_float2(s01, __int_as_float(tok0));
      ladder_add(S, c1, s01, an1);
    }
    if (p11) {
      S.stage[warp][c1][sc1 + __popc(b01) + __popc(b11 & lt_mask)] =
          make_float2(s11, __int_as_float(tok1));
      ladder_add(S, c1, s11, an1);
    }
    scp += n0 + (n1 << 8);
  };

  // After the first, units come from the slab's shared counter: every warp of the
  // slab's CTAs takes the next unit when it needs one, so faster SMs score more units.
  // Lane 0 takes its next unit one unit ahead (the atomic's latency hides behind a unit
  // of work); the units a warp takes are queued in shared memory for its consume cursor.
  int* uq = S.uq[warp];
  int pre = lane == 0 ? atomicAdd(next_unit, 1) : 0;
  auto take = [&]() {
    const int u = __shfl_sync(0xffffffffu, pre, 0);
    if (lane == 0) pre = u < Uh ? atomicAdd(next_unit, 1) : Uh;
    return min(u, Uh);
  };
  int ij = 0, nq = 0;                  // issue position (unit iu, tile ij), units queued
  if (lane == 0) uq[0] = iu;
  nq = 1;
  __syncwarp();
  int cu = iu, cj = 0, qh = 0;         // consume position, queue head
  auto advance_issue = [&]() {
    if (++ij == tpu) {
      ij = 0;
      iu = iu < Uh ? take() : Uh;
      if (lane == 0) uq[nq % kUnitQueue] = iu;
      ++nq;
      __syncwarp();
    }
  };
  for (int t = 0; t < kScoreStages; ++t) {
    if (t >= n_pre) issue(t, iu, ij);  // the first n_pre went out before the wait
    advance_issue();
  }

  float m0 = -INFINITY, l0 = 0.f, m1 = -INFINITY, l1 = 0.f;
  int t = 0;
  bool aborted = false;
  for (; cu < Uh; ++t) {
    const int st = t % kScoreStages;
    const bool ok = mbar_wait_limit(my_bars + 8u * st, (uint32_t)((t / kScoreStages) & 1),
                                    B.wait_polls);
    if (!__all_sync(0xffffffffu, ok)) {
      aborted = true;
      break;
    }
    const unsigned char* tb = my_tiles + (size_t)st * kTileBytes;
    // A fragments: lane (g, t4) takes the 16-byte chunks 4v + t4 of rows g and g + 8.
    uint4 ra[4], rb[4];
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      ra[v] = *reinterpret_cast<const uint4*>(tb + g * 256 + 16 * (4 * v + t4));
      rb[v] = *reinterpret_cast<const uint4*>(tb + (g + 8) * 256 + 16 * (4 * v + t4));
    }
    // two accumulators halve the dependent MMA chain
    float acc[4] = {0.f, 0.f, 0.f, 0.f}, acd[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      mma_16816(acc, ra[v].x, rb[v].x, ra[v].y, rb[v].y, qf[2 * v][0], qf[2 * v][1]);
      mma_16816(acd, ra[v].z, rb[v].z, ra[v].w, rb[v].w, qf[2 * v + 1][0], qf[2 * v + 1][1]);
    }
    const int u = cu, j = cj;
    if (++cj == tpu) {
      cj = 0;
      ++qh;
      cu = uq[qh % kUnitQueue];
    }
    issue(t + kScoreStages, iu, ij);   // the stage's data now sits in registers
    advance_issue();

    if (j == 0) {
      m0 = m1 = -INFINITY;
      l0 = l1 = 0.f;
    }
    const float thr0 = hv0 ? vthr[c0] : INFINITY;
    const float thr1 = hv1 ? vthr[c1] : INFINITY;
    const int r0 = kTileRows * j + g;
    const bool v0 = r0 < Tu, v1 = r0 + 8 < Tu;
    const float s00 = (acc[0] + acd[0]) * kScoreScale, s01 = (acc[1] + acd[1]) * kScoreScale;
    const float s10 = (acc[2] + acd[2]) * kScoreScale, s11 = (acc[3] + acd[3]) * kScoreScale;
    stats_update(m0, l0, s00, v0, s10, v1);
    stats_update(m1, l1, s01, v0, s11, v1);
    const bool pass = (hv0 && ((v0 && s00 >= thr0) || (v1 && s10 >= thr0))) ||
                      (hv1 && ((v0 && s01 >= thr1) || (v1 && s11 >= thr1)));
    if (__any_sync(0xffffffffu, pass)) append(s00, s01, s10, s11, u * Tu + r0, v0, v1, thr0, thr1);
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
        if (hv0) P.ustats[(int64_t)L0 * P.ucap + u] = make_float2(m0, l0);
        if (hv1) P.ustats[(int64_t)L1 * P.ucap + u] = make_float2(m1, l1);
      }
    }
  }
  flush();
  // unused reserved slots are marked empty (score -inf)
  for (int x = g; x < rl0; x += 8) P.cand_pair[cbase0 + rp0 + x].x = -INFINITY;
  for (int x = g; x < rl1; x += 8) P.cand_pair[cbase1 + rp1 + x].x = -INFINITY;
  if (aborted) {
    // report, then let the copies already in flight land before the CTA exits (with the
    // default limit: the copies were issued and complete)
    if (lane == 0) atomicOr(P.status, kStatusTimeout);
    // stages of tiles t .. t + kScoreStages - 1 that were issued (units < Uh)
    int ru = cu, rj = cj, rq = qh;
    for (int r = t; r < t + kScoreStages && ru < Uh; ++r) {
      mbar_wait_bounded(my_bars + 8u * (r % kScoreStages), (uint32_t)((r / kScoreStages) & 1));
      if (++rj == tpu) {
        rj = 0;
        ++rq;
        ru = rq < nq ? uq[rq % kUnitQueue] : Uh;
      }
    }
  }
  __threadfence_block();
  if (lane == 0) atomicAdd(&S.all_done, 1);
}

int score_chunks_per_slab(int n_slabs_total, int hist_units, int sm_count) {
  // Pick the chunk length (in units) that minimises waves x chunk length over the
  // resident CTA slots; ties go to fewer CTAs.
  if (hist_units <= 0 || n_slabs_total <= 0) return 0;
  const int64_t slots = (int64_t)sm_count * kScoreCtasPerSm;
  int best_c = 1;
  int64_t best_cost = INT64_MAX;
  for (int c = 1; c <= hist_units && c <= kMaxChunksPerSlab; ++c) {
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

int score_slots(int sm_count) { return sm_count * kScoreCtasPerSm; }

cudaError_t launch_score(const Batch& B, cudaStream_t s) {
  if (B.score_ctas <= 0) return cudaSuccess;
  const int smem = kScoreWarps * kScoreStages * kTileBytes;
  cudaError_t e = ensure_smem((const void*)k_score, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(k_score, dim3(B.score_ctas), dim3(kScoreThreads), (size_t)smem, s, B);
}

}  // namespace ss
