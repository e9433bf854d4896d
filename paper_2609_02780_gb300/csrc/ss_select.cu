// Evidence selection after key scoring (Sec. 4.2, Eq. 11-12):
//   k_select   exact top-k of every list from its candidate array, softmax statistics
//              from the per-unit (max, sum) pairs, normalised weights, unit votes
//              (one per (list, selected token) in the unit, integer atomics)
//   k_mass     attention mass of every history unit (summed weights of all tokens)
//   k_pool     the vote-ranked pool: top min(pool_mult * K, |H|) units by
//              (votes desc, mass desc, unit id asc)
//   k_gram / k_maxmin  greedy max-min diversity over the pool's descriptors, then each
//              pick plus its preceding units, deduplicated, ascending (Eq. 12)
// No floating-point atomics: every float reduction has a fixed order, so results are
// bit-identical from run to run.
#include "ss_internal.cuh"
#include "ss_device.cuh"

namespace ss {

// k_select runs 1024 threads per list with room for 16384 survivors, or, when the lists
// outnumber the SMs, 512 threads with room for 8192 so that two lists share an SM.
constexpr int kMassUnits = 32;     // history units per mass block
template <int kThreads>
constexpr int sel_cap() { return kThreads >= 1024 ? 16384 : 8192; }  // survivors in smem
constexpr int kFineBins = 2048;  // second-level score histogram of k_select

__device__ __forceinline__ unsigned long long cand_key(float s, int32_t id) {
  // Larger key = better: score desc, then id asc.
  return ((unsigned long long)float_to_ordered(s) << 32) | (uint32_t)(~(uint32_t)id);
}

// Bitonic sort of a[0, n2) (n2 a power of two) into descending order; all threads.
__device__ void bitonic_desc(unsigned long long* a, int n2) {
  for (int size = 2; size <= n2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int t = threadIdx.x; t < (n2 >> 1); t += blockDim.x) {
        const int i = 2 * t - (t & (stride - 1));
        const int j = i + stride;
        const bool desc = (i & size) == 0;
        const unsigned long long x = a[i], y = a[j];
        if ((x < y) == desc) {
          a[i] = y;
          a[j] = x;
        }
      }
      __syncthreads();
    }
  }
}

// Descending bitonic sort of a[0, n2) for 64 <= n2 <= 2 * blockDim.x (n2 a power of two)
// with the compare-exchanges of stride < 64 done in registers: thread (warp w, lane l)
// holds elements 64 w + l and 64 w + 32 + l; strides 1..16 pair lanes (shuffles),
// stride 32 pairs a thread's two registers, longer strides go through shared memory.
__device__ __forceinline__ unsigned long long bitonic_keep(unsigned long long mine,
                                                           unsigned long long other,
                                                           bool lower, bool desc) {
  // the lower element of a pair keeps the larger key in a descending block
  const bool take_max = (lower == desc);
  return take_max ? (mine > other ? mine : other) : (mine < other ? mine : other);
}

__device__ void bitonic_desc_hybrid(unsigned long long* a, int n2) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const bool active = 64 * warp < n2;
  const int i0 = 64 * warp + lane, i1 = i0 + 32;
  unsigned long long r0 = active ? a[i0] : 0ull, r1 = active ? a[i1] : 0ull;
  auto reg_stages = [&](int size, int top) {
    for (int stride = top; stride > 0; stride >>= 1) {
      if (stride == 32) {
        const bool desc = (i0 & size) == 0;
        const unsigned long long x0 = r0, x1 = r1;
        r0 = bitonic_keep(x0, x1, true, desc);
        r1 = bitonic_keep(x1, x0, false, desc);
      } else {
        const unsigned long long o0 = __shfl_xor_sync(0xffffffffu, r0, stride);
        const unsigned long long o1 = __shfl_xor_sync(0xffffffffu, r1, stride);
        const bool lower = (lane & stride) == 0;
        r0 = bitonic_keep(r0, o0, lower, (i0 & size) == 0);
        r1 = bitonic_keep(r1, o1, lower, (i1 & size) == 0);
      }
    }
  };
  for (int size = 2; size <= min(n2, 64); size <<= 1) reg_stages(size, size >> 1);
  for (int size = 128; size <= n2; size <<= 1) {
    if (active) {
      a[i0] = r0;
      a[i1] = r1;
    }
    __syncthreads();
    for (int stride = size >> 1; stride >= 64; stride >>= 1) {
      for (int t = threadIdx.x; t < (n2 >> 1); t += blockDim.x) {
        const int i = 2 * t - (t & (stride - 1));
        const int j = i + stride;
        const bool desc = (i & size) == 0;
        const unsigned long long x = a[i], y = a[j];
        if ((x < y) == desc) {
          a[i] = y;
          a[j] = x;
        }
      }
      __syncthreads();
    }
    r0 = active ? a[i0] : 0ull;
    r1 = active ? a[i1] : 0ull;
    reg_stages(size, 32);
  }
  __syncthreads();
  if (active) {
    a[i0] = r0;
    a[i1] = r1;
  }
  __syncthreads();
}

// Descending sort of keys[0, ns) by bucketing on the score (the upper 32 bits of a key):
// 2048 buckets over [lo, hi] (every key's score lies there), a counting scatter in
// bucket order into the upper half of `keys`, then every key placed by its rank inside
// its bucket. Needs ns <= kSelCap / 2 and buckets of at most kBucketMax keys; returns
// false, with keys untouched, when a bucket is larger (then the caller sorts another
// way). All threads of the block call it.
constexpr int kBucketMax = 32;

template <int kThreads>
__device__ bool bucket_sort_desc(unsigned long long* keys, int ns, float lo, float hi,
                                 int* hist, int* cursor, int* sflag) {
  const int tid = threadIdx.x;
  const uint32_t klo = float_to_ordered(lo), khi = float_to_ordered(hi);
  // buckets linear in the ordered score bits, in fp32 (rounding keeps the map
  // monotonic, which is all the order needs)
  const float scale = (float)kFineBins / ((float)(khi - klo) + 1.0f);
  auto bucket = [&](unsigned long long key) -> int {
    const uint32_t ok = (uint32_t)(key >> 32);
    const uint32_t d = ok > klo ? ok - klo : 0u;
    const int b = (int)((float)d * scale);
    return kFineBins - 1 - min(b, kFineBins - 1);  // best scores first
  };
  for (int b = tid; b < kFineBins; b += blockDim.x) hist[b] = 0;
  if (tid == 0) *sflag = 0;
  __syncthreads();
  for (int i = tid; i < ns; i += blockDim.x) atomicAdd(&hist[bucket(keys[i])], 1);
  __syncthreads();
  // exclusive scan of the bucket counts (each thread owns consecutive buckets)
  constexpr int kPerT = kFineBins / kThreads;
  int c[kPerT], tot = 0;
#pragma unroll
  for (int q = 0; q < kPerT; ++q) {
    c[q] = hist[kPerT * tid + q];
    tot += c[q];
    if (c[q] > kBucketMax) *sflag = 1;
  }
  __shared__ int sw[32];
  int run = block_excl_scan(tot, sw);
  const bool big = *sflag != 0;
  __syncthreads();
  if (big) return false;
#pragma unroll
  for (int q = 0; q < kPerT; ++q) {
    hist[kPerT * tid + q] = run;
    cursor[kPerT * tid + q] = run;
    run += c[q];
  }
  __syncthreads();  // every bucket's start is set before any thread scatters
  // scatter into the upper half (ns <= half the capacity), bucket by bucket
  unsigned long long* tmp = keys + sel_cap<kThreads>() / 2;
  for (int i = tid; i < ns; i += blockDim.x) {
    const unsigned long long key = keys[i];
    tmp[atomicAdd(&cursor[bucket(key)], 1)] = key;
  }
  __syncthreads();
  // every key's place inside its bucket: the bucket's keys above it (equal keys by
  // position), at most kBucketMax comparisons per key
  for (int i = tid; i < ns; i += blockDim.x) {
    const unsigned long long key = tmp[i];
    const int b = bucket(key);
    const int b0 = hist[b], b1 = cursor[b];  // after the scatter: the bucket's end
    int r = 0;
    for (int j = b0; j < b1; ++j) {
      const unsigned long long y = tmp[j];
      r += (y > key || (y == key && j < i)) ? 1 : 0;
    }
    keys[b0 + r] = key;
  }
  __syncthreads();
  return true;
}

__device__ __forceinline__ int next_pow2(int x) {
  int p = 1;
  while (p < x) p <<= 1;
  return p;
}

// ---------------------------------------------------------------------------
// Exact top-k of one list (Eq. 11). The candidate array holds every token whose score
// reached a lower bound `lo` of the list's k-th best score. A 2048-bin histogram of
// the candidates over [lo, max] locates the bin of the n-th best (n = min(k, tokens));
// the candidates from that bin up are sorted in shared memory by (score desc, id asc).
// If they do not fit (massive ties), an 8-pass radix select on the 64-bit keys over
// the candidate array finds the n-th key exactly.
// ---------------------------------------------------------------------------
// kGeneral: the general path (one list per layer, or centroid candidates). Its lists
// hold every candidate (a dense row), its softmax statistics come from that row, and
// with one list per layer the row holds the head-averaged weights themselves.
template <bool kGeneral, int kThreads>
__global__ void __launch_bounds__(kThreads, 1024 / kThreads) k_select_t(const __grid_constant__ Batch B) {
  constexpr int kSelCap = sel_cap<kThreads>();
  extern __shared__ unsigned long long skeys[];
  __shared__ int s_hist[kFineBins];
  __shared__ int s_cursor[kFineBins];
  __shared__ int s_flag;
  __shared__ float s_m[32], s_l[32];
  __shared__ int s_n, s_bstar, s_rem;
  __shared__ unsigned long long s_prefix;
  __shared__ float s_lb;

  pdl_wait();
  pdl_release();
  const int pi = blockIdx.y;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  if (retrieval_timed_out(P)) return;
  // rows of weights rather than scores: one list per layer (head-averaged weights) or
  // per-query-head lists of row-averaged weights; their candidate ids are the positions
  const bool mean = kGeneral && (B.head_agg == 1 || B.q_agg == 2);
  const int n_lists = (kGeneral && B.head_agg == 1) ? P.P : P.P * P.Hq;
  const int L = blockIdx.x;
  if (L >= n_lists) return;
  const int tid = threadIdx.x, lane = tid & 31;
  const int k = B.k;

  float M = -INFINITY, Ls = 0.f;
  const int64_t n_tok = kGeneral ? (int64_t)P.n_cand : (int64_t)P.Uh * P.Tu;
  int n = (int)min((int64_t)k, n_tok);
  float lo = -INFINITY;
  if constexpr (!kGeneral) {
    const uint32_t gthr = P.gthr[L];  // the bound the score kernel published
    // Warp 0 first derives a tighter bound from the list's completed ladder of
    // appended-score counts (its loads overlap the other warps' statistics loads): if
    // the levels >= i hold n tokens, the n-th best score is at least level i's lower
    // edge (one level of margin for the rounding of the level computation).
    if (tid < 32) {
      constexpr int per = kLadderLevels / 32;
      const int* lad = P.ladder + (int64_t)L * kLadderLevels;
      const float anchor = list_anchor(P, L);
      int cntl[per];
      int sum = 0;
#pragma unroll
      for (int q = 0; q < per; ++q) {
        cntl[q] = lad[kLadderLevels - 1 - (per * lane + q)];
        sum += cntl[q];
      }
      int cum = sum;
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, cum, off);
        if (lane >= off) cum += y;
      }
      const unsigned hit = __ballot_sync(0xffffffffu, cum >= n);
      if (hit == 0u) {
        if (lane == 0) s_lb = -INFINITY;
      } else {
        const int f = __ffs(hit) - 1;
        if (lane == f) {
          int run = cum - sum, qf = per - 1;
#pragma unroll
          for (int q = 0; q < per; ++q) {
            run += cntl[q];
            if (run >= n && qf == per - 1 && q < per - 1) qf = q;
          }
          const int lv = kLadderLevels - 1 - (per * lane + qf);
          s_lb = anchor + (float)(lv - kLadderZero - 1) / kLadderPerUnit;
        }
      }
    }
    // softmax statistics from the per-unit pairs in a fixed order (thread t takes units
    // t, t + 1024, ...; then a fixed tree), whichever warps scored the units; four
    // loads in flight per thread
    const float2* us = P.ustats + (int64_t)L * P.ucap;
    const int Uh = P.Uh;
    for (int u0 = tid; u0 < Uh; u0 += 4 * (int)blockDim.x) {
      float2 v[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int u = u0 + e * blockDim.x;
        v[e] = u < Uh ? us[u] : make_float2(0.f, 0.f);
      }
#pragma unroll
      for (int e = 0; e < 4; ++e)
        if (u0 + e * (int)blockDim.x < Uh) ml_combine(M, Ls, v[e].x, v[e].y);
    }
    block_ml(M, Ls, s_m, s_l);  // its barriers also publish s_lb
    if (tid == 0) P.list_ml[L] = make_float2(M, Ls);
    lo = fmaxf(ordered_to_float(gthr), s_lb);
  }

  int32_t* tok_out = P.topk_tok + (int64_t)L * k;
  float* w_out = P.topk_w + (int64_t)L * k;
  float* s_out = P.topk_s ? P.topk_s + (int64_t)L * k : nullptr;
  if (n == 0) {
    if (kGeneral && tid == 0) P.list_ml[L] = make_float2(-INFINITY, 0.f);
    for (int r = tid; r < k; r += blockDim.x) {
      tok_out[r] = -1;
      w_out[r] = 0.f;
      if (s_out) s_out[r] = -INFINITY;
    }
    return;
  }
  const int cnt = kGeneral ? P.n_cand : P.cand_cnt[L];
  // candidates: (score, id) pairs appended by the score kernel, or the general path's
  // dense rows of values and ids
  const float* cs = (B.head_agg == 1 ? P.aval : P.cand_s) + (int64_t)L * P.cand_cap;
  const int32_t* ci = P.cand_id + (int64_t)L * P.cand_cap;
  const float2* cp = P.cand_pair + (int64_t)L * P.cand_cap;
  auto sc_at = [&](int x) -> float {
    if constexpr (kGeneral) return cs[x];
    else return cp[x].x;
  };
  auto id_at = [&](int x) -> int32_t {
    if constexpr (kGeneral) return mean ? (int32_t)x : ci[x];
    else return __float_as_int(cp[x].y);
  };
  // Visits every candidate x < cnt with its value. A dense row of weights (16-byte
  // aligned, its capacity a multiple of 64) is read in 16-byte loads, eight per thread in
  // flight: thread t takes the groups of four x = 4 g .. 4 g + 3 for g = t, t + T, ...;
  // other rows and the score kernel's candidate lists one value at a time, four in flight.
  auto each = [&](auto&& f) {
    if (kGeneral && mean) {
      const float4* c4 = reinterpret_cast<const float4*>(cs);
      const int n4 = (cnt + 3) >> 2;
      for (int g0 = tid; g0 < n4; g0 += 8 * (int)blockDim.x) {
        float4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int g = g0 + u * blockDim.x;
          v[u] = g < n4 ? c4[g] : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int x = 4 * (g0 + u * (int)blockDim.x);
          if (x < cnt) f(x, v[u].x);
          if (x + 1 < cnt) f(x + 1, v[u].y);
          if (x + 2 < cnt) f(x + 2, v[u].z);
          if (x + 3 < cnt) f(x + 3, v[u].w);
        }
      }
    } else {
      for (int x0 = tid; x0 < cnt; x0 += 4 * (int)blockDim.x) {
        float v[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int x = x0 + e * blockDim.x;
          v[e] = x < cnt ? sc_at(x) : 0.f;
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int x = x0 + e * blockDim.x;
          if (x < cnt) f(x, v[e]);
        }
      }
    }
  };
  // A dense row of weights (values in [0, 1]) also gets its histogram in the same pass:
  // 32 bins per octave from the value's bits (exactly monotonic in the value), the top bin
  // holding [2^-1/32 .. 1], bin 0 everything below 2^-64.
  const bool wbins = kGeneral && mean && cnt > 2 * kThreads;
  auto wbin = [](float v) -> int {
    const int b = (int)(__float_as_uint(fmaxf(v, 0.f)) >> 18) - (63 << 5);
    return min(max(b, 0), kFineBins - 1);
  };
  if constexpr (kGeneral) {
    // statistics of the dense row in a fixed order: (max, sum 2^(s - max)) of the
    // scores, or (max, sum) of the head-averaged weights; and its minimum (the bound)
    float m = -INFINITY, l = 0.f, mn = INFINITY;
    if (wbins) {
      for (int x = tid; x < kFineBins; x += blockDim.x) s_hist[x] = 0;
      __syncthreads();
      each([&](int, float v) {
        m = fmaxf(m, v);
        l += v;
        mn = fminf(mn, v);
        atomicAdd(&s_hist[wbin(v)], 1);
      });
      l = block_sum(l, s_l);
      m = -block_min(-m, s_m);
    } else if (mean) {
      each([&](int, float v) {
        m = fmaxf(m, v);
        l += v;
        mn = fminf(mn, v);
      });
      l = block_sum(l, s_l);
      m = -block_min(-m, s_m);
    } else {
      each([&](int, float v) {
        ml_combine(m, l, v, 1.f);
        mn = fminf(mn, v);
      });
      block_ml(m, l, s_m, s_l);
    }
    lo = block_min(mn, s_m);
    M = m;
    Ls = l;
    if (tid == 0) P.list_ml[L] = make_float2(M, Ls);
  }
  if (lo == -INFINITY) {
    // no bound: start from the smallest real candidate (unused reserved slots hold
    // -inf and are never candidates)
    float mn = INFINITY;
    each([&](int, float s) {
      if (s > -INFINITY) mn = fminf(mn, s);
    });
    lo = block_min(mn, s_m);
  }
  // A dense row of more than 2048 candidates goes straight to the histogram below.
  const bool dense = kGeneral && cnt > 2 * kThreads;
  // collect the candidates at or above the bound (warp-aggregated slot counter)
  if (tid == 0) s_n = 0;
  __syncthreads();
  if constexpr (!kGeneral) {
    // each thread loads 4 x 2 consecutive (score, id) slots per round (16-byte loads; the
    // list's slots start 256-byte aligned); a warp claims its output slots with one atomic
    constexpr int kU = 4;
    const float4* cp4 = reinterpret_cast<const float4*>(cp);
    const int n2p = (cnt + 1) >> 1;
    const float4 ninf = make_float4(-INFINITY, 0.f, -INFINITY, 0.f);
    for (int b0 = 0; b0 < n2p; b0 += kU * (int)blockDim.x) {
      float4 v4[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int x2 = b0 + u * blockDim.x + tid;
        v4[u] = x2 < n2p ? cp4[x2] : ninf;
      }
      unsigned kb = 0u;
#pragma unroll
      for (int e = 0; e < 2 * kU; ++e) {
        const int x = 2 * (b0 + (e >> 1) * blockDim.x + tid) + (e & 1);
        const float v = (e & 1) ? v4[e >> 1].z : v4[e >> 1].x;
        if (x < cnt && v >= lo) kb |= 1u << e;
      }
      const int c = __popc(kb);
      int incl = c;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
      }
      int base = 0;
      if (lane == 31 && incl) base = atomicAdd(&s_n, incl);
      int pos = __shfl_sync(0xffffffffu, base, 31) + incl - c;
#pragma unroll
      for (int e = 0; e < 2 * kU; ++e) {
        if ((kb >> e) & 1u) {
          const float v = (e & 1) ? v4[e >> 1].z : v4[e >> 1].x;
          const float idf = (e & 1) ? v4[e >> 1].w : v4[e >> 1].y;
          if (pos < kSelCap) skeys[pos] = cand_key(v, __float_as_int(idf));
          ++pos;
        }
      }
    }
  } else if (!dense) {
    // each thread loads 4 x 4 consecutive slots per round (16-byte loads; the list's slots
    // start 256-byte aligned); a warp claims the round's output slots with one atomic
    constexpr int kU = 4;
    const float4* cs4 = reinterpret_cast<const float4*>(cs);
    const int n4 = (cnt + 3) >> 2;
    const float4 ninf = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
    for (int b0 = 0; b0 < n4; b0 += kU * (int)blockDim.x) {
      float4 v4[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int x4 = b0 + u * blockDim.x + tid;
        v4[u] = x4 < n4 ? cs4[x4] : ninf;
      }
      float v[4 * kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        v[4 * u] = v4[u].x;
        v[4 * u + 1] = v4[u].y;
        v[4 * u + 2] = v4[u].z;
        v[4 * u + 3] = v4[u].w;
      }
      unsigned kb = 0u;
#pragma unroll
      for (int e = 0; e < 4 * kU; ++e) {
        const int x = 4 * (b0 + (e >> 2) * blockDim.x + tid) + (e & 3);
        if (x < cnt && v[e] >= lo) kb |= 1u << e;
      }
      const int c = __popc(kb);
      int incl = c;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
      }
      int base = 0;
      if (lane == 31 && incl) base = atomicAdd(&s_n, incl);
      int pos = __shfl_sync(0xffffffffu, base, 31) + incl - c;
#pragma unroll
      for (int e = 0; e < 4 * kU; ++e) {
        if ((kb >> e) & 1u) {
          const int x = 4 * (b0 + (e >> 2) * blockDim.x + tid) + (e & 3);
          if (pos < kSelCap) skeys[pos] = cand_key(v[e], id_at(x));
          ++pos;
        }
      }
    }
  }
  __syncthreads();
  int ns = dense ? kSelCap + 1 : s_n;
  if (ns > kSelCap) {
    // Too many: a 2048-bin histogram of the candidates over [lo, max] (linear) locates the
    // bin of the n-th best; keep the candidates from that bin up.
    // (a dense row of weights has its histogram from the statistics pass, in the bins
    // of the value's bits)
    const float hi = M;
    const float scale = (hi > lo) ? (float)kFineBins / (hi - lo) : 0.f;
    auto fbin = [&](float s) -> int {
      if (wbins) return wbin(s);
      const int b = (int)((s - lo) * scale);
      return min(max(b, 0), kFineBins - 1);
    };
    if (!wbins) {
      for (int x = tid; x < kFineBins; x += blockDim.x) s_hist[x] = 0;
      __syncthreads();
      each([&](int, float s) {
        if (s >= lo) atomicAdd(&s_hist[fbin(s)], 1);
      });
    }
    __syncthreads();
    if (tid < 32) {
      constexpr int per = kFineBins / 32;  // lane 0 holds the top bins
      int sum = 0;
      for (int q = 0; q < per; ++q) sum += s_hist[kFineBins - 1 - (per * lane + q)];
      int cum = sum;
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, cum, off);
        if (lane >= off) cum += y;
      }
      const unsigned hit = __ballot_sync(0xffffffffu, cum >= n);
      if (hit == 0u) {
        if (lane == 0) s_bstar = -1;
      } else {
        const int f = __ffs(hit) - 1;
        if (lane == f) {
          int run = cum - sum;
          int q = 0;
          for (; q < per - 1; ++q) {
            run += s_hist[kFineBins - 1 - (per * lane + q)];
            if (run >= n) break;
          }
          s_bstar = kFineBins - 1 - (per * lane + q);
        }
      }
      if (lane == 0) s_n = 0;
    }
    __syncthreads();
    const int bstar = s_bstar;
    if (bstar < 0 && tid == 0) atomicOr(P.status, kStatusInternal);
    const int bmin = max(bstar, 0);
    each([&](int x, float s) {
      if (s >= lo && fbin(s) >= bmin) {
        const int pos = atomicAdd(&s_n, 1);
        if (pos < kSelCap) skeys[pos] = cand_key(s, id_at(x));
      }
    });
    __syncthreads();
    ns = s_n;
  }
  if (ns > kSelCap) {
    // Radix select of the n-th largest key, 8 bits at a time from the top.
    if (tid == 0) {
      s_prefix = 0ull;
      s_rem = n;
    }
    __syncthreads();
    for (int shift = 56; shift >= 0; shift -= 8) {
      for (int x = tid; x < 256; x += blockDim.x) s_hist[x] = 0;
      __syncthreads();
      const unsigned long long prefix = s_prefix;
      const unsigned long long hmask = (shift == 56) ? 0ull : (~0ull << (shift + 8));
      for (int x = tid; x < cnt; x += blockDim.x) {
        const float s = sc_at(x);
        if (s < lo) continue;
        const unsigned long long key = cand_key(s, id_at(x));
        if ((key & hmask) != (prefix & hmask)) continue;
        atomicAdd(&s_hist[(key >> shift) & 255u], 1);
      }
      __syncthreads();
      if (tid == 0) {
        int acc = 0, d = 255;
        for (; d > 0; --d) {
          if (acc + s_hist[d] >= s_rem) break;
          acc += s_hist[d];
        }
        s_rem -= acc;
        s_prefix = prefix | ((unsigned long long)d << shift);
      }
      __syncthreads();
    }
    const unsigned long long kth = s_prefix;
    if (tid == 0) s_n = 0;
    __syncthreads();
    for (int x = tid; x < cnt; x += blockDim.x) {
      const float s = sc_at(x);
      if (s < lo) continue;
      const unsigned long long key = cand_key(s, id_at(x));
      if (key >= kth) {
        const int pos = atomicAdd(&s_n, 1);
        if (pos < kSelCap) skeys[pos] = key;
      }
    }
    __syncthreads();
    ns = min(s_n, kSelCap);
    if (s_n != n && tid == 0) atomicOr(P.status, kStatusInternal);
  }
  if (ns < n) {
    if (tid == 0) atomicOr(P.status, kStatusInternal);
    n = ns;
  }
  const bool bucketed =
      ns > 64 && ns <= kSelCap / 2 &&
      bucket_sort_desc<kThreads>(skeys, ns, lo, M, s_hist, s_cursor, &s_flag);
  if (!bucketed) {
    const int n2 = max(64, next_pow2(max(ns, 1)));
    for (int x = ns + tid; x < n2; x += blockDim.x) skeys[x] = 0ull;
    __syncthreads();
    if (n2 <= 2 * kThreads) {
      bitonic_desc_hybrid(skeys, n2);
    } else {
      bitonic_desc(skeys, n2);
    }
  }
  const float inv_l = 1.0f / Ls;
  for (int r = tid; r < k; r += blockDim.x) {
    if (r < n) {
      const unsigned long long key = skeys[r];
      const float s = ordered_to_float((uint32_t)(key >> 32));
      const int32_t id = (int32_t)(~(uint32_t)key);
      tok_out[r] = id;
      w_out[r] = mean ? s : fast_exp2(s - M) * inv_l;
      if (s_out) s_out[r] = s;
      // one vote for the token's unit (integer atomics: exact)
      if (id >= 0 && (uint32_t)id < kCentroidIdBase) {
        if (id / P.Tu < P.Uh) atomicAdd(&P.votes[id / P.Tu], 1);
      } else if (kGeneral && id >= 0) {
        // a centroid: its slab's count of lists that selected it (each selection is one
        // vote per member token, cast per unit by the mass kernel)
        const int e = id - (int)kCentroidIdBase, w = e / P.n_c, c = e - w * P.n_c;
        const int slab = (L / P.Hq) * P.Hkv + (L % P.Hq) / P.G;
        atomicAdd(P.csel + ((int64_t)slab * P.wcap + w) * P.n_c + c, 1);
      }
    } else {
      tok_out[r] = -1;
      w_out[r] = 0.f;
      if (s_out) s_out[r] = -INFINITY;
    }
  }
  (void)lane;
}

template <bool kGeneral, int kThreads>
cudaError_t launch_select_t(const Batch& B, int max_lists, cudaStream_t s) {
  const int smem = sel_cap<kThreads>() * (int)sizeof(unsigned long long);
  // all of the SM's unified memory as shared memory, so that two 512-thread lists fit
  cudaError_t e = ensure_smem((const void*)k_select_t<kGeneral, kThreads>, smem, 100);
  if (e != cudaSuccess) return e;
  return launch_pdl(k_select_t<kGeneral, kThreads>, dim3(max_lists, B.n), dim3(kThreads),
                    (size_t)smem, s, B);
}

cudaError_t launch_select(const Batch& B, int max_lists, int sm_count, cudaStream_t s) {
  if ((int64_t)max_lists * B.n <= sm_count) return launch_select_t<false, 1024>(B, max_lists, s);
  return launch_select_t<false, 512>(B, max_lists, s);
}

cudaError_t launch_select_general(const Batch& B, int max_lists, int sm_count, cudaStream_t s) {
  if ((int64_t)max_lists * B.n <= sm_count) return launch_select_t<true, 1024>(B, max_lists, s);
  return launch_select_t<true, 512>(B, max_lists, s);
}

// ---------------------------------------------------------------------------
// Attention mass of every history unit: over lists in a fixed order, the sum of
// 2^(m_u - M) l_u / L, i.e. the normalised weights of all the unit's tokens. A block
// covers 32 units with 32 warps: warp w sums lists w, w + 32, ..., then the 32 partial
// sums are added in warp order (deterministic).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) k_mass(const __grid_constant__ Batch B) {
  __shared__ float part[32][33];
  const int pi = blockIdx.y;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  const int n_lists = P.P * P.Hq;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if ((int)blockIdx.x * kMassUnits >= P.Uh) return;
  const int u = blockIdx.x * kMassUnits + lane;
  // The per-unit pairs of the warp's first lists are loaded before the wait for the
  // select kernel: they come from the score kernel, which completed before the select
  // kernel started (only the lists' totals come from the select kernel).
  constexpr int kPre = 4;
  float2 st0[kPre];
#pragma unroll
  for (int i = 0; i < kPre; ++i) {
    const int L = warp + 32 * i;
    st0[i] = u < P.Uh && L < n_lists ? P.ustats[(int64_t)L * P.ucap + u]
                                     : make_float2(-INFINITY, 0.f);
  }
  pdl_wait();
  pdl_release();
  if (retrieval_timed_out(P)) return;
  float acc = 0.f;
  if (u < P.Uh) {
#pragma unroll
    for (int i = 0; i < kPre; ++i) {
      const int L = warp + 32 * i;
      if (L < n_lists) {
        const float2 m = P.list_ml[L];
        if (st0[i].x != -INFINITY) acc += st0[i].y * fast_exp2(st0[i].x - m.x) / m.y;
      }
    }
#pragma unroll 4
    for (int L = warp + 32 * kPre; L < n_lists; L += 32) {
      const float2 st = P.ustats[(int64_t)L * P.ucap + u];
      const float2 m = P.list_ml[L];
      if (st.x != -INFINITY) acc += st.y * fast_exp2(st.x - m.x) / m.y;
    }
  }
  part[warp][lane] = acc;
  __syncthreads();
  if (warp == 0 && u < P.Uh) {
    float mm = 0.f;
#pragma unroll 8
    for (int w = 0; w < 32; ++w) mm += part[w][lane];
    P.mass[u] = mm;
  }
}

cudaError_t launch_mass(const Batch& B, int max_hist_units, cudaStream_t s) {
  const int blocks = (max_hist_units + kMassUnits - 1) / kMassUnits;
  if (blocks == 0) return cudaSuccess;
  return launch_pdl(k_mass, dim3(blocks, B.n), dim3(1024), 0, s, B);
}

// ---------------------------------------------------------------------------
// Vote-ranked pool: all history units sorted in shared memory by
// (votes desc, mass desc, id asc); the first pool_n are the pool.
// ---------------------------------------------------------------------------
__device__ __forceinline__ bool unit_before(unsigned long long ka, int ia,
                                            unsigned long long kb, int ib) {
  return ka > kb || (ka == kb && ia < ib);
}

constexpr int kVoteBins = 4096;
constexpr int kRankMax = 1024;   // candidates ranked by pairwise comparison

__global__ void __launch_bounds__(1024) k_pool(const __grid_constant__ Batch B) {
  extern __shared__ unsigned char smem_raw[];
  __shared__ int vh[kVoteBins];
  __shared__ int sw[32];
  __shared__ int s_v, s_c, s_vmax;
  const int tid = threadIdx.x;
  // shared-memory set-up before the wait for the previous kernel
  for (int x = tid; x < kVoteBins; x += blockDim.x) vh[x] = 0;
  if (tid == 0) {
    s_c = 0;
    s_vmax = 0;
  }
  pdl_wait();
  pdl_release();
  const Prob& P = B.p[blockIdx.x];
  if (retrieval_timed_out(P)) return;   // counts stay 0 (reset by the prep kernel)
  const int Uh = P.Uh, pn = P.pool_n;
  if (tid == 0) P.counts[0] = pn;
  if (pn == 0) return;
  // (1) histogram of votes (clipped): the pool's smallest vote level V is the highest
  //     level whose units and all better ones number at least pool_n
  // every thread's units' votes are loaded at once and kept for step (2)
  constexpr int kUnitsPerThread = kMaxHistUnits / 1024;
  int vt[kUnitsPerThread];
#pragma unroll
  for (int q = 0; q < kUnitsPerThread; ++q) {
    const int u = q * 1024 + tid;
    vt[q] = u < Uh ? P.votes[u] : -1;
  }
  __syncthreads();  // the zeroed bins
#pragma unroll
  for (int q = 0; q < kUnitsPerThread; ++q) {
    if (q * 1024 >= Uh) break;
    const int b = vt[q] >= 0 ? min(vt[q], kVoteBins - 1) : -1;
    const unsigned same = __match_any_sync(0xffffffffu, b);   // most units share a few levels
    if (b >= 0 && (__ffs(same) - 1) == (tid & 31)) atomicAdd(&vh[b], __popc(same));
  }
  __syncthreads();
  {
    constexpr int per = kVoteBins / 1024;   // 4 levels per thread, thread 0 the top ones
    int c = 0;
    for (int q = 0; q < per; ++q) c += vh[kVoteBins - 1 - (per * tid + q)];
    const int incl = block_excl_scan(c, sw) + c;
    if (incl >= pn && incl - c < pn) {
      int run = incl - c, q = 0;
      for (; q < per - 1; ++q) {
        run += vh[kVoteBins - 1 - (per * tid + q)];
        if (run >= pn) break;
      }
      s_v = kVoteBins - 1 - (per * tid + q);
    }
  }
  __syncthreads();
  const int V = s_v;
  // (2) the units at or above level V, ranked by (votes desc, mass desc, id asc)
  unsigned long long* ck = reinterpret_cast<unsigned long long*>(smem_raw);
  int* ci = reinterpret_cast<int*>(ck + kRankMax);
#pragma unroll
  for (int q = 0; q < kUnitsPerThread; ++q) {
    const int u = q * 1024 + tid;
    if (u < Uh && min(vt[q], kVoteBins - 1) >= V) {
      const int pos = atomicAdd(&s_c, 1);
      if (pos < kRankMax) {
        ck[pos] = ((unsigned long long)(uint32_t)vt[q] << 32) | __float_as_uint(P.mass[u]);
        ci[pos] = u;
        atomicMax(&s_vmax, vt[q]);
      }
    }
  }
  __syncthreads();
  const int C = s_c;
  if (C <= kRankMax) {
    // rank = the number of candidates ordered before; the block's threads split the
    // comparisons: thread t counts for candidate t % C over part t / C of the others.
    // When the votes fit 19 bits one 64-bit key orders a candidate exactly: votes, the
    // mass's bits (31: masses are sums of non-negative weights, so the sign bit is clear
    // and the bits order as the values) and 16383 - id (14 bits: ids < kMaxHistUnits),
    // so a comparison is one 64-bit compare.
    static_assert(kMaxHistUnits <= (1 << 14), "unit ids must fit 14 bits");
    const bool packed = s_vmax < (1 << 19);
    int* rk = reinterpret_cast<int*>(ci + kRankMax);
    for (int x = tid; x < C; x += blockDim.x) {
      rk[x] = 0;
      if (packed) {
        const unsigned long long v = ck[x] >> 32, mb = (uint32_t)ck[x] & 0x7fffffffu;
        ck[x] = (v << 45) | (mb << 14) | (unsigned long long)(16383 - ci[x]);
      }
    }
    __syncthreads();
    const int parts = max(1, (int)blockDim.x / max(C, 1));
    const int i = tid % max(C, 1), part = tid / max(C, 1);
    if (C > 0 && part < parts) {
      const unsigned long long mk = ck[i];
      const int mi = ci[i];
      const int o0 = (int)(((int64_t)C * part) / parts), o1 = (int)(((int64_t)C * (part + 1)) / parts);
      int r[4] = {0, 0, 0, 0};  // independent partial counts keep the loads in flight
      int o = o0;
      if (packed) {
        for (; o + 4 <= o1; o += 4) {
#pragma unroll
          for (int e = 0; e < 4; ++e) r[e] += ck[o + e] > mk ? 1 : 0;
        }
        for (; o < o1; ++o) r[0] += ck[o] > mk ? 1 : 0;
      } else {
        for (; o + 4 <= o1; o += 4) {
#pragma unroll
          for (int e = 0; e < 4; ++e) r[e] += unit_before(ck[o + e], ci[o + e], mk, mi) ? 1 : 0;
        }
        for (; o < o1; ++o) r[0] += unit_before(ck[o], ci[o], mk, mi) ? 1 : 0;
      }
      atomicAdd(&rk[i], r[0] + r[1] + r[2] + r[3]);
    }
    __syncthreads();
    for (int x = tid; x < C; x += blockDim.x)
      if (rk[x] < pn) P.pool[rk[x]] = ci[x];
    return;
  }
  // (3) too many ties at level V: sort every history unit
  const int n2 = next_pow2(max(Uh, 1));
  unsigned long long* keys = reinterpret_cast<unsigned long long*>(smem_raw);
  int* ids = reinterpret_cast<int*>(keys + n2);
  __syncthreads();
  for (int x = tid; x < n2; x += blockDim.x) {
    if (x < Uh) {
      keys[x] = ((unsigned long long)(uint32_t)P.votes[x] << 32) | __float_as_uint(P.mass[x]);
      ids[x] = x;
    } else {
      keys[x] = 0ull;
      ids[x] = 0x7fffffff;
    }
  }
  __syncthreads();
  for (int size = 2; size <= n2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int t = tid; t < (n2 >> 1); t += blockDim.x) {
        const int i = 2 * t - (t & (stride - 1));
        const int j = i + stride;
        const bool first_half = (i & size) == 0;
        const unsigned long long ki = keys[i], kj = keys[j];
        const int ii = ids[i], ij = ids[j];
        const bool swap = first_half ? unit_before(kj, ij, ki, ii) : unit_before(ki, ii, kj, ij);
        if (swap) {
          keys[i] = kj;
          keys[j] = ki;
          ids[i] = ij;
          ids[j] = ii;
        }
      }
      __syncthreads();
    }
  }
  for (int r = tid; r < pn; r += blockDim.x) P.pool[r] = ids[r];
}

cudaError_t launch_pool(const Batch& B, int max_hist_units, cudaStream_t s) {
  int n2 = 1;
  while (n2 < max_hist_units) n2 <<= 1;
  const int smem = max(n2, kRankMax) * (int)(sizeof(unsigned long long) + sizeof(int)) +
                   kRankMax * (int)sizeof(int);
  cudaError_t e = ensure_smem((const void*)k_pool, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(k_pool, dim3(B.n), dim3(1024), (size_t)smem, s, B);
}

// ---------------------------------------------------------------------------
// Max-min diversity (DivTopK): Gram matrix of the pool's descriptors, then the
// greedy rule. Start from the pool's best unit; each step adds the unselected unit
// whose smallest distance 1 - k_c . k_s to the picks is largest, ties to the better
// pool rank.
// ---------------------------------------------------------------------------
// Gram matrix of the pool's descriptors, stored as its packed upper triangle
// (row a holds G[a][a..pool)). One 16 x 16 tile of the upper triangle per CTA, rows
// staged in shared memory with a one-float pad per row.
constexpr int kGramTile = 16;

__device__ __forceinline__ int tri_off(int a, int pn) { return a * pn - (a * (a - 1)) / 2; }

// Storage of the triangle (total = pn (pn + 1) / 2 entries) in the workspace: fp32 up to
// kMaxMinSmemPool ranks (staged whole into shared memory by k_maxmin), 24-bit fixed
// point up to kMaxMinFixedPool ranks (also staged: the 16 high bits of every entry from
// the region's start, the 8 low bits from the next 16-byte boundary; 2^-22 steps, far
// below the fp32 Gram's own rounding at the distances compared), fp32 read from global
// memory beyond.
constexpr int kMaxMinSmemPool = 320;
constexpr int kMaxMinFixedPool = 384;
__host__ __device__ __forceinline__ int round16(int bytes) { return (bytes + 15) & ~15; }
__host__ __device__ __forceinline__ int tri_entries(int pn) { return pn * (pn + 1) / 2; }
__host__ __device__ __forceinline__ bool gram_fixed24(int pn) {
  return pn > kMaxMinSmemPool && pn <= kMaxMinFixedPool;
}
// bytes of the triangle that k_maxmin copies into shared memory
__host__ __device__ __forceinline__ int gram_stage_bytes(int pn) {
  if (pn <= kMaxMinSmemPool) return round16(4 * tri_entries(pn));
  if (pn <= kMaxMinFixedPool) return round16(2 * tri_entries(pn)) + round16(tri_entries(pn));
  return 0;
}
// pool ranks per lane of the greedy (its instantiation) for a pool of pn ranks
__host__ __device__ __forceinline__ int maxmin_per(int pn) {
  const int need = (pn + 31) / 32;
  if (pn <= kMaxMinSmemPool) return need <= 1 ? 1 : need <= 2 ? 2 : need <= 4 ? 4 : need <= 8 ? 8 : 16;
  if (pn <= kMaxMinFixedPool) return 12;
  return need <= 16 ? 16 : 32;
}
// Entries of the triangle's storage that the greedy reads: the row of rank b is read at
// tri_off(b) - b + c for every lane rank c >= b, so the ranks past the pool (c up to
// 32 maxmin_per - 1) reach past the triangle's end (values never used).
__host__ __device__ __forceinline__ int maxmin_reach(int pn) {
  return tri_entries(pn) - pn + 32 * maxmin_per(pn);
}
// shared-memory bytes k_maxmin needs for a pool of pn ranks: the staged triangle and
// the reads past it (fixed point: the high parts' reads past end inside the low part)
__host__ __device__ __forceinline__ int gram_smem_bytes(int pn) {
  const int t = tri_entries(pn), r = maxmin_reach(pn);
  if (pn <= kMaxMinSmemPool) return round16(4 * (r > t ? r : t));
  if (pn <= kMaxMinFixedPool) return round16(2 * t) + round16(r > t ? r : t);
  return 0;
}

__global__ void __launch_bounds__(256) k_gram(const __grid_constant__ Batch B) {
  extern __shared__ float gsm[];
  pdl_wait();
  pdl_release();
  const Prob& P = B.p[blockIdx.y];
  if (retrieval_timed_out(P)) return;
  const int pn = P.pool_n;
  const int dim = P.Hkv * kHeadDim;
  const int T = (pn + kGramTile - 1) / kGramTile;
  int ta = 0, rem = blockIdx.x;  // blockIdx.x -> tile (ta, tb), ta <= tb
  while (ta < T && rem >= T - ta) {
    rem -= T - ta;
    ++ta;
  }
  if (ta >= T) return;
  const int tb = ta + rem;
  const int ld = dim + 4;  // rows 16-byte aligned; float4 reads of 8 rows hit distinct banks
  float* A = gsm;
  float* Bm = gsm + kGramTile * ld;
  __shared__ int ua[kGramTile], ub[kGramTile];
  if (threadIdx.x < kGramTile) {
    const int a = ta * kGramTile + threadIdx.x, b = tb * kGramTile + threadIdx.x;
    ua[threadIdx.x] = a < pn ? P.pool[a] : -1;
    ub[threadIdx.x] = b < pn ? P.pool[b] : -1;
  }
  __syncthreads();
  const int d4 = dim / 4;
  // the rows' float4s, 8 + 8 per thread in flight before any is stored
  constexpr int kB = 8;
  for (int x0 = 0; x0 < kGramTile * d4; x0 += kB * blockDim.x) {
    float4 va[kB], vb[kB];
#pragma unroll
    for (int q = 0; q < kB; ++q) {
      const int x = x0 + q * blockDim.x + threadIdx.x;
      const int r = x / d4, e = 4 * (x - r * d4);
      const bool in = x < kGramTile * d4;
      va[q] = in && ua[r] >= 0 ? *reinterpret_cast<const float4*>(P.desc + (int64_t)ua[r] * dim + e)
                               : make_float4(0.f, 0.f, 0.f, 0.f);
      vb[q] = in && ub[r] >= 0 ? *reinterpret_cast<const float4*>(P.desc + (int64_t)ub[r] * dim + e)
                               : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int q = 0; q < kB; ++q) {
      const int x = x0 + q * blockDim.x + threadIdx.x;
      if (x < kGramTile * d4) {
        const int r = x / d4, e = 4 * (x - r * d4);
        *reinterpret_cast<float4*>(A + r * ld + e) = va[q];
        *reinterpret_cast<float4*>(Bm + r * ld + e) = vb[q];
      }
    }
  }
  __syncthreads();
  const int r = threadIdx.x / kGramTile, c = threadIdx.x % kGramTile;
  // four independent FMA chains (chain e takes the dimensions = e mod 4), fed by float4
  // reads (dim % 4 == 0)
  float a4[4] = {0.f, 0.f, 0.f, 0.f};
  const float4* A4 = reinterpret_cast<const float4*>(A + r * ld);
  const float4* B4 = reinterpret_cast<const float4*>(Bm + c * ld);
#pragma unroll 4
  for (int d4 = 0; d4 < dim / 4; ++d4) {
    const float4 x = A4[d4], y = B4[d4];
    a4[0] = fmaf(x.x, y.x, a4[0]);
    a4[1] = fmaf(x.y, y.y, a4[1]);
    a4[2] = fmaf(x.z, y.z, a4[2]);
    a4[3] = fmaf(x.w, y.w, a4[3]);
  }
  const float acc = (a4[0] + a4[1]) + (a4[2] + a4[3]);
  const int a = ta * kGramTile + r, b = tb * kGramTile + c;
  if (a < pn && b < pn && a <= b) {
    const int x = tri_off(a, pn) + (b - a);
    if (gram_fixed24(pn)) {
      uint8_t* g8 = reinterpret_cast<uint8_t*>(P.gram);
      const int v = __float2int_rn(fminf(fmaxf(acc, -1.99f), 1.99f) * 4194304.0f);
      reinterpret_cast<uint16_t*>(g8)[x] = (uint16_t)((uint32_t)v >> 8);
      g8[round16(2 * tri_entries(pn)) + x] = (uint8_t)((uint32_t)v & 0xffu);
    } else {
      P.gram[x] = acc;
    }
  }
}

// Greedy max-min (DivTopK) by one warp over the packed Gram triangle, then the
// expansion (Nbr of Eq. 12). Lane l owns the pool ranks l, l + 32, ...; kPer = ranks
// per lane. The triangle sits in shared memory as fp32 up to 320 ranks (201 KB), as
// 24-bit fixed point up to 384 ranks (222 KB), else in global memory.
constexpr int kMaxMinThreads = kMaxHistUnits / 32;  // one bitmap word per thread

struct TriF32 {  // fp32 triangle (shared or global memory)
  const float* p;
  __device__ __forceinline__ float operator()(int i) const { return p[i]; }
};
struct TriFix24 {  // 24-bit fixed point split into 16 high and 8 low bits
  const uint16_t* hi;
  const uint8_t* lo;
  __device__ __forceinline__ float operator()(int i) const {
    const int x = ((int)(((uint32_t)hi[i] << 16) | ((uint32_t)lo[i] << 8))) >> 8;
    return (float)x * (1.0f / 4194304.0f);
  }
};

template <int kPer, class Tri>
__device__ void greedy_maxmin(const Prob& P, const Tri pk, int* sel, int pn, int ns) {
  const int lane = threadIdx.x & 31;
  float mind[kPer];
  int toff[kPer];  // start of candidate c's row in the packed triangle
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    const int c = lane + 32 * q;
    toff[q] = tri_off(c, pn);
    mind[q] = c < pn ? 1.0f - pk(c) : -INFINITY;  // row 0 of the triangle is G[0][*]
  }
  uint32_t taken = lane == 0 ? 1u : 0u;  // bit q: rank lane + 32 q is picked
  if (lane == 0) sel[0] = 0;
  for (int step = 1; step < ns; ++step) {
    // best distance over the unpicked ranks, then the smallest rank holding it; distances
    // are >= 0 (or NaN, which ranks last), so their bit patterns order as unsigned ints
    uint32_t vv[kPer];
    int ii[kPer];
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int c = lane + 32 * q;
      const float m = mind[q];
      vv[q] = (c < pn && !((taken >> q) & 1u) && m == m)  // NaN ranks last
                  ? __float_as_uint(fmaxf(m, 0.0f)) + 1u
                  : 0u;
      ii[q] = c;
    }
    // pairwise (tree) reduction; the lower half keeps ties, i.e. the smaller rank
#pragma unroll
    for (int w = 1; w < kPer; w <<= 1) {
#pragma unroll
      for (int q = 0; q + w < kPer; q += 2 * w) {
        if (vv[q + w] > vv[q]) {
          vv[q] = vv[q + w];
          ii[q] = ii[q + w];
        }
      }
    }
    const uint32_t bv = vv[0];
    const int bi = bv ? ii[0] : 0x7fffffff;
    const uint32_t best_v = __reduce_max_sync(0xffffffffu, bv);
    const int best = (int)__reduce_min_sync(0xffffffffu, (bv == best_v && bv) ? (uint32_t)bi : 0x7fffffffu);
    if (best < 0 || best >= pn) {
      if (lane == 0) atomicOr(P.status, kStatusInternal);
      return;
    }
    if ((best & 31) == lane) taken |= 1u << (best >> 5);
    if (lane == 0) sel[step] = best;  // a pool rank; mapped to its unit afterwards
    // row best of the triangle: ranks >= best are contiguous, ranks < best sit in
    // column best of their own rows
    // all loads of the row are issued before any is used; ranks past the pool read
    // past the triangle (storage sized by maxmin_reach), their distance stays -inf
    const int rowoff = tri_off(best, pn) - best;
    float g[kPer];
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int c = lane + 32 * q;
      g[q] = pk(c >= best ? rowoff + c : toff[q] + best - c);
    }
#pragma unroll
    for (int q = 0; q < kPer; ++q) mind[q] = fminf(mind[q], 1.0f - g[q]);
  }
}

__global__ void __launch_bounds__(kMaxMinThreads) k_maxmin(const __grid_constant__ Batch B) {
  extern __shared__ float4 pks4[];
  __shared__ uint32_t bits[kMaxHistUnits / 32];
  __shared__ int spool[kMaxPool];
  __shared__ int ssel[kMaxPool];
  __shared__ __align__(8) uint64_t tri_bar;
  // the expansion's arguments, copied from the parameter block by another warp while
  // warp 0 runs the greedy (its constant-cache misses stay off the serial path)
  __shared__ int* xa_ptr[4];  // sel, exp_units, frames, counts
  __shared__ int xa_int[2];   // frames per unit, n_prev
  const Prob& P = B.p[blockIdx.x];
  const int pn = P.pool_n, ns = P.n_sel;
  const int tid = threadIdx.x, warp = tid >> 5;
  // Before the wait for the Gram kernel: the pool (written by the pool kernel, which
  // completed before the Gram kernel started) and the shared-memory set-up.
  for (int x = tid; x < pn; x += blockDim.x) spool[x] = P.pool[x];
  const int Uh = P.Uh;
  const int nwords = (Uh + 31) >> 5;
  for (int x = tid; x < nwords; x += blockDim.x) bits[x] = 0u;
  if (tid == 32) {
    xa_ptr[0] = P.sel;
    xa_ptr[1] = P.exp_units;
    xa_ptr[2] = P.frames;
    xa_ptr[3] = P.counts;
    xa_int[0] = P.fpu;
    xa_int[1] = B.n_prev;
  }
  const bool in_smem = pn <= kMaxMinSmemPool;
  const bool fixed24 = gram_fixed24(pn);
  const int hi_bytes = round16(2 * tri_entries(pn));
  const uint16_t* fhi = reinterpret_cast<const uint16_t*>(pks4);
  const uint8_t* flo = reinterpret_cast<const uint8_t*>(pks4) + hi_bytes;
  // one thread stages the triangle with bulk copies (both parts of the fixed-point form
  // lie at 16-byte boundaries; the rounded-up tails stay inside the workspace region)
  const bool staged = ns > 0 && (in_smem || fixed24);
  const uint32_t bar = smem_u32(&tri_bar);
  if (staged && tid == 0) {
    mbar_init(bar, 1u);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  pdl_wait();
  pdl_release();
  // the last kernel of a retrieval: it also copies the status word for a host caller
  auto publish_status = [&]() {
    if (P.host_status) *(volatile uint32_t*)P.host_status = *(volatile const uint32_t*)P.status;
  };
  if (retrieval_timed_out(P)) {   // no copy was issued
    if (tid == 0) publish_status();
    return;
  }
  if (staged && tid == 0) {
    const uint8_t* g8 = reinterpret_cast<const uint8_t*>(P.gram);
    mbar_expect_tx(bar, (uint32_t)gram_stage_bytes(pn));
    if (in_smem) {
      bulk_load(smem_u32(pks4), g8, (uint32_t)round16(4 * tri_entries(pn)), bar);
    } else {
      bulk_load(smem_u32(pks4), g8, (uint32_t)hi_bytes, bar);
      bulk_load(smem_u32(flo), g8 + hi_bytes, (uint32_t)round16(tri_entries(pn)), bar);
    }
  }
  __syncthreads();
  // One warp does the rest: warps parked at a barrier would slow its serial greedy.
  if (warp != 0) return;
  const int lane = tid;
  if (staged && !mbar_wait_bounded(bar, 0u)) {
    // report, then let the copies in flight land before the CTA exits
    if (lane == 0) {
      atomicOr(P.status, kStatusTimeout);
      __threadfence();
      publish_status();
    }
    mbar_wait_bounded(bar, 0u);
    return;
  }
  if (ns > 0) {
    // separate call sites keep the triangle's address space (shared or global) known
    // to the compiler, so the greedy's reads are plain shared-memory loads when staged
    const int per = maxmin_per(pn);
    if (in_smem) {
      const TriF32 sk{reinterpret_cast<const float*>(pks4)};
      if (per <= 1) greedy_maxmin<1>(P, sk, ssel, pn, ns);
      else if (per <= 2) greedy_maxmin<2>(P, sk, ssel, pn, ns);
      else if (per <= 4) greedy_maxmin<4>(P, sk, ssel, pn, ns);
      else if (per <= 8) greedy_maxmin<8>(P, sk, ssel, pn, ns);
      else greedy_maxmin<16>(P, sk, ssel, pn, ns);   // pool <= 320 here
    } else if (fixed24) {
      greedy_maxmin<12>(P, TriFix24{fhi, flo}, ssel, pn, ns);   // 320 < pool <= 384
    } else {
      const TriF32 gk{P.gram};
      if (per <= 16) greedy_maxmin<16>(P, gk, ssel, pn, ns);
      else greedy_maxmin<32>(P, gk, ssel, pn, ns);
    }
  }
  __syncwarp();
  int* const sel_out = xa_ptr[0];
  int* const exp_out = xa_ptr[1];
  int* const frames_out = xa_ptr[2];
  const int fpu = xa_int[0], n_prev = xa_int[1];
  // the picks' units, then the expansion: each pick and its n_prev predecessors,
  // deduplicated, ascending
  for (int r = lane; r < ns; r += 32) {
    const int rk = ssel[r];  // left unset past a failed step (status already raised)
    const int u = rk >= 0 && rk < pn ? spool[rk] : -1;
    sel_out[r] = u;
    for (int j = 0; j <= n_prev; ++j) {
      const int v = u - j;
      if (v >= 0 && v < Uh) atomicOr(&bits[v >> 5], 1u << (v & 31));
    }
  }
  __syncwarp();
  // lane l compacts the words [l * wpl, (l + 1) * wpl) in order
  const int wpl = (nwords + 31) / 32;
  const int x0 = min(nwords, lane * wpl), x1 = min(nwords, x0 + wpl);
  int c = 0;
  for (int x = x0; x < x1; ++x) c += __popc(bits[x]);
  int incl = c;
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += y;
  }
  int q = incl - c;
  for (int x = x0; x < x1; ++x) {
    uint32_t rest = bits[x];
    while (rest) {
      const int u = x * 32 + __ffs(rest) - 1;
      rest &= rest - 1u;
      exp_out[q] = u;
      for (int f = 0; f < fpu; ++f) frames_out[q * fpu + f] = u * fpu + f;
      ++q;
    }
  }
  if (lane == 31) {
    int* const counts = xa_ptr[3];
    counts[1] = ns;
    counts[2] = incl;
    counts[3] = incl * fpu;
  }
  __syncwarp();
  if (lane == 0) {
    __threadfence();
    publish_status();
  }
}

cudaError_t launch_maxmin(const Batch& B, int max_pool, cudaStream_t s) {
  int max_dim = 0;
  for (int j = 0; j < B.n; ++j) max_dim = max(max_dim, B.p[j].Hkv * kHeadDim);
  if (max_pool > 0) {
    const int T = (max_pool + kGramTile - 1) / kGramTile;
    const int smem = 2 * kGramTile * (max_dim + 4) * (int)sizeof(float);
    cudaError_t e = ensure_smem((const void*)k_gram, smem);
    if (e != cudaSuccess) return e;
    dim3 grid(T * (T + 1) / 2, B.n);
    e = launch_pdl(k_gram, grid, dim3(kGramTile * kGramTile), (size_t)smem, s, B);
    if (e != cudaSuccess) return e;
  }
  // the largest staged triangle of any problem of the batch (the two forms' sizes are
  // not monotonic across the switch to fixed point)
  int smem = 16;
  for (int j = 0; j < B.n; ++j) smem = max(smem, gram_smem_bytes(B.p[j].pool_n));
  cudaError_t e = ensure_smem((const void*)k_maxmin, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(k_maxmin, dim3(B.n), dim3(kMaxMinThreads), (size_t)smem, s, B);
}

}  // namespace ss
