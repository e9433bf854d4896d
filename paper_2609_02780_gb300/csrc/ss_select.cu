// Evidence selection after key scoring (Sec. 4.2, Eq. 11-12):
//   k_select    exact top-k of every list from its candidate array, softmax
//               statistics from the per-unit (max, sum) pairs, normalised weights
//   k_votes_mass unit votes (one per (list, selected token) in the unit) and the
//               attention mass of every history unit (summed weights of all tokens)
//   k_pool      the vote-ranked pool: top min(pool_mult * K, |H|) units by
//               (votes desc, mass desc, unit id asc)
//   k_gram / k_maxmin  greedy max-min diversity over the pool's descriptors
//   k_expand    each pick plus its preceding units, deduplicated, ascending (Eq. 12)
// No floating-point atomics: every float reduction has a fixed order, so results are
// bit-identical from run to run.
#include "ss_internal.cuh"

namespace ss {

constexpr int kSelThreads = 1024;
constexpr int kSelCap = 16384;   // survivors sorted in shared memory
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

__device__ __forceinline__ int next_pow2(int x) {
  int p = 1;
  while (p < x) p <<= 1;
  return p;
}

// Block reduction of (max, sum 2^(s - max)) pairs in a fixed order; result to all.
__device__ void block_ml(float& m, float& l, float* sm, float* sl) {
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

__device__ float block_min(float v, float* sm) {
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

// ---------------------------------------------------------------------------
// Exact top-k of one list (Eq. 11). The candidate array holds every token whose score
// reached a lower bound `lo` of the list's k-th best score. A 2048-bin histogram of
// the candidates over [lo, max] locates the bin of the n-th best (n = min(k, tokens));
// the candidates from that bin up are sorted in shared memory by (score desc, id asc).
// If they do not fit (massive ties), an 8-pass radix select on the 64-bit keys over
// the candidate array finds the n-th key exactly.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kSelThreads) k_select(const __grid_constant__ Batch B) {
  extern __shared__ unsigned long long skeys[];
  __shared__ int s_hist[kFineBins];
  __shared__ float s_m[32], s_l[32];
  __shared__ int s_n, s_bstar, s_rem;
  __shared__ unsigned long long s_prefix;

  const int pi = blockIdx.y;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  const int n_lists = P.P * P.Hq;
  const int L = blockIdx.x;
  if (L >= n_lists) return;
  const int tid = threadIdx.x, lane = tid & 31;
  const int k = B.k;

  float M = -INFINITY, Ls = 0.f;
  const float2* us = P.ustats + (int64_t)L * P.ucap;
  for (int u = tid; u < P.Uh; u += blockDim.x) {
    const float2 v = us[u];
    ml_combine(M, Ls, v.x, v.y);
  }
  block_ml(M, Ls, s_m, s_l);
  if (tid == 0) P.list_ml[L] = make_float2(M, Ls);

  int32_t* tok_out = P.topk_tok + (int64_t)L * k;
  float* w_out = P.topk_w + (int64_t)L * k;
  const int64_t n_tok = (int64_t)P.Uh * P.Tu;
  int n = (int)min((int64_t)k, n_tok);
  if (n == 0) {
    for (int r = tid; r < k; r += blockDim.x) {
      tok_out[r] = -1;
      w_out[r] = 0.f;
    }
    return;
  }
  const int cnt = P.cand_cnt[L];
  const float* cs = P.cand_s + (int64_t)L * P.cand_cap;
  const int32_t* ci = P.cand_id + (int64_t)L * P.cand_cap;
  float lo = ordered_to_float(P.gthr[L]);
  if (lo == -INFINITY) {
    // no threshold was established: start from the smallest real candidate (unused
    // reserved slots hold -inf and are never candidates)
    float mn = INFINITY;
    for (int x = tid; x < cnt; x += blockDim.x) {
      const float s = cs[x];
      if (s > -INFINITY) mn = fminf(mn, s);
    }
    lo = block_min(mn, s_m);
  }
  const float hi = M;
  const float scale = (hi > lo) ? (float)kFineBins / (hi - lo) : 0.f;
  auto fbin = [&](float s) -> int {
    const int b = (int)((s - lo) * scale);
    return min(max(b, 0), kFineBins - 1);
  };

  for (int x = tid; x < kFineBins; x += blockDim.x) s_hist[x] = 0;
  __syncthreads();
  for (int x = tid; x < cnt; x += blockDim.x) {
    const float s = cs[x];
    if (s >= lo) atomicAdd(&s_hist[fbin(s)], 1);
  }
  __syncthreads();
  if (tid < 32) {
    // lane 0 holds the top 64 bins, lane 31 the bottom 64
    constexpr int per = kFineBins / 32;
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
  if (bstar < 0) {
    // fewer candidates than n: the lower bound was not one (must not happen)
    if (tid == 0) atomicOr(P.status, kStatusInternal);
  }
  const int bmin = max(bstar, 0);
  for (int x = tid; x < cnt; x += blockDim.x) {
    const float s = cs[x];
    if (s >= lo && fbin(s) >= bmin) {
      const int pos = atomicAdd(&s_n, 1);
      if (pos < kSelCap) skeys[pos] = cand_key(s, ci[x]);
    }
  }
  __syncthreads();
  int ns = s_n;
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
        const float s = cs[x];
        if (s < lo) continue;
        const unsigned long long key = cand_key(s, ci[x]);
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
      const float s = cs[x];
      if (s < lo) continue;
      const unsigned long long key = cand_key(s, ci[x]);
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
  const int n2 = next_pow2(max(ns, 1));
  for (int x = ns + tid; x < n2; x += blockDim.x) skeys[x] = 0ull;
  __syncthreads();
  bitonic_desc(skeys, n2);
  const float inv_l = 1.0f / Ls;
  for (int r = tid; r < k; r += blockDim.x) {
    if (r < n) {
      const unsigned long long key = skeys[r];
      const float s = ordered_to_float((uint32_t)(key >> 32));
      tok_out[r] = (int32_t)(~(uint32_t)key);
      w_out[r] = fast_exp2(s - M) * inv_l;
    } else {
      tok_out[r] = -1;
      w_out[r] = 0.f;
    }
  }
  (void)lane;
}

cudaError_t launch_select(const Batch& B, int max_lists, cudaStream_t s) {
  const int smem = kSelCap * (int)sizeof(unsigned long long);
  cudaError_t e = cudaFuncSetAttribute(k_select, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  dim3 grid(max_lists, B.n);
  k_select<<<grid, kSelThreads, smem, s>>>(B);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Unit votes (v_t of Sec. 4.2) and attention mass. Integer atomics only (exact);
// the mass of unit u sums, over lists in order, 2^(m_u - M) l_u / L, i.e. the
// normalised weights of all the unit's tokens.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_votes_mass(const __grid_constant__ Batch B,
                                                    int vote_blocks) {
  const int pi = blockIdx.y;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  const int n_lists = P.P * P.Hq;
  if ((int)blockIdx.x < vote_blocks) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e < (int64_t)n_lists * B.k) {
      const int32_t tok = P.topk_tok[e];
      if (tok >= 0 && tok / P.Tu < P.Uh) atomicAdd(&P.votes[tok / P.Tu], 1);
    }
    return;
  }
  const int u = (blockIdx.x - vote_blocks) * blockDim.x + threadIdx.x;
  if (u >= P.Uh) return;
  float acc = 0.f;
  for (int L = 0; L < n_lists; ++L) {
    const float2 st = P.ustats[(int64_t)L * P.ucap + u];
    const float2 ml = P.list_ml[L];
    if (st.x != -INFINITY) acc += st.y * fast_exp2(st.x - ml.x) / ml.y;
  }
  P.mass[u] = acc;
}

cudaError_t launch_votes_mass(const Batch& B, int max_lists, int max_hist_units,
                              cudaStream_t s) {
  const int vote_blocks = (int)(((int64_t)max_lists * B.k + 255) / 256);
  const int mass_blocks = (max_hist_units + 255) / 256;
  if (vote_blocks + mass_blocks == 0) return cudaSuccess;
  dim3 grid(vote_blocks + mass_blocks, B.n);
  k_votes_mass<<<grid, 256, 0, s>>>(B, vote_blocks);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Vote-ranked pool: all history units sorted in shared memory by
// (votes desc, mass desc, id asc); the first pool_n are the pool.
// ---------------------------------------------------------------------------
__device__ __forceinline__ bool unit_before(unsigned long long ka, int ia,
                                            unsigned long long kb, int ib) {
  return ka > kb || (ka == kb && ia < ib);
}

__global__ void __launch_bounds__(1024) k_pool(const __grid_constant__ Batch B) {
  extern __shared__ unsigned char smem_raw[];
  const Prob& P = B.p[blockIdx.x];
  const int Uh = P.Uh;
  const int n2 = next_pow2(max(Uh, 1));
  unsigned long long* keys = reinterpret_cast<unsigned long long*>(smem_raw);
  int* ids = reinterpret_cast<int*>(keys + n2);
  for (int x = threadIdx.x; x < n2; x += blockDim.x) {
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
      for (int t = threadIdx.x; t < (n2 >> 1); t += blockDim.x) {
        const int i = 2 * t - (t & (stride - 1));
        const int j = i + stride;
        const bool first_half = (i & size) == 0;
        const unsigned long long ki = keys[i], kj = keys[j];
        const int ii = ids[i], ij = ids[j];
        // first_half: entry i must come before j in the final order
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
  for (int r = threadIdx.x; r < P.pool_n; r += blockDim.x) P.pool[r] = ids[r];
  if (threadIdx.x == 0) P.counts[0] = P.pool_n;
}

cudaError_t launch_pool(const Batch& B, int max_hist_units, cudaStream_t s) {
  int n2 = 1;
  while (n2 < max_hist_units) n2 <<= 1;
  const int smem = n2 * (int)(sizeof(unsigned long long) + sizeof(int));
  cudaError_t e = cudaFuncSetAttribute(k_pool, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  k_pool<<<B.n, 1024, smem, s>>>(B);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Max-min diversity (DivTopK): Gram matrix of the pool's descriptors, then the
// greedy rule. Start from the pool's best unit; each step adds the unselected unit
// whose smallest distance 1 - k_c . k_s to the picks is largest, ties to the better
// pool rank.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_gram(const __grid_constant__ Batch B) {
  const Prob& P = B.p[blockIdx.z];
  const int pn = P.pool_n;
  const int dim = P.Hkv * kHeadDim;
  const int a0 = blockIdx.y * 32, b0 = blockIdx.x * 32;
  if (a0 >= pn || b0 >= pn) return;
  __shared__ float As[32][33], Bs[32][33];
  __shared__ int pa[32], pb[32];
  const int tx = threadIdx.x, ty = threadIdx.y;
  if (ty == 0) {
    pa[tx] = (a0 + tx < pn) ? P.pool[a0 + tx] : -1;
    pb[tx] = (b0 + tx < pn) ? P.pool[b0 + tx] : -1;
  }
  __syncthreads();
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int d0 = 0; d0 < dim; d0 += 32) {
    for (int r = ty; r < 32; r += 8) {
      As[r][tx] = pa[r] >= 0 ? P.desc[(int64_t)pa[r] * dim + d0 + tx] : 0.f;
      Bs[r][tx] = pb[r] >= 0 ? P.desc[(int64_t)pb[r] * dim + d0 + tx] : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int dd = 0; dd < 32; ++dd) {
      const float bv = Bs[tx][dd];
#pragma unroll
      for (int q = 0; q < 4; ++q) acc[q] = fmaf(As[ty + 8 * q][dd], bv, acc[q]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int a = a0 + ty + 8 * q, bcol = b0 + tx;
    if (a < pn && bcol < pn) P.gram[(int64_t)a * pn + bcol] = acc[q];
  }
}

__global__ void __launch_bounds__(1024) k_maxmin(const __grid_constant__ Batch B) {
  __shared__ float wv[32];
  __shared__ int wi[32];
  __shared__ int s_best;
  const Prob& P = B.p[blockIdx.x];
  const int pn = P.pool_n, ns = P.n_sel;
  const int r = threadIdx.x, lane = r & 31, warp = r >> 5;
  const int nw = blockDim.x >> 5;
  const bool act = r < pn;
  float mind = act ? 1.0f - P.gram[r] : -INFINITY;
  bool taken = (r == 0);
  if (r == 0 && ns > 0) P.sel[0] = P.pool[0];
  for (int step = 1; step < ns; ++step) {
    float v = -INFINITY;
    int idx = 0x7fffffff;
    if (act && !taken) {
      v = (mind == mind) ? mind : -3.0e38f;  // NaN descriptors rank last
      idx = r;
    }
    for (int off = 16; off > 0; off >>= 1) {
      const float vo = __shfl_down_sync(0xffffffffu, v, off);
      const int io = __shfl_down_sync(0xffffffffu, idx, off);
      if (vo > v || (vo == v && io < idx)) {
        v = vo;
        idx = io;
      }
    }
    if (lane == 0) {
      wv[warp] = v;
      wi[warp] = idx;
    }
    __syncthreads();
    if (warp == 0) {
      v = lane < nw ? wv[lane] : -INFINITY;
      idx = lane < nw ? wi[lane] : 0x7fffffff;
      for (int off = 16; off > 0; off >>= 1) {
        const float vo = __shfl_down_sync(0xffffffffu, v, off);
        const int io = __shfl_down_sync(0xffffffffu, idx, off);
        if (vo > v || (vo == v && io < idx)) {
          v = vo;
          idx = io;
        }
      }
      if (lane == 0) s_best = idx;
    }
    __syncthreads();
    const int best = s_best;
    if (best < 0 || best >= pn) {
      if (r == 0) atomicOr(P.status, kStatusInternal);
      break;
    }
    if (r == best) taken = true;
    if (r == 0) P.sel[step] = P.pool[best];
    if (act) mind = fminf(mind, 1.0f - P.gram[(int64_t)best * pn + r]);
  }
}

cudaError_t launch_maxmin(const Batch& B, int max_pool, cudaStream_t s) {
  if (max_pool > 0) {
    const int tiles = (max_pool + 31) / 32;
    dim3 grid(tiles, tiles, B.n);
    k_gram<<<grid, dim3(32, 8), 0, s>>>(B);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  k_maxmin<<<B.n, 1024, 0, s>>>(B);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Temporal expansion (Nbr of Eq. 12) with deduplication and temporal ordering: a
// bitmap over history units marks every pick and its n_prev predecessors; an ordered
// compaction lists the marked units ascending and their frames.
// ---------------------------------------------------------------------------
__device__ int block_excl_scan(int v, int* sw) {
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

__global__ void __launch_bounds__(1024) k_expand(const __grid_constant__ Batch B) {
  __shared__ uint32_t bits[kMaxHistUnits / 32];
  __shared__ int sw[32];
  const Prob& P = B.p[blockIdx.x];
  const int Uh = P.Uh;
  const int nwords = (Uh + 31) >> 5;
  for (int x = threadIdx.x; x < nwords; x += blockDim.x) bits[x] = 0u;
  __syncthreads();
  for (int r = threadIdx.x; r < P.n_sel; r += blockDim.x) {
    const int u = P.sel[r];
    for (int j = 0; j <= B.n_prev; ++j) {
      const int v = u - j;
      if (v >= 0 && v < Uh) atomicOr(&bits[v >> 5], 1u << (v & 31));
    }
  }
  __syncthreads();
  const int w = threadIdx.x;
  const uint32_t word = (w < nwords) ? bits[w] : 0u;
  const int c = __popc(word);
  const int off = block_excl_scan(c, sw);
  uint32_t rest = word;
  int q = off;
  while (rest) {
    const int bpos = __ffs(rest) - 1;
    rest &= rest - 1u;
    const int u = w * 32 + bpos;
    P.exp_units[q] = u;
    for (int f = 0; f < P.fpu; ++f) P.frames[q * P.fpu + f] = u * P.fpu + f;
    ++q;
  }
  if (threadIdx.x == blockDim.x - 1) {
    const int total = off + c;
    P.counts[1] = P.n_sel;
    P.counts[2] = total;
    P.counts[3] = total * P.fpu;
  }
}

cudaError_t launch_expand(const Batch& B, cudaStream_t s) {
  k_expand<<<B.n, 1024, 0, s>>>(B);
  return cudaGetLastError();
}

}  // namespace ss
