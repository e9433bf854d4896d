// The paper's long-history compression of the shallow index (Sec. 4.1, Eq. 5-7) and the
// cluster evidence of a question (Sec. 4.2, Eq. 13).
//
//   k_uc_assign  units leaving the detailed window, oldest first (one CTA, one thread
//                per descriptor entry): a unit joins the latest cluster when its
//                descriptor's dot product with the cluster's centroid reaches tau, and
//                the centroid becomes Norm((n c + k) / (n + 1)); otherwise it starts the
//                next cluster (Eq. 6). Reductions in a fixed order.
//   k_uc_reps    the representative keys of every cluster the call touched: the running
//                average (n K + K_t) / (n + 1) of its members' keys at each (layer, key
//                head, token slot, dim), members in order (Eq. 7), fp32.
//   k_uc_scores  Eq. 13: score_j = (1/Hq) sum_h q_h . c_j[g(h)] / sqrt(d) against the query
//                state of the last shallow layer.
//   k_uc_top     the top K_l clusters by (score desc, id asc).
// Clustered units are a prefix of the unit sequence; retrieval scores the detailed units
// after it (the index view is offset; k_uc_shift moves the outputs back to stream
// numbering).
#include "ss_internal.cuh"
#include "ss_device.cuh"

namespace ss {

// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) k_uc_assign(UcJob J) {
  __shared__ float sm[32];
  __shared__ int s_stop;
  const int e = threadIdx.x;             // descriptor entry (blockDim.x = D)
  const int D = J.D;
  int cur = *J.n_clusters - 1;           // the latest cluster (continued from earlier calls)
  float c = 0.f;
  int n = 0;
  if (cur >= 0) {
    c = J.cdesc[(int64_t)cur * D + e];
    n = J.ccount[cur];
  }
  const int n0 = n;                      // the continued cluster's members before this call
  if (e == 0) s_stop = 0;
  const int cur0 = cur;
  __syncthreads();
  for (int t = J.u0; t < J.u0 + J.n; ++t) {
    const float k = J.desc[(int64_t)t * D + e];
    bool join = false;
    if (cur >= 0) join = block_sum(k * c, sm) >= J.tau;
    if (join) {
      const float v = ((float)n * c + k) / (float)(n + 1);
      const float nrm2 = block_sum(v * v, sm);
      c = nrm2 > 0.f ? v / sqrtf(nrm2) : 0.f;
      ++n;
    } else {
      if (cur >= 0) {                    // the finished cluster
        J.cdesc[(int64_t)cur * D + e] = c;
        if (e == 0) J.ccount[cur] = n;
      }
      if (cur + 1 >= J.cap) {
        if (e == 0) {
          s_stop = 1;
          atomicOr(J.status, kStatusInternal);   // more clusters than the capacity
        }
        __syncthreads();
        break;
      }
      ++cur;
      c = k;
      n = 1;
      if (e == 0) {
        J.cfirst[cur] = t;               // its first member in this call
        J.cprev[cur] = 0;                // members before this call
      }
    }
    if (e == 0) J.unit_cluster[t] = cur;
  }
  if (cur >= 0 && !s_stop) {
    J.cdesc[(int64_t)cur * D + e] = c;
    if (e == 0) J.ccount[cur] = n;
  }
  if (e == 0) {
    // the continued cluster's members before this call, and its first member now
    if (cur0 >= 0) {
      J.cprev[cur0] = n0;
      J.cfirst[cur0] = J.u0;
    }
    *J.n_clusters = cur + 1;
    *J.first_touched = cur0 >= 0 ? cur0 : 0;
  }
}

// ---------------------------------------------------------------------------
// Grid (element blocks, touched-cluster slot): cluster j = first_touched + slot. Each
// thread owns one (slab, token slot, dim) element of the representative and folds the
// cluster's members of this call into it in unit order.
__global__ void __launch_bounds__(256) k_uc_reps(UcJob J) {
  const int j = *J.first_touched + (int)blockIdx.y;
  if (j >= *J.n_clusters) return;
  const int64_t per = (int64_t)J.n_slabs * J.Tu * kHeadDim;
  const int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (x >= per) return;
  const int slab = (int)(x / ((int64_t)J.Tu * kHeadDim));
  const int64_t rem = x - (int64_t)slab * J.Tu * kHeadDim;   // token slot * d + dim
  float* rep = J.creps + (int64_t)j * per + x;
  int n = J.cprev[j];
  float v = n > 0 ? *rep : 0.f;
  const __nv_bfloat16* kp = J.keys + (int64_t)slab * J.ncap * kHeadDim + rem;
  for (int t = J.cfirst[j]; t < J.u0 + J.n && J.unit_cluster[t] == j; ++t) {
    const float k = __bfloat162float(kp[(int64_t)t * J.Tu * kHeadDim]);
    v = ((float)n * v + k) / (float)(n + 1);
    ++n;
  }
  *rep = v;
}

// ---------------------------------------------------------------------------
// Eq. 13 scores; the query state of the last layer is its last question row, or the
// rows' mean (fp32 in row order, rounded to bf16) for the other readings.
__global__ void __launch_bounds__(256) k_uc_scores(UcSel S) {
  __shared__ float qs[kMaxGroup * 8][kHeadDim];   // up to 64 query heads
  const int i = S.P - 1;
  const int64_t row_stride = (int64_t)S.Hq * kHeadDim;
  for (int x = threadIdx.x; x < S.Hq * kHeadDim; x += blockDim.x) {
    const int h = x / kHeadDim, d = x - h * kHeadDim;
    const __nv_bfloat16* q0 = S.q + (int64_t)i * S.R * row_stride + (int64_t)h * kHeadDim + d;
    float v;
    if (S.q_agg == 0) {
      v = __bfloat162float(q0[(int64_t)(S.R - 1) * row_stride]);
    } else {
      float acc = 0.f;
      for (int r = 0; r < S.R; ++r) acc = __fadd_rn(acc, __bfloat162float(q0[(int64_t)r * row_stride]));
      v = __fdiv_rn(acc, (float)S.R);
    }
    qs[h][d] = __bfloat162float(__float2bfloat16_rn(v));
  }
  __syncthreads();
  const int n_c = *S.n_clusters;
  const int G = S.Hq / S.Hkv;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // one warp per cluster: lane l takes dims l, l + 32, ... of every head
  for (int j = blockIdx.x * 8 + warp; j < n_c; j += gridDim.x * 8) {
    const float* c = S.cdesc + (int64_t)j * S.Hkv * kHeadDim;
    float acc = 0.f;
    for (int h = 0; h < S.Hq; ++h) {
      const float* cg = c + (h / G) * kHeadDim;
#pragma unroll
      for (int d = lane; d < kHeadDim; d += 32) acc = fmaf(qs[h][d], cg[d], acc);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    if (lane == 0) S.work[j] = acc / (sqrtf((float)kHeadDim) * (float)S.Hq);
  }
}

// The top K_l clusters: 64-bit keys (ordered score, then id) sorted in shared memory.
__global__ void __launch_bounds__(1024) k_uc_top(UcSel S) {
  extern __shared__ unsigned long long keys[];
  const int n_c = *S.n_clusters;
  int n2 = 1;
  while (n2 < n_c) n2 <<= 1;
  for (int x = threadIdx.x; x < n2; x += blockDim.x) {
    unsigned long long kk = 0ull;        // padding sorts last
    if (x < n_c)
      kk = ((unsigned long long)float_to_ordered(S.work[x]) << 32) | (uint32_t)(~(uint32_t)x);
    keys[x] = kk;
  }
  __syncthreads();
  // bitonic sort, descending
  for (int size = 2; size <= n2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int x = threadIdx.x; x < n2; x += blockDim.x) {
        const int y = x ^ stride;
        if (y > x) {
          const bool desc = (x & size) == 0;
          const unsigned long long a = keys[x], b = keys[y];
          if ((a < b) == desc) {
            keys[x] = b;
            keys[y] = a;
          }
        }
      }
      __syncthreads();
    }
  }
  const int m = n_c < S.k_l ? n_c : S.k_l;
  for (int r = threadIdx.x; r < S.k_l; r += blockDim.x) {
    if (r < m) {
      const unsigned long long kk = keys[r];
      S.ids[r] = (int32_t)(~(uint32_t)kk);
      S.scores[r] = ordered_to_float((uint32_t)(kk >> 32));
    } else {
      S.ids[r] = -1;
      S.scores[r] = -INFINITY;
    }
  }
  if (threadIdx.x == 0) *S.count = m;
}

// ---------------------------------------------------------------------------
// After a retrieval over the detailed units of an index with clustered units: token ids,
// pool, selection, expansion and frames back to stream numbering; the clustered units'
// votes and mass are 0.
__global__ void __launch_bounds__(256) k_uc_shift(const __grid_constant__ Batch B) {
  pdl_wait();
  pdl_release();
  const Prob& P = B.p[blockIdx.y];
  const int off = P.unit_offset;
  if (off <= 0) return;
  const int n_lists = (B.head_agg == 1) ? P.P : P.P * P.Hq;
  const int64_t tok_off = (int64_t)off * P.Tu;
  const int64_t nt = (int64_t)n_lists * B.k;
  const int stride = gridDim.x * blockDim.x;
  const int x0 = blockIdx.x * blockDim.x + threadIdx.x;
  for (int64_t x = x0; x < nt; x += stride)
    if (P.topk_tok[x] >= 0) P.topk_tok[x] = (int32_t)(P.topk_tok[x] + tok_off);
  for (int x = x0; x < off; x += stride) {
    P.votes_base[x] = 0;
    P.mass_base[x] = 0.f;
  }
  if (x0 == 0) {
    const int n_pool = P.counts[0], n_sel = P.counts[1], n_exp = P.counts[2], n_fr = P.counts[3];
    for (int r = 0; r < n_pool; ++r) P.pool[r] += off;
    for (int r = 0; r < n_sel; ++r) P.sel[r] += off;
    for (int r = 0; r < n_exp; ++r) P.exp_units[r] += off;
    for (int r = 0; r < n_fr; ++r) P.frames[r] += off * P.fpu;
  }
}

cudaError_t launch_uc_shift(const Batch& B, cudaStream_t s) {
  return launch_pdl(k_uc_shift, dim3(64, B.n), dim3(256), 0, s, B);
}

cudaError_t launch_uc_cluster(const UcJob& J, cudaStream_t s) {
  k_uc_assign<<<1, J.D, 0, s>>>(J);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t per = (int64_t)J.n_slabs * J.Tu * kHeadDim;
  // one slot per cluster the call can touch: the continued one and one per unit
  k_uc_reps<<<dim3((unsigned)((per + 255) / 256), (unsigned)(J.n + 1)), 256, 0, s>>>(J);
  return cudaGetLastError();
}

cudaError_t launch_uc_select(const UcSel& S, int cap, cudaStream_t s) {
  k_uc_scores<<<152, 256, 0, s>>>(S);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  int n2 = 1;
  while (n2 < cap) n2 <<= 1;
  const size_t smem = (size_t)n2 * 8;
  e = ensure_smem((const void*)k_uc_top, (int)smem);
  if (e != cudaSuccess) return e;
  k_uc_top<<<1, 1024, smem, s>>>(S);
  return cudaGetLastError();
}

}  // namespace ss
