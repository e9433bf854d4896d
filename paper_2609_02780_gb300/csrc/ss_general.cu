// The general retrieval path: lists that need every candidate's score.
//
//   * One list per layer (Sec. 4.2, "average over attention heads"): the weight of token
//     p in layer i is alpha_{i,p} = (1/Hq) sum_h w_{i,h,p}, where w_{i,h,.} is head h's
//     softmax over the history (Eq. 11 then ranks tokens by alpha). Every head's
//     normaliser must be known before any alpha, so the scores of all tokens are kept.
//   * Compressed windows (the cluster-compressed index): a compressed window contributes
//     its centroids as candidates instead of its tokens; the softmax runs over the raw
//     tokens of the uncovered history units and the centroids together. A selected
//     centroid votes once per member token (for the member's unit) and its weight is
//     shared among the window's units by member count.
//
// Kernels (after the query preparation of the default path):
//   k_cluster_map  ranks the history units that no window covers (candidate order)
//   k_dense        scores every candidate of every list into a dense row (tensor cores)
//   k_head_stats   per-head softmax statistics (one list per layer only)
//   k_alpha        head-averaged weights of every token (one list per layer only)
//   k_centroid_weight  each centroid's weight summed over its slab's lists
//   k_mass_general attention mass of every history unit from the dense rows
// The top-k of a dense row is k_select's general variant (ss_select.cu).
#include "ss_internal.cuh"
#include "ss_device.cuh"

namespace ss {

constexpr int kDenseWarps = 8;

// ---------------------------------------------------------------------------
// Raw history units (those no compressed window covers), ascending: raw_units[r] and
// raw_rank[u] = r (or -1). One block per problem.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) k_cluster_map(const __grid_constant__ Batch B) {
  __shared__ int sw[32];
  pdl_wait();
  pdl_release();
  const int pi = blockIdx.y;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  const int Uh = P.Uh, tid = threadIdx.x;
  const int per = (Uh + blockDim.x - 1) / blockDim.x;
  const int u0 = min(Uh, tid * per), u1 = min(Uh, u0 + per);
  int c = 0;
  for (int u = u0; u < u1; ++u) c += P.win_slot[u / P.wu] < 0;
  int r = block_excl_scan(c, sw);
  for (int u = u0; u < u1; ++u) {
    if (P.win_slot[u / P.wu] < 0) {
      P.raw_units[r] = u;
      P.raw_rank[u] = r++;
    } else {
      P.raw_rank[u] = -1;
    }
  }
}

// Key row and candidate id of candidate j of a slab's lists.
__device__ __forceinline__ const __nv_bfloat16* candidate_row(const Prob& P, bool clusters,
                                                             int slab, int j, int& id) {
  if (!clusters || j < P.n_raw_tok) {
    int tok = j;
    if (clusters) {
      const int ru = j / P.Tu;
      tok = P.raw_units[ru] * P.Tu + (j - ru * P.Tu);
    }
    id = tok;
    return P.keys + ((int64_t)slab * P.ncap + tok) * kHeadDim;
  }
  const int e = j - P.n_raw_tok;  // window w = e / n_c, centroid c = e % n_c
  id = (int)kCentroidIdBase + e;
  return P.cent + ((int64_t)slab * P.wcap * P.n_c + e) * kHeadDim;
}

// ---------------------------------------------------------------------------
// Dense scores: s = q_eff[i][h] . row * log2(e) / sqrt(d) for every candidate of every
// list of the slab (the G query heads of key head g), on the tensor cores with the
// default path's fragment layout. Grid (x, slab, problem); each warp takes 16-row tiles.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kDenseWarps * 32) k_dense(const __grid_constant__ Batch B) {
  pdl_wait();
  pdl_release();
  const int pi = blockIdx.z;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  const int slab = blockIdx.y;
  if (slab >= P.P * P.Hkv) return;
  const bool clusters = B.use_clusters != 0;
  const bool mean = B.head_agg == 1;
  if (clusters) {
    // this call's per-centroid selection counts start at zero (the select kernel adds)
    const int per_slab = P.wcap * P.n_c;
    for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < per_slab; e += gridDim.x * blockDim.x)
      P.csel[(int64_t)slab * per_slab + e] = 0;
  }
  const int i = slab / P.Hkv, gk = slab - i * P.Hkv, G = P.G;
  const int list0 = i * P.Hq + gk * G;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> 2, t4 = lane & 3;
  uint32_t qf[8][2];
  {
    const uint32_t* qw = reinterpret_cast<const uint32_t*>(P.qeff);
    const int64_t qoff = (int64_t)(list0 + g) * (kHeadDim / 2);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int e = 8 * (4 * (j >> 1) + t4) + 4 * (j & 1);
      qf[j][0] = g < G ? qw[qoff + (e >> 1)] : 0u;
      qf[j][1] = g < G ? qw[qoff + (e >> 1) + 1] : 0u;
    }
  }
  const int c0 = 2 * t4, c1 = 2 * t4 + 1;
  const int ntile = (P.n_cand + 15) / 16;
  const uint4 z = make_uint4(0u, 0u, 0u, 0u);
  for (int tile = blockIdx.x * kDenseWarps + warp; tile < ntile;
       tile += gridDim.x * kDenseWarps) {
    const int j0 = tile * 16 + g, j1 = j0 + 8;
    int id0 = -1, id1 = -1;
    const __nv_bfloat16* p0 = j0 < P.n_cand ? candidate_row(P, clusters, slab, j0, id0) : nullptr;
    const __nv_bfloat16* p1 = j1 < P.n_cand ? candidate_row(P, clusters, slab, j1, id1) : nullptr;
    uint4 ra[4], rb[4];
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      ra[v] = p0 ? ld_stream(p0 + 8 * (4 * v + t4)) : z;
      rb[v] = p1 ? ld_stream(p1 + 8 * (4 * v + t4)) : z;
    }
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      mma_16816(acc, ra[v].x, rb[v].x, ra[v].y, rb[v].y, qf[2 * v][0], qf[2 * v][1]);
      mma_16816(acc, ra[v].z, rb[v].z, ra[v].w, rb[v].w, qf[2 * v + 1][0], qf[2 * v + 1][1]);
    }
    // acc: (row g, head c0), (row g, head c1), (row g + 8, head c0), (row g + 8, head c1)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int h = (e & 1) ? c1 : c0;
      const int j = (e & 2) ? j1 : j0;
      const int id = (e & 2) ? id1 : id0;
      if (h < G && j < P.n_cand) {
        const int64_t o = (int64_t)(list0 + h) * P.cand_cap + j;
        P.cand_s[o] = acc[e] * kScoreScale;
        if (!mean) P.cand_id[o] = id;
      }
    }
  }
}

// ---------------------------------------------------------------------------
// One list per layer: (M, L) of every head's scores (fixed order), then
// alpha_{i,p} = (1/Hq) sum_h 2^(s_{i,h,p} - M_{i,h}) / L_{i,h}, heads in order.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) k_head_stats(const __grid_constant__ Batch B) {
  __shared__ float sm[32], sl[32];
  pdl_wait();
  pdl_release();
  const int pi = blockIdx.y;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  const int L = blockIdx.x;
  if (L >= P.P * P.Hq) return;
  const float* row = P.cand_s + (int64_t)L * P.cand_cap;
  float m = -INFINITY, l = 0.f;
  for (int x = threadIdx.x; x < P.n_cand; x += blockDim.x) ml_combine(m, l, row[x], 1.f);
  block_ml(m, l, sm, sl);
  if (threadIdx.x == 0) P.head_ml[L] = make_float2(m, l);
}

__global__ void __launch_bounds__(256) k_alpha(const __grid_constant__ Batch B) {
  pdl_wait();
  pdl_release();
  const int pi = blockIdx.z;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  const int i = blockIdx.y;
  if (i >= P.P) return;
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= P.n_cand) return;
  float a = 0.f;
  for (int h = 0; h < P.Hq; ++h) {
    const int L = i * P.Hq + h;
    const float2 ml = P.head_ml[L];
    a += fast_exp2(P.cand_s[(int64_t)L * P.cand_cap + j] - ml.x) * (1.0f / ml.y);
  }
  P.aval[(int64_t)i * P.cand_cap + j] = a / (float)P.Hq;   // (its id is its position j)
}

// ---------------------------------------------------------------------------
// Weight of every centroid summed over the G lists of its slab (heads in order):
// cw[slab][e] = sum_h 2^(s_{list0 + h, e} - M) / L.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_centroid_weight(const __grid_constant__ Batch B) {
  pdl_wait();
  pdl_release();
  const int pi = blockIdx.z;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  const int slab = blockIdx.y;
  if (slab >= P.P * P.Hkv) return;
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= P.n_cand - P.n_raw_tok) return;
  const int i = slab / P.Hkv, gk = slab - i * P.Hkv;
  const int list0 = i * P.Hq + gk * P.G;
  // the group's (at most kMaxGroup) scores and statistics loaded together, summed in head
  // order
  float2 ml[kMaxGroup];
  float sv[kMaxGroup];
#pragma unroll
  for (int h = 0; h < kMaxGroup; ++h)
    if (h < P.G) {
      ml[h] = P.list_ml[list0 + h];
      sv[h] = P.cand_s[(int64_t)(list0 + h) * P.cand_cap + P.n_raw_tok + e];
    }
  float a = 0.f;
#pragma unroll
  for (int h = 0; h < kMaxGroup; ++h)
    if (h < P.G) a += fast_exp2(sv[h] - ml[h].x) * (1.0f / ml[h].y);
  P.cw[(int64_t)slab * P.wcap * P.n_c + e] = a;
}

// ---------------------------------------------------------------------------
// Attention mass of every history unit: the sum over lists of the normalised weights of
// the unit's tokens; a compressed unit gets, from each centroid of its window, the
// centroid's weight times (members in the unit) / (members). One block per unit; the
// threads take the (list, token) or (slab, centroid) terms in a fixed order, then a
// fixed tree.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_mass_general(const __grid_constant__ Batch B) {
  __shared__ float sm[32];
  pdl_wait();
  pdl_release();
  const int pi = blockIdx.y;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  const int u = blockIdx.x;
  if (u >= P.Uh) return;
  const int Tu = P.Tu, tid = threadIdx.x;
  float acc = 0.f;
  if (B.head_agg == 1) {
    for (int t = tid; t < P.P * Tu; t += blockDim.x) {
      const int i = t / Tu, r = t - i * Tu;
      acc += P.aval[(int64_t)i * P.cand_cap + (int64_t)u * Tu + r];
    }
  } else if (B.q_agg == 2) {
    // per-query-head lists of row-averaged weights: the rows hold the weights
    for (int t = tid; t < P.P * P.Hq * Tu; t += blockDim.x) {
      const int L = t / Tu, r = t - L * Tu;
      acc += P.cand_s[(int64_t)L * P.cand_cap + (int64_t)u * Tu + r];
    }
  } else {
    const int rr = B.use_clusters ? P.raw_rank[u] : u;
    if (rr >= 0) {
      const int64_t j0 = (int64_t)rr * Tu;
      for (int t = tid; t < P.P * P.Hq * Tu; t += blockDim.x) {
        const int L = t / Tu, r = t - L * Tu;
        const float2 ml = P.list_ml[L];
        acc += fast_exp2(P.cand_s[(int64_t)L * P.cand_cap + j0 + r] - ml.x) * (1.0f / ml.y);
      }
    } else {
      // a compressed unit: its mass and its votes, both from the window's centroids (a
      // centroid's weight shared by member count; one vote per member token for every
      // list that selected the centroid)
      const int w = P.win_slot[u / P.wu];
      const int x = u - P.win_u0[w];
      const int n_c = P.n_c;
      int vs = 0;
      // four (slab, centroid) items per thread at a time: their member counts, weights,
      // sizes and selection counts loaded together, then added in item order
      const int items = P.P * P.Hkv * n_c;
      for (int t0 = tid; t0 < items; t0 += 4 * (int)blockDim.x) {
        int m[4], sz[4], cs[4];
        float cwv[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int t = t0 + q * blockDim.x;
          m[q] = 0;
          sz[q] = 1;
          cs[q] = 0;
          cwv[q] = 0.f;
          if (t < items) {
            const int slab = t / n_c, c = t - slab * n_c;
            const int64_t wc = ((int64_t)slab * P.wcap + w) * n_c + c;
            m[q] = P.mcnt[wc * P.wu + x];
            cwv[q] = P.cw[wc];
            sz[q] = P.msize[wc];
            cs[q] = P.csel[wc];
          }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (m[q]) {
            acc += cwv[q] * (float)m[q] / (float)sz[q];
            vs += cs[q] * m[q];
          }
      }
      // integer block sum (exact in any order)
      __shared__ int svs;
      if (tid == 0) svs = 0;
      __syncthreads();
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) vs += __shfl_down_sync(0xffffffffu, vs, off);
      if ((tid & 31) == 0 && vs) atomicAdd(&svs, vs);
      __syncthreads();
      if (tid == 0) P.votes[u] = svs;
    }
  }
  acc = block_sum(acc, sm);
  if (tid == 0) P.mass[u] = acc;
}

// The same for rows of weights (one list per layer, or the row-averaged lists) when every
// unit's segment is 16-byte aligned (tokens per unit a multiple of 4; rows start on
// 64-value boundaries): 16-byte loads, eight per thread in flight, summed in a fixed order.
__global__ void __launch_bounds__(256) k_mass_rows(const __grid_constant__ Batch B) {
  __shared__ float sm[32];
  pdl_wait();
  pdl_release();
  const int pi = blockIdx.y;
  if (pi >= B.n) return;
  const Prob& P = B.p[pi];
  const int u = blockIdx.x;
  if (u >= P.Uh) return;
  const int Tu = P.Tu, tid = threadIdx.x;
  const float* rows = B.head_agg == 1 ? P.aval : P.cand_s;
  const int nL = B.head_agg == 1 ? P.P : P.P * P.Hq;
  const int n4 = Tu >> 2, items = nL * n4;
  float acc = 0.f;
  for (int t0 = tid; t0 < items; t0 += 8 * (int)blockDim.x) {
    float4 v[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int t = t0 + q * blockDim.x;
      v[q] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (t < items) {
        const int L = t / n4, g = t - L * n4;
        v[q] = *reinterpret_cast<const float4*>(rows + (int64_t)L * P.cand_cap +
                                                (int64_t)u * Tu + 4 * g);
      }
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) acc += (v[q].x + v[q].y) + (v[q].z + v[q].w);
  }
  acc = block_sum(acc, sm);
  if (tid == 0) P.mass[u] = acc;
}

cudaError_t launch_general_score(const Batch& B, int max_cand, int max_slabs,
                                 int max_score_lists, cudaStream_t s) {
  cudaError_t e;
  if (B.use_clusters) {
    e = launch_pdl(k_cluster_map, dim3(1, B.n), dim3(1024), 0, s, B);
    if (e != cudaSuccess) return e;
  }
  const int tiles = (max_cand + 15) / 16;
  const int bx = max(1, min((tiles + kDenseWarps - 1) / kDenseWarps, 2048));
  e = launch_pdl(k_dense, dim3(bx, max_slabs, B.n), dim3(kDenseWarps * 32), 0, s, B);
  if (e != cudaSuccess) return e;
  if (B.head_agg == 1) {
    e = launch_pdl(k_head_stats, dim3(max_score_lists, B.n), dim3(1024), 0, s, B);
    if (e != cudaSuccess) return e;
    int max_p = 0;
    for (int j = 0; j < B.n; ++j) max_p = max(max_p, B.p[j].P);
    e = launch_pdl(k_alpha, dim3((max_cand + 255) / 256, max_p, B.n), dim3(256), 0, s, B);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_mass_general(const Batch& B, int max_cent, int max_slabs,
                                int max_hist_units, cudaStream_t s) {
  if (B.use_clusters && max_cent > 0) {
    const cudaError_t e = launch_pdl(k_centroid_weight, dim3((max_cent + 255) / 256, max_slabs, B.n),
                                     dim3(256), 0, s, B);
    if (e != cudaSuccess) return e;
  }
  if (max_hist_units <= 0) return cudaSuccess;
  bool rows = (B.head_agg == 1 || B.q_agg == 2) && !B.use_clusters;
  for (int j = 0; j < B.n && rows; ++j) rows = B.p[j].Tu % 4 == 0;
  return rows ? launch_pdl(k_mass_rows, dim3(max_hist_units, B.n), dim3(256), 0, s, B)
              : launch_pdl(k_mass_general, dim3(max_hist_units, B.n), dim3(256), 0, s, B);
}

}  // namespace ss
