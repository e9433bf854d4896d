// Retrieval over an index split by token range across GPUs (one shard per GPU).
//
// Every token of a list's global top-k lies in the top-k of the shard that holds it, and
// a list's softmax statistics and every unit's attention mass combine exactly from
// per-shard statistics. So each shard scores only its own keys (Sec. 4.2; the same
// kernels as a single-GPU retrieval, up to the exact per-list top-k) and exports
//   * its per-list top-k tokens (stream token ids) with their log2-scaled scores,
//   * its per-list (M, L) and per-(list, unit) (m, l) softmax statistics,
// which one gather brings to a single host; there the merge below finishes Eq. 11 (the
// global top-k of each list and its weights), the unit votes, the attention mass, the
// vote-ranked pool, max-min diversity and the expansion of Eq. 12.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <vector>

#include "shallowstream.h"
#include "ss_internal.cuh"

namespace ss {

// After the select kernel of a shard: stream token ids (the shard's unit 0 is stream unit
// unit_begin) and the per-(list, unit) statistics of its history units.
__global__ void __launch_bounds__(256) k_shard_export(const __grid_constant__ Batch B,
                                                      int64_t tok_offset, float2* unit_stats) {
  pdl_wait();
  pdl_release();
  const Prob& P = B.p[0];
  if (retrieval_timed_out(P)) return;
  const int L = blockIdx.x;
  if (L >= P.P * P.Hq) return;
  int32_t* tok = P.topk_tok + (int64_t)L * B.k;
  for (int r = threadIdx.x; r < B.k; r += blockDim.x)
    if (tok[r] >= 0) tok[r] = (int32_t)(tok[r] + tok_offset);
  const float2* us = P.ustats + (int64_t)L * P.ucap;
  float2* out = unit_stats + (int64_t)L * P.Uh;
  for (int u = threadIdx.x; u < P.Uh; u += blockDim.x) out[u] = us[u];
}

cudaError_t launch_shard_export(const Batch& B, int64_t tok_offset, float2* unit_stats,
                                cudaStream_t s) {
  return launch_pdl(k_shard_export, dim3(B.p[0].P * B.p[0].Hq), dim3(256), 0, s, B,
                    tok_offset, unit_stats);
}

}  // namespace ss

// ---------------------------------------------------------------------------
// Host merge of the gathered shard payloads.
// ---------------------------------------------------------------------------
#define SS_EXPORT extern "C" __attribute__((visibility("default")))

namespace {
// errors go to the library's thread-local message (ss_last_error)
#define merge_fail ss::fail_status
}  // namespace

SS_EXPORT ss_status ss_merge_shards(const ss_shard* shards, int32_t n_shards, int32_t n_lists,
                                    int32_t tokens_per_unit, int32_t frames_per_unit,
                                    int32_t desc_dim, const ss_retrieve_params* p,
                                    const ss_merge_result* out) {
  using std::vector;
  if (!shards || !p || !out) return merge_fail(SS_ERR_INVALID_ARG, "NULL argument");
  if (n_shards < 1 || n_lists < 1 || tokens_per_unit < 1 || frames_per_unit < 1 || desc_dim < 1)
    return merge_fail(SS_ERR_INVALID_ARG, "sizes must be positive");
  const int k = p->k;
  if (k < 1 || p->budget_units < 1 || p->pool_mult < 1 || p->n_prev < 0)
    return merge_fail(SS_ERR_INVALID_ARG, "invalid retrieval parameters");
  if (p->head_agg != SS_H_PER_QHEAD || p->use_clusters)
    return merge_fail(SS_ERR_UNSUPPORTED, "sharded retrieval needs per-query-head lists over tokens");
  if (!out->topk_tok || !out->topk_w || !out->list_stats || !out->unit_votes || !out->unit_mass ||
      !out->pool || !out->sel_units || !out->exp_units || !out->frames || !out->counts)
    return merge_fail(SS_ERR_INVALID_ARG, "every output array is required");
  // the shards tile the history [0, U) in order
  int64_t U = 0;
  for (int s = 0; s < n_shards; ++s) {
    const ss_shard& sh = shards[s];
    if (sh.unit_begin != U)
      return merge_fail(SS_ERR_INVALID_ARG, "shard %d begins at unit %lld, expected %lld", s,
                        (long long)sh.unit_begin, (long long)U);
    if (sh.n_units < 0) return merge_fail(SS_ERR_INVALID_ARG, "shard %d: n_units < 0", s);
    if (sh.n_units > 0 && (!sh.topk_tok || !sh.topk_s || !sh.list_stats || !sh.unit_stats || !sh.desc))
      return merge_fail(SS_ERR_INVALID_ARG, "shard %d: NULL payload array", s);
    U += sh.n_units;
  }
  const int64_t Tu = tokens_per_unit;

  // (M, L) of each list over all shards (fixed shard order)
  vector<double> M(n_lists, -INFINITY), Ls(n_lists, 0.0);
  for (int li = 0; li < n_lists; ++li) {
    for (int s = 0; s < n_shards; ++s) {
      if (shards[s].n_units == 0) continue;
      const double m = shards[s].list_stats[2 * li], l = shards[s].list_stats[2 * li + 1];
      if (!(l > 0.0)) continue;
      if (m > M[li]) {
        Ls[li] = (M[li] == -INFINITY ? 0.0 : Ls[li] * std::exp2(M[li] - m)) + l;
        M[li] = m;
      } else {
        Ls[li] += l * std::exp2(m - M[li]);
      }
    }
    out->list_stats[2 * li] = (float)M[li];
    out->list_stats[2 * li + 1] = (float)Ls[li];
  }

  // each list's global top-k: the first k of the shards' candidates by (score desc, id asc)
  vector<int32_t> votes(U, 0);
  struct Cand { float s; int32_t id; };
  vector<Cand> c;
  for (int li = 0; li < n_lists; ++li) {
    c.clear();
    for (int s = 0; s < n_shards; ++s) {
      if (shards[s].n_units == 0) continue;
      const int32_t* t = shards[s].topk_tok + (int64_t)li * k;
      const float* sc = shards[s].topk_s + (int64_t)li * k;
      for (int r = 0; r < k; ++r) {
        if (t[r] < 0) break;
        if (t[r] / Tu < shards[s].unit_begin || t[r] / Tu >= shards[s].unit_begin + shards[s].n_units)
          return merge_fail(SS_ERR_INVALID_ARG, "shard %d list %d: token %d outside the shard", s, li, t[r]);
        c.push_back({sc[r], t[r]});
      }
    }
    const size_t n = std::min<size_t>((size_t)k, c.size());
    std::partial_sort(c.begin(), c.begin() + n, c.end(), [](const Cand& a, const Cand& b) {
      return a.s > b.s || (a.s == b.s && a.id < b.id);
    });
    for (int r = 0; r < k; ++r) {
      if ((size_t)r < n) {
        out->topk_tok[(int64_t)li * k + r] = c[r].id;
        out->topk_w[(int64_t)li * k + r] = (float)(std::exp2((double)c[r].s - M[li]) / Ls[li]);
        ++votes[c[r].id / Tu];
      } else {
        out->topk_tok[(int64_t)li * k + r] = -1;
        out->topk_w[(int64_t)li * k + r] = 0.f;
      }
    }
  }

  // attention mass of each unit: its per-list (m, l) under the list's global (M, L)
  vector<double> mass(U, 0.0);
  for (int s = 0; s < n_shards; ++s) {
    const ss_shard& sh = shards[s];
    for (int li = 0; li < n_lists; ++li) {
      if (!(Ls[li] > 0.0)) continue;
      const float* us = sh.unit_stats + (int64_t)li * sh.n_units * 2;
      for (int u = 0; u < sh.n_units; ++u) {
        const double m = us[2 * u], l = us[2 * u + 1];
        if (m == -INFINITY || !(l > 0.0)) continue;
        mass[sh.unit_begin + u] += l * std::exp2(m - M[li]) / Ls[li];
      }
    }
  }
  for (int64_t u = 0; u < U; ++u) {
    out->unit_votes[u] = votes[u];
    out->unit_mass[u] = (float)mass[u];
  }

  // vote-ranked pool: (votes desc, mass desc, unit asc)
  vector<int32_t> order(U);
  for (int64_t u = 0; u < U; ++u) order[u] = (int32_t)u;
  const int64_t pool_n = std::min<int64_t>((int64_t)p->pool_mult * p->budget_units, U);
  std::partial_sort(order.begin(), order.begin() + pool_n, order.end(), [&](int32_t a, int32_t b) {
    if (votes[a] != votes[b]) return votes[a] > votes[b];
    if (mass[a] != mass[b]) return mass[a] > mass[b];
    return a < b;
  });
  for (int64_t r = 0; r < pool_n; ++r) out->pool[r] = order[r];

  // max-min diversity over the pool's descriptors: start at the pool's best; add the unit
  // whose nearest pick is farthest (1 - cosine), ties to the better pool rank
  auto desc_of = [&](int32_t u) -> const float* {
    for (int s = 0; s < n_shards; ++s)
      if (u < shards[s].unit_begin + shards[s].n_units)
        return shards[s].desc + (int64_t)(u - shards[s].unit_begin) * desc_dim;
    return nullptr;
  };
  auto dist = [&](int32_t a, int32_t b) {
    const float* x = desc_of(a);
    const float* y = desc_of(b);
    double d = 0.0;
    for (int i = 0; i < desc_dim; ++i) d += (double)x[i] * (double)y[i];
    return 1.0 - d;
  };
  const int64_t n_sel = std::min<int64_t>(p->budget_units, pool_n);
  vector<int32_t> sel;
  if (n_sel > 0) {
    vector<double> mind(pool_n);
    vector<char> taken(pool_n, 0);
    taken[0] = 1;
    sel.push_back(order[0]);
    for (int64_t r = 0; r < pool_n; ++r) mind[r] = dist(order[r], order[0]);
    while ((int64_t)sel.size() < n_sel) {
      int64_t best = -1;
      for (int64_t r = 0; r < pool_n; ++r)
        if (!taken[r] && (best < 0 || mind[r] > mind[best])) best = r;
      taken[best] = 1;
      sel.push_back(order[best]);
      for (int64_t r = 0; r < pool_n; ++r)
        if (!taken[r]) mind[r] = std::min(mind[r], dist(order[r], order[best]));
    }
  }
  for (size_t r = 0; r < sel.size(); ++r) out->sel_units[r] = sel[r];

  // each pick and its n_prev preceding units, deduplicated, ascending; their frames
  vector<int32_t> ex;
  for (int32_t u : sel)
    for (int j = 0; j <= p->n_prev; ++j)
      if (u - j >= 0) ex.push_back(u - j);
  std::sort(ex.begin(), ex.end());
  ex.erase(std::unique(ex.begin(), ex.end()), ex.end());
  for (size_t r = 0; r < ex.size(); ++r) out->exp_units[r] = ex[r];
  int32_t nf = 0;
  for (int32_t u : ex)
    for (int f = 0; f < frames_per_unit; ++f) out->frames[nf++] = u * frames_per_unit + f;
  out->counts[0] = (int32_t)pool_n;
  out->counts[1] = (int32_t)sel.size();
  out->counts[2] = (int32_t)ex.size();
  out->counts[3] = nf;
  return SS_OK;
}
