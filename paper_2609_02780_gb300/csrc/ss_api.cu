// C ABI of the library (include/shallowstream.h): argument validation, device memory
// of the index, workspace layout and the launch sequence of one retrieval.
#include <atomic>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <vector>

#include <cuda.h>
#include <nvtx3/nvToolsExt.h>

#include "shallowstream.h"
#include "ss_internal.cuh"

#define SS_EXPORT extern "C" __attribute__((visibility("default")))

using namespace ss;

struct ss_index {
  ss_index_config cfg;
  ss_allocator alloc;
  bool custom_alloc;
  int device;
  int sm_count;
  int64_t ncap;        // tokens per slab
  int64_t ucap;        // units
  int64_t n_frames;
  int64_t n_units;
  __nv_bfloat16* keys;  // [P*Hkv][ncap][d]
  float* desc;          // [ucap][Hkv*d]
  // k-means compression
  int32_t win_frames;
  int32_t n_centroids;
  int32_t n_windows;
  int32_t wcap;
  std::vector<int64_t> win_first_frame;
  __nv_bfloat16* cent;  // [P*Hkv][wcap*nc][d]
  uint8_t* assign;      // [P*Hkv][ncap]
  int32_t* win_u0;      // [wcap]
  int32_t* win_slot;    // [ucap / units per window]: window of each window slot, or -1
  int32_t* mcnt;        // [P*Hkv][wcap][nc][units per window] members per (centroid, unit)
  int32_t* msize;       // [P*Hkv][wcap][nc] members per centroid
  uint32_t* kstatus;    // device word: a compression's wait gave up (kStatusTimeout)
  // long-history compression (clusters of units that left the detailed window)
  int64_t n_clustered;  // clustered units: the prefix [0, n_clustered)
  int32_t uc_cap;       // cluster capacity (0 until the first clustering)
  int32_t* unit_cluster;
  float* cdesc;
  int32_t* ccount;
  float* creps;
  int32_t* cfirst;
  int32_t* cprev;
  int32_t* uc_count;    // device: [0] clusters, [1] first cluster the last call touched
  float* uc_work;
  // stored values (the question's forward attends over keys and values)
  __nv_bfloat16* vals;  // [P*Hkv][ncap][d], allocated by the first value append
  int64_t n_vframes;    // frames whose values are stored
};

namespace {
thread_local char g_err[512] = "";

// A named NVTX range around a public call (visible to a profiler's timeline; near free when
// no tool is attached).
struct Range {
  explicit Range(const char* name) { nvtxRangePushA(name); }
  ~Range() { nvtxRangePop(); }
};
}  // namespace

ss_status ss::fail_status(ss_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return s;
}

namespace {

// Polls after which the score kernel's waits for its key copies give up (process-wide).
std::atomic<uint32_t> g_wait_polls{kDefaultWaitPolls};

ss_status fail(ss_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return s;
}

#define SS_CUDA(expr)                                                                 \
  do {                                                                                \
    cudaError_t e_ = (expr);                                                          \
    if (e_ != cudaSuccess) return fail(SS_ERR_CUDA, "%s: %s", #expr, cudaGetErrorString(e_)); \
  } while (0)

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

void* dev_alloc(ss_index* ix, size_t bytes, cudaStream_t st) {
  if (bytes == 0) bytes = 256;
  if (ix->custom_alloc) return ix->alloc.alloc(bytes, (void*)st, ix->alloc.ctx);
  void* p = nullptr;
  if (cudaMalloc(&p, bytes) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return p;
}

void dev_free(ss_index* ix, void* p) {
  if (!p) return;
  if (ix->custom_alloc) {
    ix->alloc.free(p, nullptr, ix->alloc.ctx);
  } else {
    cudaFree(p);
  }
}

int n_lists_of(const ss_index* ix, const ss_retrieve_params* p) {
  return p->head_agg == SS_H_MEAN ? ix->cfg.n_layers : ix->cfg.n_layers * ix->cfg.n_q_heads;
}

int pool_cap_of(const ss_index* ix, const ss_retrieve_params* p) {
  const int64_t pc = (int64_t)p->pool_mult * p->budget_units;
  return (int)(pc < ix->ucap ? pc : ix->ucap);
}

// Candidate slots per list: every token once, plus the unused tails of the slot
// blocks that score warps reserve.
int64_t cand_cap_of(const ss_index* ix) {
  const int64_t c = ix->ncap + (int64_t)kMaxChunksPerSlab * kScoreWarps * kReserve;
  return (c + 63) & ~(int64_t)63;  // keeps every list's slots 256-byte aligned
}

// CTAs per slab of the row-averaged passes, at most (the workspace is sized for it).
int rm_max_chunks(const ss_index* ix) {
  const int n_slabs = ix->cfg.n_layers * ix->cfg.n_kv_heads;
  const int64_t hist_tok = ix->ucap * ix->cfg.tokens_per_frame * ix->cfg.frames_per_unit;
  return rowmean_chunks(n_slabs, (int)(hist_tok > 0x3fffffff ? 0x3fffffff : hist_tok),
                        ix->sm_count);
}

// Workspace regions of one problem (offsets from the problem's base).
struct Layout {
  size_t qeff, cand_s, cand_id, cand_cnt, gthr, ladder, samp_max, ustats, next_unit, gram;
  size_t raw_units, raw_rank, cw, csel, head_ml, aval, rm;  // general path only
  size_t topk_tok, topk_w, list_ml, votes, mass, pool, sel, exp_units, frames, counts,
      status, qstage;
  size_t total;
};

Layout layout_of(const ss_index* ix, int R, const ss_retrieve_params* p) {
  Layout l{};
  size_t cur = 0;
  auto take = [&](size_t bytes) {
    const size_t o = align256(cur);
    cur = o + bytes;
    return o;
  };
  const ss_index_config& c = ix->cfg;
  const int64_t score_lists = (int64_t)c.n_layers * c.n_q_heads;
  const int64_t n_lists = n_lists_of(ix, p);
  const int64_t pc = pool_cap_of(ix, p);
  const int64_t nexp = (int64_t)p->budget_units * (1 + p->n_prev);
  l.qeff = take(score_lists * kHeadDim * 2);
  // candidate (score, id) pairs of the default path; the general path's dense score
  // and id rows are the two halves of the same region
  l.cand_s = take(score_lists * cand_cap_of(ix) * 8);
  l.cand_id = l.cand_s + score_lists * cand_cap_of(ix) * 4;
  l.cand_cnt = take(score_lists * 4);
  l.gthr = take(score_lists * 4);
  l.ladder = take(score_lists * kLadderLevels * 4);
  l.samp_max = take(score_lists * kSampleUnits * 4);
  l.ustats = take(score_lists * ix->ucap * 8);
  l.next_unit = take((int64_t)c.n_layers * c.n_kv_heads * kUnitCounterStride * 4);
  l.gram = take(pc * (pc + 1) / 2 * 4 + 4 * kMaxPool);  // + the greedy's reads past the end
  l.topk_tok = take(n_lists * p->k * 4);
  l.topk_w = take(n_lists * p->k * 4);
  l.list_ml = take(n_lists * 8);
  l.votes = take(ix->ucap * 4);
  l.mass = take(ix->ucap * 4);
  l.pool = take(pc * 4);
  l.sel = take((size_t)p->budget_units * 4);
  l.exp_units = take(nexp * 4);
  l.frames = take(nexp * c.frames_per_unit * 4);
  l.counts = take(16);
  l.status = take(4);
  l.qstage = take((size_t)c.n_layers * R * c.n_q_heads * kHeadDim * 2);
  if (p->use_clusters) {
    l.raw_units = take(ix->ucap * 4);
    l.raw_rank = take(ix->ucap * 4);
    l.cw = take((size_t)c.n_layers * c.n_kv_heads * ix->wcap * ix->n_centroids * 4);
    l.csel = take((size_t)c.n_layers * c.n_kv_heads * ix->wcap * ix->n_centroids * 4);
  }
  if (p->head_agg == SS_H_MEAN) {
    l.head_ml = take(score_lists * 8);
    l.aval = take((size_t)c.n_layers * cand_cap_of(ix) * 4);
  }
  if (p->q_agg == SS_Q_MEAN_SOFTMAX)
    l.rm = take(rowmean_workspace_bytes(c.n_layers * c.n_kv_heads, R,
                                        c.n_q_heads / c.n_kv_heads, rm_max_chunks(ix)));
  l.total = align256(cur);
  return l;
}

ss_status check_params(const ss_retrieve_params* p) {
  if (!p) return fail(SS_ERR_INVALID_ARG, "params is NULL");
  if (p->k < 1) return fail(SS_ERR_INVALID_ARG, "k must be >= 1 (got %d)", p->k);
  if (p->k > kMaxK) return fail(SS_ERR_UNSUPPORTED, "k > %d is not supported", kMaxK);
  if (p->budget_units < 1) return fail(SS_ERR_INVALID_ARG, "budget_units must be >= 1");
  if (p->pool_mult < 1) return fail(SS_ERR_INVALID_ARG, "pool_mult must be >= 1");
  if ((int64_t)p->pool_mult * p->budget_units > kMaxPool)
    return fail(SS_ERR_UNSUPPORTED, "pool_mult * budget_units > %d is not supported", kMaxPool);
  if (p->n_prev < 0) return fail(SS_ERR_INVALID_ARG, "n_prev must be >= 0");
  if (p->n_recent_units < 0) return fail(SS_ERR_INVALID_ARG, "n_recent_units must be >= 0");
  if (p->q_agg != SS_Q_LAST && p->q_agg != SS_Q_MEAN_LOGIT && p->q_agg != SS_Q_MEAN_SOFTMAX)
    return fail(SS_ERR_INVALID_ARG, "unknown q_agg %d", p->q_agg);
  if (p->q_agg == SS_Q_MEAN_SOFTMAX && (p->head_agg != SS_H_PER_QHEAD || p->use_clusters))
    return fail(SS_ERR_UNSUPPORTED, "q_agg SS_Q_MEAN_SOFTMAX needs per-query-head lists over tokens");
  if (p->head_agg != SS_H_PER_QHEAD && p->head_agg != SS_H_MEAN)
    return fail(SS_ERR_INVALID_ARG, "unknown head_agg %d", p->head_agg);
  if (p->use_clusters != 0 && p->use_clusters != 1)
    return fail(SS_ERR_INVALID_ARG, "use_clusters must be 0 or 1");
  if (p->head_agg == SS_H_MEAN && p->use_clusters)
    return fail(SS_ERR_UNSUPPORTED, "use_clusters needs per-query-head lists");
  return SS_OK;
}

// History units scored by a retrieval: the detailed units after the clustered prefix,
// minus the recent ones (Eq. 4).
int64_t hist_units_of(const ss_index* ix, const ss_retrieve_params* p) {
  const int64_t u = ix->n_units - ix->n_clustered - p->n_recent_units;
  return u > 0 ? u : 0;
}

template <typename T>
T* pick(T* user, char* base, size_t off) {
  return user ? user : reinterpret_cast<T*>(base + off);
}

// A shard of a retrieval split by token range: the select kernel also writes the lists'
// scores, and the retrieval ends with the export of the shard's payload.
struct ShardOut {
  int64_t tok_offset;
  float* topk_s;
  float2* unit_stats;
};

ss_status retrieve_impl(ss_index* const* ix, const void* const* q, const int32_t* R, int n,
                        const ss_retrieve_params* p, const ss_result* res, void* ws,
                        size_t ws_bytes, cudaStream_t st, const ss_trace* tr,
                        const ShardOut* shard = nullptr, uint32_t* host_status = nullptr) {
  if (n < 1 || n > kMaxProbs) return fail(SS_ERR_INVALID_ARG, "n must be in [1, %d]", kMaxProbs);
  if (!ix || !q || !R || !res) return fail(SS_ERR_INVALID_ARG, "NULL argument");
  ss_status s = check_params(p);
  if (s != SS_OK) return s;
  if (!ws || ((uintptr_t)ws & 255u)) return fail(SS_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  size_t need = 0;
  int dev = -1;
  for (int j = 0; j < n; ++j) {
    if (!ix[j] || !q[j]) return fail(SS_ERR_INVALID_ARG, "NULL index or query %d", j);
    if (R[j] < 1) return fail(SS_ERR_INVALID_ARG, "n_rows must be >= 1");
    if ((uintptr_t)q[j] & 1u) return fail(SS_ERR_INVALID_ARG, "query rows must be 2-byte aligned");
    if (dev < 0) dev = ix[j]->device;
    if (ix[j]->device != dev) return fail(SS_ERR_INVALID_ARG, "indexes on different devices");
    if (hist_units_of(ix[j], p) > kMaxHistUnits)
      return fail(SS_ERR_UNSUPPORTED, "more than %d history units", kMaxHistUnits);
    if (p->use_clusters && ix[j]->n_windows == 0)
      return fail(SS_ERR_STATE, "index %d has no compressed windows", j);
    if (shard && ix[j]->n_clustered > 0)
      return fail(SS_ERR_UNSUPPORTED, "a shard with clustered units");
    if (p->q_agg == SS_Q_MEAN_SOFTMAX &&
        !rowmean_supported(R[j], ix[j]->cfg.n_q_heads / ix[j]->cfg.n_kv_heads))
      return fail(SS_ERR_UNSUPPORTED,
                  "q_agg SS_Q_MEAN_SOFTMAX supports up to 64 rows and (heads per key head) x "
                  "(rows rounded up to 16) <= 512");
    const ss_result& r = res[j];
    if (!r.sel_units || !r.exp_units || !r.frames || !r.counts || !r.status)
      return fail(SS_ERR_INVALID_ARG, "result %d: sel_units, exp_units, frames, counts and status are required", j);
    need += layout_of(ix[j], R[j], p).total;
  }
  if (ws_bytes < need)
    return fail(SS_ERR_INVALID_ARG, "workspace too small: %zu < %zu bytes", ws_bytes, need);

  thread_local Batch B;  // large; built on the host and passed by value to each launch
  std::memset(&B, 0, sizeof(B));
  B.n = n;
  B.k = p->k;
  B.n_prev = p->n_prev;
  B.q_agg = p->q_agg;
  B.head_agg = p->head_agg;
  B.use_clusters = p->use_clusters;
  B.wait_polls = g_wait_polls.load(std::memory_order_relaxed);
  const bool general = p->head_agg == SS_H_MEAN || p->use_clusters ||
                       p->q_agg == SS_Q_MEAN_SOFTMAX;
  int max_lists = 0, max_uh = 0, max_pool = 0, n_slabs_total = 0;
  int max_cand = 0, max_slabs = 0, max_score_lists = 0, max_cent = 0;
  char* base = static_cast<char*>(ws);
  for (int j = 0; j < n; ++j) {
    const ss_index* x = ix[j];
    const ss_index_config& c = x->cfg;
    const Layout l = layout_of(x, R[j], p);
    Prob& P = B.p[j];
    // with clustered units the kernels see the index from its first detailed unit on;
    // k_uc_shift moves the outputs back to stream numbering
    const int64_t uoff = x->n_clustered;
    const int64_t tu = (int64_t)c.tokens_per_frame * c.frames_per_unit;
    P.unit_offset = (int)uoff;
    P.keys = x->keys + uoff * tu * kHeadDim;
    P.desc = x->desc + uoff * c.n_kv_heads * kHeadDim;
    P.ncap = x->ncap;
    P.P = c.n_layers;
    P.Hq = c.n_q_heads;
    P.Hkv = c.n_kv_heads;
    P.G = c.n_q_heads / c.n_kv_heads;
    P.fpu = c.frames_per_unit;
    P.Tu = c.tokens_per_frame * c.frames_per_unit;
    P.U = (int)(x->n_units - uoff);
    P.Uh = (int)hist_units_of(x, p);
    P.ucap = (int)(x->ucap - uoff);
    P.index_status = x->kstatus;
    P.q = static_cast<const __nv_bfloat16*>(q[j]);
    P.R = R[j];
    P.qeff = reinterpret_cast<__nv_bfloat16*>(base + l.qeff);
    P.cand_pair = reinterpret_cast<float2*>(base + l.cand_s);
    P.cand_s = reinterpret_cast<float*>(base + l.cand_s);
    P.cand_id = reinterpret_cast<int32_t*>(base + l.cand_id);
    P.cand_cap = cand_cap_of(x);
    P.cand_cnt = reinterpret_cast<int32_t*>(base + l.cand_cnt);
    P.gthr = reinterpret_cast<uint32_t*>(base + l.gthr);
    P.ladder = reinterpret_cast<int32_t*>(base + l.ladder);
    P.samp_max = reinterpret_cast<float*>(base + l.samp_max);
    P.ustats = reinterpret_cast<float2*>(base + l.ustats);
    P.next_unit = reinterpret_cast<int32_t*>(base + l.next_unit);
    P.gram = reinterpret_cast<float*>(base + l.gram);
    const ss_result& r = res[j];
    P.topk_tok = pick(r.topk_tok, base, l.topk_tok);
    P.topk_w = pick(r.topk_w, base, l.topk_w);
    P.topk_s = shard ? shard->topk_s : nullptr;
    P.list_ml = pick(reinterpret_cast<float2*>(r.list_stats), base, l.list_ml);
    P.votes_base = pick(r.unit_votes, base, l.votes);
    P.mass_base = pick(r.unit_mass, base, l.mass);
    P.votes = P.votes_base + uoff;
    P.mass = P.mass_base + uoff;
    P.pool = pick(r.pool, base, l.pool);
    P.sel = r.sel_units;
    P.exp_units = r.exp_units;
    P.frames = r.frames;
    P.counts = r.counts;
    P.status = r.status;
    P.host_status = host_status;
    const int64_t pc = (int64_t)p->pool_mult * p->budget_units;
    P.pool_n = (int)(pc < P.Uh ? pc : P.Uh);
    P.n_sample = sample_units(p->k, P.Tu, P.Uh);
    P.n_sel = P.pool_n < p->budget_units ? P.pool_n : p->budget_units;
    if (general) {
      // candidates: raw tokens of the history units no window covers, then the
      // centroids of the windows that start in the history (a prefix of the windows)
      int64_t covered = 0, n_live = 0;
      if (p->use_clusters) {
        const int fpu = c.frames_per_unit;
        const int64_t wu = x->win_frames / fpu;
        for (int64_t f : x->win_first_frame) {
          const int64_t u0 = f / fpu;
          if (u0 >= P.Uh) break;
          ++n_live;
          covered += (u0 + wu < P.Uh ? u0 + wu : P.Uh) - u0;
        }
        P.n_c = x->n_centroids;
        P.wu = (int)wu;
        P.wcap = x->wcap;
        P.cent = x->cent;
        P.mcnt = x->mcnt;
        P.msize = x->msize;
        P.win_slot = x->win_slot;
        P.win_u0 = x->win_u0;
        P.raw_units = reinterpret_cast<int32_t*>(base + l.raw_units);
        P.raw_rank = reinterpret_cast<int32_t*>(base + l.raw_rank);
        P.cw = reinterpret_cast<float*>(base + l.cw);
        P.csel = reinterpret_cast<int32_t*>(base + l.csel);
      }
      P.n_raw_tok = (int)((P.Uh - covered) * P.Tu);
      P.n_cand = (int)(P.n_raw_tok + n_live * P.n_c);
      if (p->head_agg == SS_H_MEAN) {
        P.head_ml = reinterpret_cast<float2*>(base + l.head_ml);
        P.aval = reinterpret_cast<float*>(base + l.aval);
      }
      if (p->q_agg == SS_Q_MEAN_SOFTMAX) {
        P.rm_scratch = reinterpret_cast<float2*>(base + l.rm);
        P.rm_chunks = rowmean_chunks(P.P * P.Hkv, P.Uh * P.Tu, x->sm_count);
      }
      max_cand = max(max_cand, P.n_cand);
      max_cent = max(max_cent, P.n_cand - P.n_raw_tok);
      max_slabs = max(max_slabs, P.P * P.Hkv);
      max_score_lists = max(max_score_lists, P.P * P.Hq);
    }
    max_lists = max(max_lists, p->head_agg == SS_H_MEAN ? P.P : P.P * P.Hq);
    max_uh = max(max_uh, P.Uh);
    max_pool = max(max_pool, P.pool_n);
    n_slabs_total += P.P * P.Hkv;
    base += l.total;
  }
  // Score-kernel mapping: CTAs per slab, sized with a common units-per-CTA length for
  // all problems (the CTAs of a slab share its units dynamically).
  const int c_common = score_chunks_per_slab(n_slabs_total, max_uh, ix[0]->sm_count);
  const int chunk_len = c_common > 0 ? (max_uh + c_common - 1) / c_common : 1;
  int cta = 0;
  for (int j = 0; j < n; ++j) {
    Prob& P = B.p[j];
    P.chunks = P.Uh > 0 ? (P.Uh + chunk_len - 1) / chunk_len : 0;
    P.cta_begin = cta;
    cta += P.P * P.Hkv * P.chunks;
  }
  B.score_ctas = cta;
  B.score_spread = cta <= score_slots(ix[0]->sm_count) ? 1 : 0;

  SS_CUDA(cudaSetDevice(dev));
  SS_CUDA(launch_prep(B, st));
  if (tr && tr->score_begin) SS_CUDA(cudaEventRecord((cudaEvent_t)tr->score_begin, st));
  if (p->q_agg == SS_Q_MEAN_SOFTMAX) {
    for (int j = 0; j < n; ++j)
      SS_CUDA(launch_rowmean(B, j, B.p[j].rm_scratch, B.p[j].rm_chunks, st));
  } else if (general) {
    SS_CUDA(launch_general_score(B, max_cand, max_slabs, max_score_lists, st));
  } else {
    SS_CUDA(launch_score(B, st));
  }
  if (tr && tr->score_end) SS_CUDA(cudaEventRecord((cudaEvent_t)tr->score_end, st));
  if (general) {
    SS_CUDA(launch_select_general(B, max_lists, ix[0]->sm_count, st));
    SS_CUDA(launch_mass_general(B, max_cent, max_slabs, max_uh, st));
  } else {
    SS_CUDA(launch_select(B, max_lists, ix[0]->sm_count, st));
    if (shard) {
      SS_CUDA(launch_shard_export(B, shard->tok_offset, shard->unit_stats, st));
      return SS_OK;
    }
    SS_CUDA(launch_mass(B, max_uh, st));
  }
  SS_CUDA(launch_pool(B, max_uh, st));
  SS_CUDA(launch_maxmin(B, max_pool, st));
  bool shifted = false;
  for (int j = 0; j < n; ++j) shifted = shifted || B.p[j].unit_offset > 0;
  if (shifted) SS_CUDA(launch_uc_shift(B, st));
  return SS_OK;
}

}  // namespace

SS_EXPORT const char* ss_status_string(ss_status s) {
  switch (s) {
    case SS_OK: return "SS_OK";
    case SS_ERR_INVALID_ARG: return "SS_ERR_INVALID_ARG";
    case SS_ERR_UNSUPPORTED: return "SS_ERR_UNSUPPORTED";
    case SS_ERR_CAPACITY: return "SS_ERR_CAPACITY";
    case SS_ERR_STATE: return "SS_ERR_STATE";
    case SS_ERR_ALLOC: return "SS_ERR_ALLOC";
    case SS_ERR_CUDA: return "SS_ERR_CUDA";
    case SS_ERR_TIMEOUT: return "SS_ERR_TIMEOUT";
    case SS_ERR_INTERNAL: return "SS_ERR_INTERNAL";
  }
  return "unknown status";
}

SS_EXPORT const char* ss_last_error(void) { return g_err; }

SS_EXPORT const char* ss_version(void) { return "shallowstream-gb300 0.2 (sm_103a)"; }

SS_EXPORT ss_status ss_set_wait_limit(int64_t polls) {
  if (polls < -1 || polls > (int64_t)UINT32_MAX)
    return fail(SS_ERR_INVALID_ARG, "polls must be -1 (default) or in [0, 2^32)");
  g_wait_polls.store(polls < 0 ? kDefaultWaitPolls : (uint32_t)polls, std::memory_order_relaxed);
  return SS_OK;
}

SS_EXPORT ss_status ss_index_create(const ss_index_config* cfg, const ss_allocator* alloc,
                                    void* stream, ss_index** out) {
  if (!out) return fail(SS_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (!cfg) return fail(SS_ERR_INVALID_ARG, "config is NULL");
  const ss_index_config& c = *cfg;
  if (c.n_layers < 1 || c.n_q_heads < 1 || c.n_kv_heads < 1 || c.tokens_per_frame < 1 ||
      c.frames_per_unit < 1 || c.max_frames < 1)
    return fail(SS_ERR_INVALID_ARG, "sizes must be positive");
  if (c.n_q_heads % c.n_kv_heads)
    return fail(SS_ERR_INVALID_ARG, "n_q_heads must be a multiple of n_kv_heads");
  if (c.max_frames % c.frames_per_unit)
    return fail(SS_ERR_INVALID_ARG, "max_frames must be a multiple of frames_per_unit");
  if (c.head_dim != kHeadDim) return fail(SS_ERR_UNSUPPORTED, "head_dim must be 128");
  if (c.n_q_heads / c.n_kv_heads > kMaxGroup)
    return fail(SS_ERR_UNSUPPORTED, "more than %d query heads per key head", kMaxGroup);
  if (c.n_kv_heads > 8) return fail(SS_ERR_UNSUPPORTED, "more than 8 key heads");
  if ((int64_t)c.n_layers * c.n_q_heads > 1024)
    return fail(SS_ERR_UNSUPPORTED, "more than 1024 (layer, query head) lists");
  if ((int64_t)c.tokens_per_frame * c.max_frames > (int64_t)0x3fffffff)
    return fail(SS_ERR_UNSUPPORTED, "more than 2^30 tokens per slab");
  if (alloc && (!alloc->alloc || !alloc->free))
    return fail(SS_ERR_INVALID_ARG, "allocator needs alloc and free");
  ss_index* ix = new ss_index();
  ix->cfg = c;
  ix->custom_alloc = alloc != nullptr;
  if (alloc) ix->alloc = *alloc;
  if (cudaGetDevice(&ix->device) != cudaSuccess ||
      cudaDeviceGetAttribute(&ix->sm_count, cudaDevAttrMultiProcessorCount, ix->device) != cudaSuccess) {
    cudaGetLastError();
    delete ix;
    return fail(SS_ERR_CUDA, "no usable CUDA device");
  }
  ix->ncap = c.max_frames * c.tokens_per_frame;
  ix->ucap = c.max_frames / c.frames_per_unit;
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t kb = (size_t)c.n_layers * c.n_kv_heads * ix->ncap * kHeadDim * 2;
  const size_t db = (size_t)ix->ucap * c.n_kv_heads * kHeadDim * 4;
  ix->keys = static_cast<__nv_bfloat16*>(dev_alloc(ix, kb, st));
  ix->desc = static_cast<float*>(dev_alloc(ix, db, st));
  if (!ix->keys || !ix->desc || ((uintptr_t)ix->keys & 15u) || ((uintptr_t)ix->desc & 15u)) {
    dev_free(ix, ix->keys);
    dev_free(ix, ix->desc);
    delete ix;
    return fail(SS_ERR_ALLOC, "device allocation of %zu + %zu bytes failed (or was not 16-byte aligned)", kb, db);
  }
  *out = ix;
  return SS_OK;
}

SS_EXPORT ss_status ss_index_destroy(ss_index* ix) {
  if (!ix) return SS_OK;
  dev_free(ix, ix->keys);
  dev_free(ix, ix->desc);
  dev_free(ix, ix->cent);
  dev_free(ix, ix->assign);
  dev_free(ix, ix->win_u0);
  dev_free(ix, ix->win_slot);
  dev_free(ix, ix->mcnt);
  dev_free(ix, ix->msize);
  dev_free(ix, ix->kstatus);
  dev_free(ix, ix->unit_cluster);
  dev_free(ix, ix->cdesc);
  dev_free(ix, ix->ccount);
  dev_free(ix, ix->creps);
  dev_free(ix, ix->cfirst);
  dev_free(ix, ix->cprev);
  dev_free(ix, ix->uc_count);
  dev_free(ix, ix->uc_work);
  dev_free(ix, ix->vals);
  delete ix;
  return SS_OK;
}

SS_EXPORT ss_status ss_index_append(ss_index* ix, const void* keys, int32_t n_frames,
                                    int64_t stride, void* stream) {
  Range range_("ss_index_append");
  if (!ix) return fail(SS_ERR_INVALID_ARG, "index is NULL");
  if (n_frames < 0) return fail(SS_ERR_INVALID_ARG, "n_frames must be >= 0");
  if (n_frames == 0) return SS_OK;
  if (!keys) return fail(SS_ERR_INVALID_ARG, "keys is NULL");
  if ((uintptr_t)keys & 15u) return fail(SS_ERR_INVALID_ARG, "keys must be 16-byte aligned");
  const ss_index_config& c = ix->cfg;
  const int64_t n_tok = (int64_t)n_frames * c.tokens_per_frame;
  if (stride == 0) stride = n_tok;
  if (stride < n_tok) return fail(SS_ERR_INVALID_ARG, "slab_stride_tokens < n_frames * tokens_per_frame");
  if (ix->n_frames + n_frames > c.max_frames)
    return fail(SS_ERR_CAPACITY, "append of %d frames exceeds max_frames %lld (have %lld)", n_frames,
                (long long)c.max_frames, (long long)ix->n_frames);
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  SS_CUDA(cudaSetDevice(ix->device));
  SS_CUDA(launch_append(ix->keys, ix->ncap, ix->n_frames * c.tokens_per_frame,
                        static_cast<const __nv_bfloat16*>(keys), stride,
                        c.n_layers * c.n_kv_heads, n_tok, st));
  const int64_t new_units = (ix->n_frames + n_frames) / c.frames_per_unit;
  SS_CUDA(launch_descriptors(ix->keys, ix->ncap, c.n_layers, c.n_kv_heads,
                             c.tokens_per_frame * c.frames_per_unit, ix->n_units, new_units,
                             ix->desc, st));
  ix->n_frames += n_frames;
  ix->n_units = new_units;
  return SS_OK;
}

SS_EXPORT ss_status ss_index_get_config(const ss_index* ix, ss_index_config* cfg) {
  if (!ix || !cfg) return fail(SS_ERR_INVALID_ARG, "NULL argument");
  *cfg = ix->cfg;
  return SS_OK;
}

// ---------------------------------------------------------------------------
// Checkpoint: the index's host metadata and every device array, raw, at full capacity.
// ---------------------------------------------------------------------------
namespace {

constexpr char kFileMagic[8] = {'S', 'S', 'I', 'D', 'X', 0, 0, 1};

struct FileHeader {
  ss_index_config cfg;
  int64_t n_frames, n_units, n_vframes;
  int32_t win_frames, n_centroids, n_windows, wcap;
  int64_t n_clustered;
  int32_t uc_cap, has_values;
};

// The device arrays of an index in file order, with their sizes (0 = not allocated).
struct ArrayRef {
  void** ptr;
  size_t bytes;
};

std::vector<ArrayRef> index_arrays(ss_index* ix, bool values) {
  const ss_index_config& c = ix->cfg;
  const size_t n_slabs = (size_t)c.n_layers * c.n_kv_heads;
  const size_t D = (size_t)c.n_kv_heads * kHeadDim;
  const size_t Tu = (size_t)c.tokens_per_frame * c.frames_per_unit;
  const size_t kb = n_slabs * ix->ncap * kHeadDim * 2;
  std::vector<ArrayRef> a;
  a.push_back({(void**)&ix->keys, kb});
  a.push_back({(void**)&ix->desc, (size_t)ix->ucap * D * 4});
  a.push_back({(void**)&ix->vals, values ? kb : 0});
  const bool win = ix->win_frames > 0;
  const size_t wcap = (size_t)ix->wcap, nc = (size_t)ix->n_centroids;
  const size_t wu = win ? (size_t)(ix->win_frames / c.frames_per_unit) : 1;
  const size_t n_slots = win ? ((size_t)ix->ucap + wu - 1) / wu : 0;
  a.push_back({(void**)&ix->cent, win ? n_slabs * wcap * nc * kHeadDim * 2 : 0});
  a.push_back({(void**)&ix->assign, win ? n_slabs * ix->ncap : 0});
  a.push_back({(void**)&ix->win_u0, win ? wcap * 4 : 0});
  a.push_back({(void**)&ix->win_slot, win ? n_slots * 4 : 0});
  a.push_back({(void**)&ix->mcnt, win ? n_slabs * wcap * nc * wu * 4 : 0});
  a.push_back({(void**)&ix->msize, win ? n_slabs * wcap * nc * 4 : 0});
  const size_t cap = (size_t)ix->uc_cap;
  const bool uc = cap > 0;
  a.push_back({(void**)&ix->kstatus, (win || uc) ? (size_t)256 : (size_t)0});
  a.push_back({(void**)&ix->unit_cluster, uc ? (size_t)ix->ucap * 4 : 0});
  a.push_back({(void**)&ix->cdesc, uc ? cap * D * 4 : 0});
  a.push_back({(void**)&ix->ccount, uc ? cap * 4 : 0});
  a.push_back({(void**)&ix->creps, uc ? cap * n_slabs * Tu * kHeadDim * 4 : 0});
  a.push_back({(void**)&ix->cfirst, uc ? cap * 4 : 0});
  a.push_back({(void**)&ix->cprev, uc ? cap * 4 : 0});
  a.push_back({(void**)&ix->uc_count, uc ? (size_t)256 : (size_t)0});
  a.push_back({(void**)&ix->uc_work, uc ? cap * 4 : 0});
  return a;
}

constexpr size_t kIoChunk = 64u << 20;   // host staging per copy

}  // namespace

SS_EXPORT ss_status ss_index_save(const ss_index* cix, const char* path, void* stream) {
  Range range_("ss_index_save");
  if (!cix || !path) return fail(SS_ERR_INVALID_ARG, "NULL argument");
  ss_index* ix = const_cast<ss_index*>(cix);
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  SS_CUDA(cudaSetDevice(ix->device));
  FileHeader h{};
  h.cfg = ix->cfg;
  h.n_frames = ix->n_frames;
  h.n_units = ix->n_units;
  h.n_vframes = ix->n_vframes;
  h.win_frames = ix->win_frames;
  h.n_centroids = ix->n_centroids;
  h.n_windows = ix->n_windows;
  h.wcap = ix->wcap;
  h.n_clustered = ix->n_clustered;
  h.uc_cap = ix->uc_cap;
  h.has_values = ix->vals != nullptr;
  FILE* f = fopen(path, "wb");
  if (!f) return fail(SS_ERR_INVALID_ARG, "cannot open %s for writing", path);
  void* stage = nullptr;
  if (cudaMallocHost(&stage, kIoChunk) != cudaSuccess) {
    cudaGetLastError();
    fclose(f);
    return fail(SS_ERR_ALLOC, "page-locked staging buffer");
  }
  bool ok = fwrite(kFileMagic, 1, 8, f) == 8 && fwrite(&h, sizeof(h), 1, f) == 1;
  for (int64_t fr : ix->win_first_frame) ok = ok && fwrite(&fr, 8, 1, f) == 1;
  cudaError_t ce = cudaSuccess;
  for (const ArrayRef& a : index_arrays(ix, ix->vals != nullptr)) {
    const int64_t nb = (int64_t)a.bytes;
    ok = ok && fwrite(&nb, 8, 1, f) == 1;
    for (size_t off = 0; ok && ce == cudaSuccess && off < a.bytes; off += kIoChunk) {
      const size_t n = a.bytes - off < kIoChunk ? a.bytes - off : kIoChunk;
      ce = cudaMemcpyAsync(stage, static_cast<const char*>(*a.ptr) + off, n,
                           cudaMemcpyDeviceToHost, st);
      if (ce == cudaSuccess) ce = cudaStreamSynchronize(st);
      ok = ok && ce == cudaSuccess && fwrite(stage, 1, n, f) == n;
    }
  }
  cudaFreeHost(stage);
  ok = (fclose(f) == 0) && ok;
  if (ce != cudaSuccess) return fail(SS_ERR_CUDA, "device-to-host copy: %s", cudaGetErrorString(ce));
  if (!ok) return fail(SS_ERR_INVALID_ARG, "write to %s failed", path);
  return SS_OK;
}

SS_EXPORT ss_status ss_index_load(const char* path, const ss_allocator* alloc, void* stream,
                                  ss_index** out) {
  Range range_("ss_index_load");
  if (!path || !out) return fail(SS_ERR_INVALID_ARG, "NULL argument");
  *out = nullptr;
  FILE* f = fopen(path, "rb");
  if (!f) return fail(SS_ERR_INVALID_ARG, "cannot open %s", path);
  char magic[8];
  FileHeader h{};
  if (fread(magic, 1, 8, f) != 8 || memcmp(magic, kFileMagic, 8) != 0 ||
      fread(&h, sizeof(h), 1, f) != 1) {
    fclose(f);
    return fail(SS_ERR_INVALID_ARG, "%s is not an index file of this version", path);
  }
  ss_index* ix = nullptr;
  ss_status s = ss_index_create(&h.cfg, alloc, stream, &ix);
  if (s != SS_OK) {
    fclose(f);
    return s;
  }
  const bool sane = h.n_frames >= 0 && h.n_frames <= h.cfg.max_frames && h.n_vframes >= 0 &&
                    h.n_vframes <= h.n_frames && h.n_windows >= 0 && h.wcap >= 0 &&
                    h.n_windows <= h.wcap && h.uc_cap >= 0 && h.n_clustered >= 0 &&
                    h.n_centroids >= 0 && h.n_centroids <= kMaxCentroids &&
                    h.win_frames >= 0 && h.n_units == h.n_frames / h.cfg.frames_per_unit &&
                    (h.win_frames == 0 || h.win_frames % h.cfg.frames_per_unit == 0);
  bool ok = sane;
  for (int32_t w = 0; ok && w < h.n_windows; ++w) {
    int64_t fr = 0;
    ok = fread(&fr, 8, 1, f) == 1;
    ix->win_first_frame.push_back(fr);
  }
  if (ok) {
    ix->n_frames = h.n_frames;
    ix->n_units = h.n_units;
    ix->n_vframes = h.n_vframes;
    ix->win_frames = h.win_frames;
    ix->n_centroids = h.n_centroids;
    ix->n_windows = h.n_windows;
    ix->wcap = h.wcap;
    ix->n_clustered = h.n_clustered;
    ix->uc_cap = h.uc_cap;
  }
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  void* stage = nullptr;
  if (ok && cudaMallocHost(&stage, kIoChunk) != cudaSuccess) {
    cudaGetLastError();
    stage = nullptr;
    ok = false;
  }
  cudaError_t ce = cudaSuccess;
  bool alloc_failed = false;
  if (ok) {
    // the arrays the saved index had allocated are allocated here with the same sizes
    // (the keys and descriptors come from ss_index_create)
    if (h.win_frames == 0) ix->wcap = 0;
    for (ArrayRef& a : index_arrays(ix, h.has_values != 0)) {
      int64_t nb = -1;
      if (!ok || fread(&nb, 8, 1, f) != 1 || nb != (int64_t)a.bytes) {
        ok = false;
        break;
      }
      if (a.bytes == 0) continue;
      if (!*a.ptr) {
        *a.ptr = dev_alloc(ix, a.bytes, st);
        if (!*a.ptr) {
          alloc_failed = true;
          ok = false;
          break;
        }
      }
      for (size_t off = 0; ok && off < a.bytes; off += kIoChunk) {
        const size_t n = a.bytes - off < kIoChunk ? a.bytes - off : kIoChunk;
        ok = fread(stage, 1, n, f) == n;
        if (ok) ce = cudaMemcpyAsync(static_cast<char*>(*a.ptr) + off, stage, n,
                                     cudaMemcpyHostToDevice, st);
        if (ok && ce == cudaSuccess) ce = cudaStreamSynchronize(st);
        ok = ok && ce == cudaSuccess;
      }
    }
  }
  if (stage) cudaFreeHost(stage);
  fclose(f);
  if (!ok) {
    ss_index_destroy(ix);
    if (alloc_failed) return fail(SS_ERR_ALLOC, "device allocation while loading %s", path);
    if (ce != cudaSuccess) return fail(SS_ERR_CUDA, "host-to-device copy: %s", cudaGetErrorString(ce));
    return fail(SS_ERR_INVALID_ARG, "%s is truncated or inconsistent", path);
  }
  *out = ix;
  return SS_OK;
}

SS_EXPORT ss_status ss_index_get_view(const ss_index* ix, ss_index_view* v) {
  if (!ix || !v) return fail(SS_ERR_INVALID_ARG, "NULL argument");
  v->n_frames = ix->n_frames;
  v->n_units = ix->n_units;
  v->token_capacity = ix->ncap;
  v->keys = ix->keys;
  v->descriptors = ix->desc;
  v->n_windows = ix->n_windows;
  v->window_frames = ix->win_frames;
  v->n_centroids = ix->n_centroids;
  v->centroids = ix->cent;
  v->assignment = ix->assign;
  v->window_first_unit = ix->win_u0;
  v->member_counts = ix->mcnt;
  v->member_sizes = ix->msize;
  v->n_clustered_units = ix->n_clustered;
  v->cluster_capacity = ix->uc_cap;
  v->unit_cluster = ix->unit_cluster;
  v->cluster_count = ix->uc_count;
  v->cluster_centroids = ix->cdesc;
  v->cluster_sizes = ix->ccount;
  v->cluster_keys = ix->creps;
  v->values = ix->vals;
  v->n_value_frames = ix->n_vframes;
  return SS_OK;
}

SS_EXPORT ss_status ss_index_append_values(ss_index* ix, const void* values, int32_t n_frames,
                                           int64_t stride, void* stream) {
  Range range_("ss_index_append_values");
  if (!ix) return fail(SS_ERR_INVALID_ARG, "index is NULL");
  if (n_frames < 0) return fail(SS_ERR_INVALID_ARG, "n_frames must be >= 0");
  if (n_frames == 0) return SS_OK;
  if (!values) return fail(SS_ERR_INVALID_ARG, "values is NULL");
  if ((uintptr_t)values & 15u) return fail(SS_ERR_INVALID_ARG, "values must be 16-byte aligned");
  const ss_index_config& c = ix->cfg;
  const int64_t n_tok = (int64_t)n_frames * c.tokens_per_frame;
  if (stride == 0) stride = n_tok;
  if (stride < n_tok) return fail(SS_ERR_INVALID_ARG, "slab_stride_tokens < n_frames * tokens_per_frame");
  if (ix->n_vframes + n_frames > ix->n_frames)
    return fail(SS_ERR_STATE, "values of %d frames would pass the %lld frames whose keys are stored",
                n_frames, (long long)ix->n_frames);
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  SS_CUDA(cudaSetDevice(ix->device));
  if (!ix->vals) {
    const size_t vb = (size_t)c.n_layers * c.n_kv_heads * ix->ncap * kHeadDim * 2;
    ix->vals = static_cast<__nv_bfloat16*>(dev_alloc(ix, vb, st));
    if (!ix->vals || ((uintptr_t)ix->vals & 15u)) {
      dev_free(ix, ix->vals);
      ix->vals = nullptr;
      return fail(SS_ERR_ALLOC, "device allocation of %zu bytes for the values failed", vb);
    }
  }
  SS_CUDA(launch_append(ix->vals, ix->ncap, ix->n_vframes * c.tokens_per_frame,
                        static_cast<const __nv_bfloat16*>(values), stride,
                        c.n_layers * c.n_kv_heads, n_tok, st));
  ix->n_vframes += n_frames;
  return SS_OK;
}

namespace {
ss_status forward_shape(const ss_index* ix, int32_t R, const ss_forward_params* fp, FwShape* F) {
  if (!ix || !fp) return fail(SS_ERR_INVALID_ARG, "NULL argument");
  const ss_index_config& c = ix->cfg;
  if (R < 1) return fail(SS_ERR_INVALID_ARG, "n_rows must be >= 1");
  if (!forward_supported(R, c.n_q_heads, c.n_kv_heads))
    return fail(SS_ERR_UNSUPPORTED,
                "the forward needs R <= 64 and (Hq / Hkv) * (R rounded up to 16) <= 256");
  if (fp->intermediate < 128 || fp->intermediate % 128)
    return fail(SS_ERR_INVALID_ARG, "intermediate must be a positive multiple of 128");
  if (!(fp->rms_eps > 0.f) || !(fp->rope_theta > 1.f))
    return fail(SS_ERR_INVALID_ARG, "rms_eps must be > 0 and rope_theta > 1");
  if ((int64_t)c.n_q_heads * kHeadDim > 16384)
    return fail(SS_ERR_UNSUPPORTED, "hidden size above 16384");
  F->P = c.n_layers;
  F->Hq = c.n_q_heads;
  F->Hkv = c.n_kv_heads;
  F->R = R;
  F->I = fp->intermediate;
  F->ncap = ix->ncap;
  F->n_tok = (int)(ix->n_frames * c.tokens_per_frame);
  F->sm_count = ix->sm_count;
  F->eps = fp->rms_eps;
  F->theta = (double)fp->rope_theta;
  F->pos0 = fp->pos0 < 0 ? (int64_t)F->n_tok : fp->pos0;
  F->keys = ix->keys;
  F->values = ix->vals;
  return SS_OK;
}
}  // namespace

SS_EXPORT ss_status ss_forward_workspace_size(const ss_index* ix, int32_t n_rows,
                                              const ss_forward_params* fp, size_t* bytes) {
  if (!bytes) return fail(SS_ERR_INVALID_ARG, "bytes is NULL");
  FwShape F{};
  const ss_status s = forward_shape(ix, n_rows, fp, &F);
  if (s != SS_OK) return s;
  *bytes = forward_workspace_bytes(F);
  return SS_OK;
}

SS_EXPORT ss_status ss_question_forward(ss_index* ix, const ss_layer_weights* layers,
                                        const ss_forward_params* fp, const void* h_in,
                                        int32_t n_rows, void* q_out, float* h_out,
                                        uint32_t* status, void* workspace,
                                        size_t workspace_bytes, void* stream) {
  Range range_("ss_question_forward");
  FwShape F{};
  ss_status s = forward_shape(ix, n_rows, fp, &F);
  if (s != SS_OK) return s;
  if (!layers || !h_in || !q_out || !workspace)
    return fail(SS_ERR_INVALID_ARG, "NULL argument");
  if (ix->n_clustered > 0 || ix->n_windows > 0)
    return fail(SS_ERR_UNSUPPORTED, "the forward reads an uncompressed index only");
  if (ix->n_vframes != ix->n_frames)
    return fail(SS_ERR_STATE, "values are stored for %lld of %lld frames",
                (long long)ix->n_vframes, (long long)ix->n_frames);
  if (F.n_tok > 0 && !ix->vals) return fail(SS_ERR_STATE, "the index stores no values");
  const size_t need = forward_workspace_bytes(F);
  if (workspace_bytes < need)
    return fail(SS_ERR_CAPACITY, "workspace of %zu bytes < %zu needed", workspace_bytes, need);
  auto al16 = [](const void* p) { return ((uintptr_t)p & 15u) == 0u; };
  if (((uintptr_t)workspace & 255u) || !al16(h_in) || !al16(q_out) || (h_out && !al16(h_out)) ||
      (status && ((uintptr_t)status & 3u)))
    return fail(SS_ERR_INVALID_ARG, "workspace must be 256-byte aligned, h_in, q_out and h_out 16-byte aligned");
  std::vector<FwLayerW> W(F.P);
  for (int i = 0; i < F.P; ++i) {
    const ss_layer_weights& w = layers[i];
    if (!w.ln1 || !w.wqkv || !w.wo || !w.ln2 || !w.wgu || !w.wd)
      return fail(SS_ERR_INVALID_ARG, "layer %d: a weight pointer is NULL (only bqkv may be)", i);
    for (const void* p : {w.ln1, w.wqkv, w.bqkv, w.wo, w.ln2, w.wgu, w.wd})
      if (p && !al16(p)) return fail(SS_ERR_INVALID_ARG, "layer %d: weights must be 16-byte aligned", i);
    W[i] = FwLayerW{w.ln1, w.wqkv, w.bqkv, w.wo, w.ln2, w.wgu, w.wd};
  }
  FwArgs A;
  A.layers = W.data();
  A.h_in = h_in;
  A.q_out = q_out;
  A.h_out = h_out;
  A.status = status;
  A.workspace = workspace;
  SS_CUDA(cudaSetDevice(ix->device));
  const cudaError_t e = launch_forward(F, A, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    cudaGetLastError();   // a failed launch must not surface again in later calls
    return fail(SS_ERR_CUDA, "question forward: %s", cudaGetErrorString(e));
  }
  return SS_OK;
}

SS_EXPORT ss_status ss_index_compress(ss_index* ix, const ss_compress_params* cp, void* stream) {
  Range range_("ss_index_compress");
  if (!ix || !cp) return fail(SS_ERR_INVALID_ARG, "NULL argument");
  const ss_index_config& c = ix->cfg;
  const ss_compress_params& q = *cp;
  if (q.window_frames < 1 || q.window_frames % c.frames_per_unit)
    return fail(SS_ERR_INVALID_ARG, "window_frames must be a positive multiple of frames_per_unit");
  if (q.iters < 1) return fail(SS_ERR_INVALID_ARG, "iters must be >= 1");
  if (q.first_frame < 0 || q.n_frames < 0 || q.first_frame % q.window_frames ||
      q.n_frames % q.window_frames)
    return fail(SS_ERR_INVALID_ARG, "first_frame and n_frames must be multiples of window_frames");
  if (q.first_frame + q.n_frames > ix->n_frames)
    return fail(SS_ERR_INVALID_ARG, "frames [%lld, %lld) are not all appended (have %lld)",
                (long long)q.first_frame, (long long)(q.first_frame + q.n_frames),
                (long long)ix->n_frames);
  const int64_t wt = (int64_t)q.window_frames * c.tokens_per_frame;
  if (q.n_centroids < 1 || q.n_centroids > kMaxCentroids)
    return fail(SS_ERR_UNSUPPORTED, "n_centroids must be in [1, %d]", kMaxCentroids);
  if (q.n_centroids > wt) return fail(SS_ERR_UNSUPPORTED, "n_centroids > tokens per window");
  if (wt > kMaxWindowTokens)
    return fail(SS_ERR_UNSUPPORTED, "more than %d tokens per window", kMaxWindowTokens);
  if (ix->win_frames) {
    if (q.window_frames != ix->win_frames || q.n_centroids != ix->n_centroids)
      return fail(SS_ERR_INVALID_ARG, "window_frames / n_centroids differ from the first compression");
    const int64_t end = ix->win_first_frame.back() + ix->win_frames;
    if (q.first_frame < end)
      return fail(SS_ERR_INVALID_ARG, "frames before %lld are already compressed", (long long)end);
  }
  if (ix->n_clustered > 0)
    return fail(SS_ERR_STATE, "the index already clusters units (ss_index_cluster_units)");
  if (q.n_frames == 0) return SS_OK;
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  SS_CUDA(cudaSetDevice(ix->device));
  const int n_slabs = c.n_layers * c.n_kv_heads;
  const int wu = q.window_frames / c.frames_per_unit;
  if (!ix->win_frames) {
    const int64_t wcap = c.max_frames / q.window_frames;
    const int64_t n_slots = (ix->ucap + wu - 1) / wu;
    const size_t cb = (size_t)n_slabs * wcap * q.n_centroids * kHeadDim * 2;
    const size_t ab = (size_t)n_slabs * ix->ncap;
    const size_t mb = (size_t)n_slabs * wcap * q.n_centroids * wu * 4;
    const size_t sb = (size_t)n_slabs * wcap * q.n_centroids * 4;
    ix->cent = static_cast<__nv_bfloat16*>(dev_alloc(ix, cb, st));
    ix->assign = static_cast<uint8_t*>(dev_alloc(ix, ab, st));
    ix->mcnt = static_cast<int32_t*>(dev_alloc(ix, mb, st));
    ix->msize = static_cast<int32_t*>(dev_alloc(ix, sb, st));
    ix->win_u0 = static_cast<int32_t*>(dev_alloc(ix, (size_t)wcap * 4, st));
    ix->win_slot = static_cast<int32_t*>(dev_alloc(ix, (size_t)n_slots * 4, st));
    ix->kstatus = static_cast<uint32_t*>(dev_alloc(ix, 256, st));
    if (!ix->cent || !ix->assign || !ix->mcnt || !ix->msize || !ix->win_u0 || !ix->win_slot ||
        !ix->kstatus) {
      dev_free(ix, ix->cent);
      dev_free(ix, ix->assign);
      dev_free(ix, ix->mcnt);
      dev_free(ix, ix->msize);
      dev_free(ix, ix->win_u0);
      dev_free(ix, ix->win_slot);
      dev_free(ix, ix->kstatus);
      ix->cent = nullptr;
      ix->assign = nullptr;
      ix->mcnt = ix->msize = ix->win_u0 = ix->win_slot = nullptr;
      ix->kstatus = nullptr;
      return fail(SS_ERR_ALLOC, "device allocation of the cluster arrays failed");
    }
    SS_CUDA(cudaMemsetAsync(ix->win_slot, 0xff, (size_t)n_slots * 4, st));
    SS_CUDA(cudaMemsetAsync(ix->kstatus, 0, 4, st));
    ix->wcap = (int32_t)wcap;
    ix->win_frames = q.window_frames;
    ix->n_centroids = q.n_centroids;
  }
  const int n_new = (int)(q.n_frames / q.window_frames);
  SS_CUDA(launch_kmeans(ix->keys, ix->ncap, n_slabs, ix->cent, ix->assign, ix->mcnt, ix->msize,
                        ix->win_u0, ix->win_slot, ix->wcap, ix->n_windows, n_new, q.first_frame,
                        q.window_frames, c.tokens_per_frame, c.frames_per_unit, q.n_centroids,
                        q.iters, ix->kstatus, st));
  for (int j = 0; j < n_new; ++j)
    ix->win_first_frame.push_back(q.first_frame + (int64_t)j * q.window_frames);
  ix->n_windows += n_new;
  return SS_OK;
}

SS_EXPORT ss_status ss_index_cluster_units(ss_index* ix, int64_t n_units, float tau,
                                           int32_t max_clusters, void* stream) {
  Range range_("ss_index_cluster_units");
  if (!ix) return fail(SS_ERR_INVALID_ARG, "index is NULL");
  if (n_units < 0) return fail(SS_ERR_INVALID_ARG, "n_units must be >= 0");
  if (tau != tau) return fail(SS_ERR_INVALID_ARG, "tau is NaN");
  if (ix->n_windows > 0)
    return fail(SS_ERR_STATE, "the index already has k-means windows (ss_index_compress)");
  if (ix->n_clustered + n_units > ix->n_units)
    return fail(SS_ERR_INVALID_ARG, "only %lld detailed units are complete",
                (long long)(ix->n_units - ix->n_clustered));
  const ss_index_config& c = ix->cfg;
  const int D = c.n_kv_heads * kHeadDim;
  if (ix->uc_cap == 0) {
    if (max_clusters < 1 || max_clusters > ix->ucap || max_clusters > 16384)
      return fail(SS_ERR_INVALID_ARG, "max_clusters must be in [1, min(unit capacity, 16384)]");
  } else if (max_clusters != ix->uc_cap) {
    return fail(SS_ERR_INVALID_ARG, "max_clusters differs from the first clustering call");
  }
  if (n_units == 0) return SS_OK;
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  SS_CUDA(cudaSetDevice(ix->device));
  const int n_slabs = c.n_layers * c.n_kv_heads;
  const int64_t Tu = (int64_t)c.tokens_per_frame * c.frames_per_unit;
  if (ix->uc_cap == 0) {
    const int64_t cap = max_clusters;
    ix->unit_cluster = static_cast<int32_t*>(dev_alloc(ix, (size_t)ix->ucap * 4, st));
    ix->cdesc = static_cast<float*>(dev_alloc(ix, (size_t)cap * D * 4, st));
    ix->ccount = static_cast<int32_t*>(dev_alloc(ix, (size_t)cap * 4, st));
    ix->creps = static_cast<float*>(dev_alloc(ix, (size_t)cap * n_slabs * Tu * kHeadDim * 4, st));
    ix->cfirst = static_cast<int32_t*>(dev_alloc(ix, (size_t)cap * 4, st));
    ix->cprev = static_cast<int32_t*>(dev_alloc(ix, (size_t)cap * 4, st));
    ix->uc_count = static_cast<int32_t*>(dev_alloc(ix, 256, st));
    ix->uc_work = static_cast<float*>(dev_alloc(ix, (size_t)cap * 4, st));
    if (!ix->kstatus) ix->kstatus = static_cast<uint32_t*>(dev_alloc(ix, 256, st));
    if (!ix->unit_cluster || !ix->cdesc || !ix->ccount || !ix->creps || !ix->cfirst ||
        !ix->cprev || !ix->uc_count || !ix->uc_work || !ix->kstatus) {
      void** arrs[] = {(void**)&ix->unit_cluster, (void**)&ix->cdesc, (void**)&ix->ccount,
                       (void**)&ix->creps, (void**)&ix->cfirst, (void**)&ix->cprev,
                       (void**)&ix->uc_count, (void**)&ix->uc_work};
      for (void** a : arrs) {
        dev_free(ix, *a);
        *a = nullptr;
      }
      return fail(SS_ERR_ALLOC, "device allocation of the cluster arrays failed");
    }
    SS_CUDA(cudaMemsetAsync(ix->unit_cluster, 0xff, (size_t)ix->ucap * 4, st));
    SS_CUDA(cudaMemsetAsync(ix->uc_count, 0, 256, st));
    SS_CUDA(cudaMemsetAsync(ix->kstatus, 0, 4, st));
    ix->uc_cap = max_clusters;
  }
  UcJob J;
  J.desc = ix->desc;
  J.keys = ix->keys;
  J.ncap = ix->ncap;
  J.n_slabs = n_slabs;
  J.Tu = (int)Tu;
  J.D = D;
  J.u0 = (int)ix->n_clustered;
  J.n = (int)n_units;
  J.tau = tau;
  J.cap = ix->uc_cap;
  J.n_clusters = ix->uc_count;
  J.cdesc = ix->cdesc;
  J.ccount = ix->ccount;
  J.creps = ix->creps;
  J.unit_cluster = ix->unit_cluster;
  J.cfirst = ix->cfirst;
  J.cprev = ix->cprev;
  J.first_touched = ix->uc_count + 1;
  J.status = ix->kstatus;
  SS_CUDA(launch_uc_cluster(J, st));
  ix->n_clustered += n_units;
  return SS_OK;
}

SS_EXPORT ss_status ss_index_units_over_budget(const ss_index* ix, int64_t budget_bytes,
                                               int64_t near_term_units, int64_t* n_units) {
  if (!ix || !n_units) return fail(SS_ERR_INVALID_ARG, "NULL argument");
  if (budget_bytes < 0 || near_term_units < 0)
    return fail(SS_ERR_INVALID_ARG, "budget_bytes and near_term_units must be >= 0");
  const ss_index_config& c = ix->cfg;
  const int64_t unit_bytes = (int64_t)c.n_layers * c.n_kv_heads * c.tokens_per_frame *
                             c.frames_per_unit * kHeadDim * 2;
  const int64_t detailed = ix->n_units - ix->n_clustered;
  int64_t keep = budget_bytes / unit_bytes;
  if (keep < near_term_units) keep = near_term_units;
  *n_units = detailed > keep ? detailed - keep : 0;
  return SS_OK;
}

SS_EXPORT ss_status ss_select_clusters(ss_index* ix, const void* q, int32_t R, int32_t q_agg,
                                       int32_t k_l, int32_t* ids, float* scores,
                                       int32_t* count, void* stream) {
  Range range_("ss_select_clusters");
  if (!ix || !q || !ids || !scores || !count) return fail(SS_ERR_INVALID_ARG, "NULL argument");
  if (R < 1) return fail(SS_ERR_INVALID_ARG, "n_rows must be >= 1");
  if (q_agg != SS_Q_LAST && q_agg != SS_Q_MEAN_LOGIT && q_agg != SS_Q_MEAN_SOFTMAX)
    return fail(SS_ERR_INVALID_ARG, "unknown q_agg %d", q_agg);
  if (k_l < 1 || k_l > 1024) return fail(SS_ERR_UNSUPPORTED, "k_l must be in [1, 1024]");
  if (ix->uc_cap == 0) return fail(SS_ERR_STATE, "the index has no unit clusters");
  const ss_index_config& c = ix->cfg;
  UcSel S;
  S.q = static_cast<const __nv_bfloat16*>(q);
  S.P = c.n_layers;
  S.R = R;
  S.Hq = c.n_q_heads;
  S.Hkv = c.n_kv_heads;
  S.q_agg = q_agg;
  S.k_l = k_l;
  S.cdesc = ix->cdesc;
  S.n_clusters = ix->uc_count;
  S.work = ix->uc_work;
  S.ids = ids;
  S.scores = scores;
  S.count = count;
  SS_CUDA(cudaSetDevice(ix->device));
  SS_CUDA(launch_uc_select(S, ix->uc_cap, static_cast<cudaStream_t>(stream)));
  return SS_OK;
}

SS_EXPORT ss_status ss_retrieve_workspace_size(const ss_index* const* ix, int32_t n,
                                               const int32_t* R, const ss_retrieve_params* p,
                                               size_t* bytes) {
  if (!ix || !R || !bytes) return fail(SS_ERR_INVALID_ARG, "NULL argument");
  if (n < 1 || n > kMaxProbs) return fail(SS_ERR_INVALID_ARG, "n must be in [1, %d]", kMaxProbs);
  ss_status s = check_params(p);
  if (s != SS_OK) return s;
  size_t total = 0;
  for (int j = 0; j < n; ++j) {
    if (!ix[j]) return fail(SS_ERR_INVALID_ARG, "NULL index %d", j);
    if (R[j] < 1) return fail(SS_ERR_INVALID_ARG, "n_rows must be >= 1");
    total += layout_of(ix[j], R[j], p).total;
  }
  *bytes = total;
  return SS_OK;
}

SS_EXPORT ss_status ss_retrieve(ss_index* ix, const void* q, int32_t R,
                                const ss_retrieve_params* p, const ss_result* res, void* ws,
                                size_t ws_bytes, void* stream, const ss_trace* tr) {
  Range range_("ss_retrieve");
  ss_index* const arr[1] = {ix};
  const void* const qa[1] = {q};
  return retrieve_impl(arr, qa, &R, 1, p, res, ws, ws_bytes, static_cast<cudaStream_t>(stream), tr);
}

SS_EXPORT ss_status ss_retrieve_batched(ss_index* const* ix, const void* const* q,
                                        const int32_t* R, int32_t n,
                                        const ss_retrieve_params* p, const ss_result* res,
                                        void* ws, size_t ws_bytes, void* stream,
                                        const ss_trace* tr) {
  Range range_("ss_retrieve_batched");
  return retrieve_impl(ix, q, R, n, p, res, ws, ws_bytes, static_cast<cudaStream_t>(stream), tr);
}

SS_EXPORT ss_status ss_retrieve_shard(ss_index* ix, const void* q, int32_t R,
                                      const ss_retrieve_params* p, int64_t unit_begin,
                                      const ss_shard_result* out, void* ws, size_t ws_bytes,
                                      void* stream) {
  Range range_("ss_retrieve_shard");
  if (!ix || !out) return fail(SS_ERR_INVALID_ARG, "NULL argument");
  ss_status s = check_params(p);
  if (s != SS_OK) return s;
  if (p->head_agg != SS_H_PER_QHEAD || p->use_clusters)
    return fail(SS_ERR_UNSUPPORTED, "sharded retrieval needs per-query-head lists over tokens");
  if (unit_begin < 0) return fail(SS_ERR_INVALID_ARG, "unit_begin must be >= 0");
  if (!out->topk_tok || !out->topk_s || !out->list_stats || !out->unit_stats || !out->status)
    return fail(SS_ERR_INVALID_ARG, "every shard output array is required");
  const int64_t Tu = (int64_t)ix->cfg.tokens_per_frame * ix->cfg.frames_per_unit;
  if ((unit_begin + ix->ucap) * Tu > (int64_t)0x3fffffff)
    return fail(SS_ERR_UNSUPPORTED, "stream token ids past 2^30");
  // the per-list outputs go straight to the caller's arrays; the rest of ss_result is
  // the workspace's
  ss_result r{};
  r.topk_tok = out->topk_tok;
  r.list_stats = out->list_stats;
  r.status = out->status;
  const Layout l = layout_of(ix, R < 1 ? 1 : R, p);
  if (!ws || ws_bytes < l.total) return fail(SS_ERR_INVALID_ARG, "workspace too small");
  char* base = static_cast<char*>(ws);
  r.sel_units = reinterpret_cast<int32_t*>(base + l.sel);
  r.exp_units = reinterpret_cast<int32_t*>(base + l.exp_units);
  r.frames = reinterpret_cast<int32_t*>(base + l.frames);
  r.counts = reinterpret_cast<int32_t*>(base + l.counts);
  ShardOut so{unit_begin * Tu, out->topk_s, reinterpret_cast<float2*>(out->unit_stats)};
  ss_index* const arr[1] = {ix};
  const void* const qa[1] = {q};
  return retrieve_impl(arr, qa, &R, 1, p, &r, ws, ws_bytes, static_cast<cudaStream_t>(stream),
                       nullptr, &so);
}

SS_EXPORT ss_status ss_status_sync(const uint32_t* status, void* stream) {
  if (!status) return fail(SS_ERR_INVALID_ARG, "status is NULL");
  SS_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
  uint32_t v = 0;
  SS_CUDA(cudaMemcpy(&v, status, sizeof(v), cudaMemcpyDeviceToHost));
  if (v & kStatusTimeout) return fail(SS_ERR_TIMEOUT, "a bounded device-side wait gave up");
  if (v & kStatusInternal) return fail(SS_ERR_INTERNAL, "a device-side consistency check failed");
  return SS_OK;
}

SS_EXPORT ss_status ss_retrieve_host(ss_index* ix, const void* q_host, int32_t R,
                                     const ss_retrieve_params* p, const ss_host_result* out,
                                     void* ws, size_t ws_bytes, void* stream) {
  Range range_("ss_retrieve_host");
  if (!ix || !q_host || !out || !out->sel_units || !out->exp_units || !out->frames || !out->counts)
    return fail(SS_ERR_INVALID_ARG, "NULL argument");
  ss_status s = check_params(p);
  if (s != SS_OK) return s;
  if (R < 1) return fail(SS_ERR_INVALID_ARG, "n_rows must be >= 1");
  if (!ws || ((uintptr_t)ws & 255u)) return fail(SS_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  const Layout l = layout_of(ix, R, p);
  if (ws_bytes < l.total)
    return fail(SS_ERR_INVALID_ARG, "workspace too small: %zu < %zu bytes", ws_bytes, l.total);
  const ss_index_config& c = ix->cfg;
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  char* base = static_cast<char*>(ws);
  const size_t qbytes = (size_t)c.n_layers * R * c.n_q_heads * kHeadDim * 2;
  SS_CUDA(cudaSetDevice(ix->device));
  // Question rows in page-locked host memory are read by the kernels in place (the device
  // maps them; on GB300 through NVLink-C2C); pageable rows are copied into the workspace.
  const void* q_dev = nullptr;
  {
    cudaPointerAttributes a{};
    if (cudaPointerGetAttributes(&a, q_host) == cudaSuccess && a.type == cudaMemoryTypeHost &&
        a.devicePointer)
      q_dev = a.devicePointer;
    cudaGetLastError();
  }
  if (!q_dev) {
    if (p->q_agg == SS_Q_LAST) {
      // only each layer's last question row is read: one strided copy of those rows
      const size_t row = (size_t)c.n_q_heads * kHeadDim * 2;
      SS_CUDA(cudaMemcpy2DAsync(base + l.qstage + (size_t)(R - 1) * row, (size_t)R * row,
                                static_cast<const char*>(q_host) + (size_t)(R - 1) * row,
                                (size_t)R * row, row, (size_t)c.n_layers,
                                cudaMemcpyHostToDevice, st));
    } else {
      SS_CUDA(cudaMemcpyAsync(base + l.qstage, q_host, qbytes, cudaMemcpyHostToDevice, st));
    }
    q_dev = base + l.qstage;
  }
  // The selection, expansion, frames, counts and status copy are written by the kernels
  // straight into page-locked host memory that the library keeps per host thread
  // (allocated on the thread's first call, grown to the largest selection seen).
  const size_t nsel = (size_t)p->budget_units;
  const size_t nexp = nsel * (1 + p->n_prev);
  const size_t nfr = nexp * c.frames_per_unit;
  const size_t o_exp = align256(nsel * 4), o_fr = o_exp + align256(nexp * 4),
               o_cnt = o_fr + align256(nfr * 4), o_st = o_cnt + 256, span = o_st + 256;
  struct PinnedStage {
    char* p = nullptr;
    char* d = nullptr;
    size_t bytes = 0;
    ~PinnedStage() {
      if (p) cudaFreeHost(p);
    }
  };
  static thread_local PinnedStage stage;
  if (stage.bytes < span) {
    if (stage.p) cudaFreeHost(stage.p);
    stage.p = stage.d = nullptr;
    stage.bytes = 0;
    SS_CUDA(cudaHostAlloc(reinterpret_cast<void**>(&stage.p), span, cudaHostAllocMapped));
    SS_CUDA(cudaHostGetDevicePointer(reinterpret_cast<void**>(&stage.d), stage.p, 0));
    stage.bytes = span;
  }
  ss_result r{};
  r.sel_units = reinterpret_cast<int32_t*>(stage.d);
  r.exp_units = reinterpret_cast<int32_t*>(stage.d + o_exp);
  r.frames = reinterpret_cast<int32_t*>(stage.d + o_fr);
  r.counts = reinterpret_cast<int32_t*>(stage.d + o_cnt);
  r.status = reinterpret_cast<uint32_t*>(base + l.status);   // device-side atomics stay in HBM
  uint32_t* host_status = reinterpret_cast<uint32_t*>(stage.d + o_st);
  *reinterpret_cast<volatile uint32_t*>(stage.p + o_st) = 0xffffffffu;  // set by the last kernel
  {
    ss_index* const arr[1] = {ix};
    const void* const qa[1] = {q_dev};
    s = retrieve_impl(arr, qa, &R, 1, p, &r, ws, ws_bytes, st, nullptr, nullptr, host_status);
  }
  if (s != SS_OK) return s;
  SS_CUDA(cudaStreamSynchronize(st));
  const uint32_t v = *reinterpret_cast<volatile uint32_t*>(stage.p + o_st);
  if (v == 0xffffffffu) return fail(SS_ERR_INTERNAL, "the retrieval did not report its status");
  if (v & kStatusTimeout) return fail(SS_ERR_TIMEOUT, "a bounded device-side wait gave up");
  if (v & kStatusInternal) return fail(SS_ERR_INTERNAL, "a device-side consistency check failed");
  std::memcpy(out->sel_units, stage.p, nsel * 4);
  std::memcpy(out->exp_units, stage.p + o_exp, nexp * 4);
  std::memcpy(out->frames, stage.p + o_fr, nfr * 4);
  std::memcpy(out->counts, stage.p + o_cnt, 16);
  return SS_OK;
}

// ---------------------------------------------------------------------------
// Retrieval without any allocation. Some callers cannot allocate device memory at
// question time: a serving loop whose device memory is all committed to its KV cache
// pool (a cudaMalloc there can fail outright), a host that links only this C library
// and has no device allocator of its own, and latency-bound loops that cannot afford
// cudaFree's implicit device synchronisation. For them the workspace lives in the
// module's own memory: a fixed array of kStaticScratchBytes per device, reserved when
// the library's device code is loaded.
// ---------------------------------------------------------------------------
namespace {

constexpr size_t kStaticScratchBytes = size_t(64) << 20;  // 64 MiB
constexpr int kMaxStaticDevices = 64;

__device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

std::mutex g_static_mu;
void* g_static_ptr[kMaxStaticDevices] = {};
void* g_static_ctx[kMaxStaticDevices] = {};   // the context each address belongs to

// The current CUDA context (driver cuCtxGetCurrent, found through the runtime so that
// the library needs no link to the driver library).
ss_status current_context(void** ctx) {
  using Fn = CUresult (*)(CUcontext*);
  static Fn fn = nullptr;
  if (!fn) {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q{};
    const cudaError_t e = cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000,
                                                           cudaEnableDefault, &q);
    if (e != cudaSuccess || !f || q != cudaDriverEntryPointSuccess)
      return fail(SS_ERR_CUDA, "cuCtxGetCurrent is not available");
    fn = reinterpret_cast<Fn>(f);
  }
  CUcontext c = nullptr;
  if (fn(&c) != CUDA_SUCCESS || !c) return fail(SS_ERR_CUDA, "no current CUDA context");
  *ctx = c;
  return SS_OK;
}

// The scratch's device address on `dev` (which must be current). It is looked up on the
// first call in each CUDA context of the device: once per device, unless the device's
// context is destroyed and made again (cudaDeviceReset), which loads the library's
// device code again at another address.
ss_status static_scratch(int dev, void** out) {
  if (dev < 0 || dev >= kMaxStaticDevices)
    return fail(SS_ERR_UNSUPPORTED, "device %d: static scratch supports devices [0, %d)", dev,
                kMaxStaticDevices);
  std::lock_guard<std::mutex> lock(g_static_mu);
  void* ctx = nullptr;
  ss_status s = current_context(&ctx);
  if (s != SS_OK) return s;
  if (!g_static_ptr[dev] || g_static_ctx[dev] != ctx) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess)
      return fail(SS_ERR_CUDA, "cudaGetSymbolAddress(static scratch): %s", cudaGetErrorString(e));
    g_static_ptr[dev] = p;
    g_static_ctx[dev] = ctx;
  }
  *out = g_static_ptr[dev];
  return SS_OK;
}

}  // namespace

SS_EXPORT ss_status ss_retrieve_static(ss_index* ix, const void* q, int32_t R,
                                       const ss_retrieve_params* p, const ss_result* res,
                                       void* stream) {
  Range range_("ss_retrieve_static");
  if (!ix || !q || !p || !res) return fail(SS_ERR_INVALID_ARG, "NULL argument");
  ss_status s = check_params(p);
  if (s != SS_OK) return s;
  if (R < 1) return fail(SS_ERR_INVALID_ARG, "n_rows must be >= 1");
  const size_t need = layout_of(ix, R, p).total;
  if (need > kStaticScratchBytes)
    return fail(SS_ERR_CAPACITY,
                "this retrieval needs %zu bytes of workspace; the static scratch holds %zu",
                need, kStaticScratchBytes);
  SS_CUDA(cudaSetDevice(ix->device));
  void* ws = nullptr;
  s = static_scratch(ix->device, &ws);
  if (s != SS_OK) return s;
  return ss_retrieve(ix, q, R, p, res, ws, kStaticScratchBytes, stream, nullptr);
}
