// Internal declarations shared by the library's CUDA translation units.
//
// Every retrieval stage is one kernel launch over a batch of independent problems
// (one question against one index). The batch travels by value as a __grid_constant__
// kernel parameter, so launches need no host-to-device copy and can be captured in a
// CUDA graph.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <map>
#include <mutex>
#include <utility>

#include "shallowstream.h"

namespace ss {

// Records a printf-style message as the calling thread's last error (ss_last_error) and
// returns `s`.
ss_status fail_status(ss_status s, const char* fmt, ...);

constexpr int kHeadDim = 128;          // d (only 128 is supported)
constexpr int kMaxProbs = 32;          // problems per batched launch
constexpr int kMaxK = 4096;            // top-k per list
constexpr int kMaxPool = 1024;         // pool = pool_mult * budget
constexpr int kMaxHistUnits = 16384;   // history units per problem (pool sort in smem)
constexpr int kMaxGroup = 8;           // query heads per key head
constexpr uint32_t kCentroidIdBase = 0x40000000u;
constexpr int kMaxCentroids = 128;     // per window (k-means compression)
constexpr int kMaxWindowTokens = 65536;

// Score-kernel geometry: kScoreWarps compute warps + 2 threshold warps per CTA (each
// threshold warp serves half of the group's lists).
#ifndef SS_SCORE_WARPS
#define SS_SCORE_WARPS 8
#endif
constexpr int kScoreWarps = SS_SCORE_WARPS;
constexpr int kThresholdWarps = 2;
constexpr int kScoreThreads = (kScoreWarps + kThresholdWarps) * 32;
#ifndef SS_SCORE_CTAS_PER_SM
#define SS_SCORE_CTAS_PER_SM 2
#endif
constexpr int kScoreCtasPerSm = SS_SCORE_CTAS_PER_SM;
#ifndef SS_SCORE_STAGES
#define SS_SCORE_STAGES 2
#endif
constexpr int kScoreStages = SS_SCORE_STAGES;  // bulk-copy stages per compute warp
constexpr int kTileRows = 16;                  // key rows per stage (one MMA tile)
constexpr int kTileBytes = kTileRows * kHeadDim * 2;
// Threshold ladder of each list: level i counts appended scores in
// [A + (i - kLadderZero) / kLadderPerUnit, + 1 / kLadderPerUnit) where A is the list's
// anchor (largest score of a small key sample); the top level also takes everything
// above. kLadderLevels levels span [A - 12, A + 4) log2 units.
constexpr int kLadderLevels = 256;
constexpr int kLadderZero = 192;
constexpr float kLadderPerUnit = 16.0f;
constexpr int kSampleUnits = 4;        // history units scored for the ladder anchor
// Candidate slots a warp reserves per list at a time (no atomic per append).
constexpr int kReserve = 64;
constexpr int kMaxChunksPerSlab = 128;
// Words between two slabs' unit counters of the score kernel (one 128-byte line each).
constexpr int kUnitCounterStride = 32;

// Device status word bits (ss_result::status).
constexpr uint32_t kStatusInternal = 1u;
constexpr uint32_t kStatusTimeout = 2u;
// Polls after which a bounded wait gives up (it also gives up after ~1 s).
constexpr uint32_t kDefaultWaitPolls = 1u << 26;

// log2(e) / sqrt(128): scores are kept in the log2 domain, s2 = (q.k) * kScoreScale,
// so softmax weights are 2^(s2 - M) / L.
constexpr float kScoreScale = 0.12751743082459868f;

struct Prob {
  // index
  const __nv_bfloat16* keys;   // [P*Hkv][ncap][d]
  const float* desc;           // [ucap][Hkv*d]
  int64_t ncap;                // token capacity per slab
  int P, Hq, Hkv, G, Tu, fpu;
  int U;                       // complete units
  int Uh;                      // history units [0, Uh)
  int ucap;
  // question
  const __nv_bfloat16* q;      // [P][R][Hq][d]
  int R;
  // workspace
  __nv_bfloat16* qeff;         // [P][Hq][d]
  float2* cand_pair;           // [n_score_lists][cand_cap] (score, id bits): the score
                               // kernel's appended candidates
  float* cand_s;               // [n_score_lists][cand_cap] dense rows (general path),
  int32_t* cand_id;            // over the same memory as cand_pair
  int64_t cand_cap;
  int32_t* cand_cnt;           // [n_score_lists]
  uint32_t* gthr;              // [n_score_lists] ordered-float threshold
  int32_t* ladder;             // [n_score_lists][kLadderLevels] appended-score counts
  float* samp_max;             // [n_score_lists][kSampleUnits] maxima of the sampled units
  int n_sample;                // sampled units Z (0..kSampleUnits)
  float2* ustats;              // [n_score_lists][ucap] per-unit (max, sum 2^(s-max))
  int32_t* next_unit;          // [P*Hkv][kUnitCounterStride] next history unit to score
                               // in each slab (word 0 of each line)
  float* gram;                 // packed upper triangle of the pool's Gram matrix
  // outputs
  int32_t* topk_tok;           // [n_lists][k]
  float* topk_w;
  float* topk_s;               // [n_lists][k] log2-scaled scores of the list, or NULL
  float2* list_ml;             // [n_lists] (M, L)
  int32_t* votes;              // [ucap]
  float* mass;                 // [ucap]
  int32_t* pool;
  int32_t* sel;
  int32_t* exp_units;
  int32_t* frames;
  int32_t* counts;             // n_pool, n_sel, n_exp, n_frames
  uint32_t* status;
  uint32_t* host_status;       // copy of the final status word in mapped host memory, or NULL
  // general path (one list per layer, or centroids of compressed windows as candidates):
  // every candidate is scored into a dense row per list
  int n_cand;                  // candidates per list
  int n_raw_tok;               // of which raw history tokens (the rest are centroids)
  int n_c, wu, wcap;           // centroids per window, units per window, window capacity
  const __nv_bfloat16* cent;   // [P*Hkv][wcap*n_c][d]
  const int32_t* mcnt;         // [P*Hkv][wcap][n_c][wu]
  const int32_t* msize;        // [P*Hkv][wcap][n_c]
  const int32_t* win_slot;     // [ucap / wu] window of each window slot or -1
  const int32_t* win_u0;       // [wcap] first unit of each window
  const uint32_t* index_status;  // device word of the index's compressions, or NULL
  int32_t* raw_units;          // [ucap] history units not covered by a window, ascending
  int32_t* raw_rank;           // [ucap] position of a unit in raw_units, or -1
  float* cw;                   // [P*Hkv][wcap*n_c] summed weight of each centroid over
                               // the G lists of its slab
  int32_t* csel;               // [P*Hkv][wcap*n_c] lists of its slab that selected each
                               // centroid
  float2* head_ml;             // [P*Hq] (M, L) of each head's softmax (one list per layer)
  float2* rm_scratch;          // row-averaged lists: per-row softmax statistics
  int rm_chunks;               // CTAs per slab of the row-averaged passes
  float* aval;                 // [P][cand_cap] head-averaged weight of every token
  // an index with clustered units: the view above starts at its first detailed unit
  int unit_offset;             // clustered units before it (0: none)
  int32_t* votes_base;         // the caller's votes / mass arrays in stream numbering
  float* mass_base;
  // launch mapping of the score kernel
  int cta_begin;               // first score CTA of this problem
  int chunks;                  // score CTAs per slab (they share the slab's units)
  int pool_n;                  // min(pool_mult * budget, Uh)
  int n_sel;                   // min(budget, pool_n)
};

struct Batch {
  Prob p[kMaxProbs];
  int n;
  int k;
  int n_prev;
  int q_agg;                   // 0 last row, 1 row mean, 2 mean of the rows' softmaxes
  int head_agg;
  int use_clusters;
  int score_ctas;              // total CTAs of the score kernel
  int score_spread;            // 1: one wave; slab = CTA index mod slabs
  uint32_t wait_polls;         // limit of the score kernel's waits for its key copies
};
static_assert(sizeof(Batch) <= 32000, "kernel parameter block too large");

// Online clustering of units leaving the detailed window (one call).
struct UcJob {
  const float* desc;           // [ucap][D]
  const __nv_bfloat16* keys;   // [n_slabs][ncap][d]
  int64_t ncap;
  int n_slabs, Tu, D;
  int u0, n;                   // the units leaving, in order
  float tau;
  int cap;                     // cluster capacity
  int32_t* n_clusters;         // device count
  float* cdesc;                // [cap][D] centroids
  int32_t* ccount;             // [cap] members
  float* creps;                // [cap][n_slabs][Tu][d] representative keys
  int32_t* unit_cluster;       // [ucap]
  int32_t* cfirst;             // [cap] first member unit in the current call
  int32_t* cprev;              // [cap] members before the current call
  int32_t* first_touched;      // device: the first cluster the call touched
  uint32_t* status;            // device status word of the index
};

// Cluster evidence of a question (Eq. 13).
struct UcSel {
  const __nv_bfloat16* q;      // [P][R][Hq][d]
  int P, R, Hq, Hkv, q_agg, k_l;
  const float* cdesc;
  const int32_t* n_clusters;
  float* work;                 // [cap] scores
  int32_t* ids;                // [k_l]
  float* scores;               // [k_l]
  int32_t* count;              // [1]
};

// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t float_to_ordered(float f) {
  uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float ordered_to_float(uint32_t o) {
  uint32_t u = (o & 0x80000000u) ? (o & 0x7fffffffu) : ~o;
  return __uint_as_float(u);
}

// 2^x with the SFU's approximate exp2 (flushes denormal results to zero).
__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Combines two (max, sum of 2^(s - max)) pairs; an empty pair has max = -inf, sum 0.
__device__ __forceinline__ void ml_combine(float& m, float& l, float mo, float lo) {
  float M = fmaxf(m, mo);
  float a = (m == -INFINITY) ? 0.f : l * fast_exp2(m - M);
  float b = (mo == -INFINITY) ? 0.f : lo * fast_exp2(mo - M);
  m = M;
  l = a + b;
}

// Ladder anchor A of list L: the largest sampled score (0 if nothing was sampled).
__device__ __forceinline__ float list_anchor(const Prob& P, int L) {
  float a = -INFINITY;
  for (int z = 0; z < P.n_sample; ++z) a = fmaxf(a, P.samp_max[L * kSampleUnits + z]);
  return (a == -INFINITY || a != a) ? 0.f : a;
}

// Programmatic dependent launch: every retrieval kernel may start while its predecessor
// in the stream drains. pdl_wait() blocks until the predecessor grid has completed and
// its writes are visible; pdl_release() lets the successor start launching.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_release() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// True when an earlier kernel of this retrieval gave up a bounded wait: the later
// kernels then skip their work (the caller reads SS_ERR_TIMEOUT from the status word).
// Read after pdl_wait(): no kernel that runs at the same time writes the word.
__device__ __forceinline__ bool retrieval_timed_out(const Prob& P) {
  return (*(volatile const uint32_t*)P.status & kStatusTimeout) != 0u;
}

__device__ __forceinline__ int problem_of_block(const Batch& B, int b) {
  int pi = 0;
  while (pi + 1 < B.n && B.p[pi + 1].cta_begin <= b) ++pi;
  return pi;
}

}  // namespace ss

// Launchers (host side), one per translation unit.
namespace ss {
// Launches `kernel` with programmatic stream serialization (see pdl_wait).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
// Raises a kernel's dynamic shared-memory limit (and sets its carveout, when asked) on
// the current device, once per larger size: the attributes persist in the context, so a
// call that needs no more than an earlier one costs a map lookup instead of driver calls.
inline cudaError_t ensure_smem(const void* kernel, int bytes, int carveout = -1) {
  static std::mutex mu;
  static std::map<std::pair<const void*, int>, int> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  auto it = done.find({kernel, dev});
  if (it != done.end() && it->second >= bytes) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) return e;
  if (carveout >= 0) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, carveout);
    if (e != cudaSuccess) return e;
  }
  done[{kernel, dev}] = bytes;
  return cudaSuccess;
}
cudaError_t launch_prep(const Batch& B, cudaStream_t s);
int sample_units(int k, int tokens_per_unit, int hist_units);
cudaError_t launch_score(const Batch& B, cudaStream_t s);
cudaError_t launch_select(const Batch& B, int max_lists, int sm_count, cudaStream_t s);
cudaError_t launch_select_general(const Batch& B, int max_lists, int sm_count, cudaStream_t s);
cudaError_t launch_general_score(const Batch& B, int max_cand, int max_slabs,
                                 int max_score_lists, cudaStream_t s);
cudaError_t launch_mass_general(const Batch& B, int max_cent, int max_slabs,
                                int max_hist_units, cudaStream_t s);
cudaError_t launch_mass(const Batch& B, int max_hist_units, cudaStream_t s);

cudaError_t launch_pool(const Batch& B, int max_hist_units, cudaStream_t s);
bool rowmean_supported(int R, int G);
size_t rowmean_workspace_bytes(int n_slabs, int R, int G, int max_chunks);
int rowmean_chunks(int n_slabs, int hist_tokens, int sm_count);
cudaError_t launch_rowmean(const Batch& B, int pi, float2* scratch, int chunks, cudaStream_t s);
cudaError_t launch_uc_shift(const Batch& B, cudaStream_t s);
cudaError_t launch_uc_cluster(const UcJob& J, cudaStream_t s);
cudaError_t launch_uc_select(const UcSel& S, int cap, cudaStream_t s);
cudaError_t launch_shard_export(const Batch& B, int64_t tok_offset, float2* unit_stats,
                                cudaStream_t s);
cudaError_t launch_maxmin(const Batch& B, int max_pool, cudaStream_t s);
cudaError_t launch_append(__nv_bfloat16* keys, int64_t ncap, int64_t tok0,
                          const __nv_bfloat16* src, int64_t src_stride_tokens,
                          int n_slabs, int64_t n_tokens, cudaStream_t s);
size_t kmeans_smem_bytes(int n_c, int window_tokens);
cudaError_t launch_kmeans(const __nv_bfloat16* keys, int64_t ncap, int n_slabs,
                          __nv_bfloat16* cent, uint8_t* assign, int32_t* mcnt, int32_t* msize,
                          int32_t* win_u0, int32_t* win_slot, int wcap, int w_begin, int n_new,
                          int64_t first_frame, int window_frames, int tokens_per_frame,
                          int frames_per_unit, int n_c, int iters, uint32_t* status,
                          cudaStream_t s);
cudaError_t launch_descriptors(const __nv_bfloat16* keys, int64_t ncap, int P, int Hkv,
                               int Tu, int64_t u_begin, int64_t u_end, float* desc,
                               cudaStream_t s);
int score_chunks_per_slab(int n_slabs_total, int hist_units, int sm_count);
int score_slots(int sm_count);

// The question's forward through the shallow layers (ss_forward.cu).
struct FwShape {
  int P, Hq, Hkv, R, I;
  int64_t ncap;                 // tokens per slab of the index's arrays
  int n_tok;                    // stored tokens per slab
  int sm_count;
  float eps;
  double theta;
  int64_t pos0;
  const void* keys;             // bf16 [P][Hkv][ncap][d]
  const void* values;           // bf16 [P][Hkv][ncap][d]
};
struct FwLayerW {
  const void *ln1, *wqkv, *bqkv, *wo, *ln2, *wgu, *wd;
};
struct FwArgs {
  const FwLayerW* layers;       // [P]
  const void* h_in;             // bf16 [R][D]
  void* q_out;                  // bf16 [P][R][Hq][d]
  float* h_out;                 // fp32 [R][D] or NULL
  uint32_t* status;             // device word or NULL (then in the workspace)
  void* workspace;
};
bool forward_supported(int R, int Hq, int Hkv);
size_t forward_workspace_bytes(const FwShape& F);
cudaError_t launch_forward(const FwShape& F, const FwArgs& A, cudaStream_t st);
}  // namespace ss
