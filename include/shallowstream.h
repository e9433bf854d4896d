/*
 * shallowstream.h - C ABI of a GB300 (sm_103a) library for ShallowStream's
 * query-time evidence retrieval over a shallow-layer key index
 * (arxiv 2609.02780, Sec. 4.1 "Query-Agnostic Shallow Index Construction" and
 * Sec. 4.2 "Query-Time Answering").
 *
 * The library keeps, in HBM, the bf16 keys that the shallow layers [0, P) produced
 * for every stored video unit (the full-history shallow cache, Eq. 2) plus one
 * descriptor per unit (Eq. 3). Given a question's query vectors at those layers
 * (Eq. 10) it scores every stored history key, turns the scores into attention
 * weights, keeps the top-k tokens of every list (Eq. 11), counts each unit's votes,
 * ranks a pool of units by votes and attention mass, picks a diverse subset by
 * greedy max-min in descriptor space and adds each pick's preceding units (Eq. 12).
 * An optional k-means compression replaces windows of frames by centroids that
 * retrieval scores instead of the windows' tokens.
 *
 * Conventions for every call:
 *   - Returns an ss_status; nothing throws or aborts across the ABI. On failure the
 *     call has launched nothing and ss_last_error() (thread-local) describes why.
 *   - "device" pointers are CUDA device (or managed) addresses on the index's
 *     device; "host" pointers are CPU addresses. Pointers are borrowed, never freed.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream). Calls that launch
 *     work are asynchronous: outputs are valid once the stream reaches that point.
 *   - Device memory for an index comes only from the ss_allocator given at create
 *     time (or cudaMalloc/cudaFree when it is NULL). Per-call scratch is the caller's
 *     `workspace` buffer (size from ss_retrieve_workspace_size).
 *   - Key and query layouts are bf16, row-major, head_dim contiguous; only
 *     head_dim == 128 and n_q_heads / n_kv_heads <= 8 are supported.
 *   - A handle must not be used by two host threads at once.
 *
 * Notation: P shallow layers, Hq query heads, Hkv key heads, G = Hq / Hkv (query
 * head h reads key head h / G), d = 128, T_f tokens per frame, T_u = T_f *
 * frames_per_unit tokens per unit, U stored units, token id p = unit * T_u + slot.
 */
#ifndef SHALLOWSTREAM_H
#define SHALLOWSTREAM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SS_OK = 0,
  SS_ERR_INVALID_ARG = 1,   /* a NULL, negative, misaligned or inconsistent argument */
  SS_ERR_UNSUPPORTED = 2,   /* valid request outside the supported shapes */
  SS_ERR_CAPACITY = 3,      /* index capacity (max_frames) or a buffer is too small */
  SS_ERR_STATE = 4,         /* call not allowed in the handle's current state */
  SS_ERR_ALLOC = 5,         /* the allocator returned NULL */
  SS_ERR_CUDA = 6,          /* a CUDA runtime call failed (message in ss_last_error) */
  SS_ERR_TIMEOUT = 7,       /* a bounded device-side wait gave up (device status) */
  SS_ERR_INTERNAL = 8       /* a device-side consistency check failed (device status) */
} ss_status;

typedef struct ss_index ss_index;  /* opaque; host-side metadata only */

/* Device memory provider. alloc returns a device pointer aligned to 256 bytes (or
 * NULL); free releases it. `stream` is the stream passed to the call that
 * allocates; `ctx` is passed through. */
typedef struct {
  void* (*alloc)(size_t bytes, void* stream, void* ctx);
  void (*free)(void* ptr, void* stream, void* ctx);
  void* ctx;
} ss_allocator;

/* Shape and capacity of an index (Sec. 3 notation; Table 4: a unit is 2 frames for
 * Qwen3-VL and 1 for LLaVA-OneVision). */
typedef struct {
  int32_t n_layers;          /* P >= 1, the shallow layers [0, P) */
  int32_t n_q_heads;         /* Hq, multiple of n_kv_heads, Hq / Hkv <= 8 */
  int32_t n_kv_heads;        /* Hkv, 1..8 */
  int32_t head_dim;          /* d, must be 128 */
  int32_t tokens_per_frame;  /* T_f >= 1 visual tokens per frame */
  int32_t frames_per_unit;   /* >= 1 */
  int64_t max_frames;        /* capacity in frames, a multiple of frames_per_unit */
} ss_index_config;

/* Read-only view of an index's state and device arrays (for inspection). */
typedef struct {
  int64_t n_frames;          /* frames appended so far */
  int64_t n_units;           /* complete units (descriptors valid for [0, n_units)) */
  int64_t token_capacity;    /* N_cap tokens per (layer, key head) slab */
  const void* keys;          /* device bf16 [P][Hkv][N_cap][d] */
  const float* descriptors;  /* device fp32 [U_cap][Hkv * d] */
  int32_t n_windows;         /* compressed windows so far */
  int32_t window_frames;     /* 0 until the first compression */
  int32_t n_centroids;
  const void* centroids;     /* device bf16 [P][Hkv][W_cap * n_centroids][d] or NULL */
  const uint8_t* assignment; /* device uint8 [P][Hkv][N_cap]: centroid of each token of a
                                compressed window (window-local id) or NULL */
  const int32_t* window_first_unit; /* device int32 [W_cap] or NULL */
  const int32_t* member_counts; /* device int32 [P][Hkv][W_cap][n_centroids][window units]:
                                   members of each centroid in each unit of its window */
  const int32_t* member_sizes;  /* device int32 [P][Hkv][W_cap][n_centroids] */
  /* long-history compression (ss_index_cluster_units) */
  int64_t n_clustered_units;    /* units [0, n) have left the detailed window */
  int32_t cluster_capacity;     /* 0 until the first clustering */
  const int32_t* unit_cluster;  /* device int32 [U_cap]: cluster of a clustered unit, -1 */
  const int32_t* cluster_count; /* device int32 [1]: clusters so far */
  const float* cluster_centroids; /* device fp32 [capacity][Hkv * d] (unit norm) */
  const int32_t* cluster_sizes; /* device int32 [capacity] members */
  const float* cluster_keys;    /* device fp32 [capacity][P][Hkv][T_u][d] representative keys */
  /* stored values (ss_index_append_values), read by the question's forward only */
  const void* values;           /* device bf16 [P][Hkv][N_cap][d] or NULL */
  int64_t n_value_frames;       /* frames whose values are stored */
} ss_index_view;

/* k-means compression of the frames [first_frame, first_frame + n_frames) in
 * windows of window_frames (see ss_index_compress). */
typedef struct {
  int32_t window_frames;     /* frames per window, a multiple of frames_per_unit */
  int32_t n_centroids;       /* 1..128 and <= window_frames * T_f (<= 65536 tokens) */
  int32_t iters;             /* Lloyd rounds >= 1 */
  int64_t first_frame;       /* multiple of window_frames */
  int64_t n_frames;          /* multiple of window_frames */
} ss_compress_params;

/* Which question rows attend (Sec. 4.2 uses the final prompt token):
 *   SS_Q_LAST         the last row;
 *   SS_Q_MEAN_LOGIT   the rows' mean (fp32 sum in row order / R, rounded to bf16): its
 *                     logit is the rows' mean logit;
 *   SS_Q_MEAN_SOFTMAX every row attends on its own; a list's weight of a token is the
 *                     mean over the rows of the rows' softmax weights, and the list ranks
 *                     tokens by it (two passes over the keys: each row's softmax
 *                     statistics, then the weights; per-query-head lists over tokens only,
 *                     R <= 64 and (Hq / Hkv) * (R rounded up to 16) <= 512). */
typedef enum { SS_Q_LAST = 0, SS_Q_MEAN_LOGIT = 1, SS_Q_MEAN_SOFTMAX = 2 } ss_q_agg;
typedef enum { SS_H_PER_QHEAD = 0, SS_H_MEAN = 1 } ss_head_agg;

/* Evidence-selection parameters (Sec. 4.2; Table 4 gives k = 64, pool 32 = 4 x 8,
 * K = 8, one preceding unit, 6 recent units). */
typedef struct {
  int32_t k;                 /* top-k tokens per list, 1..4096 */
  int32_t budget_units;      /* K units chosen by max-min, >= 1 */
  int32_t pool_mult;         /* pool = pool_mult * K (paper: 4), pool <= 1024 */
  int32_t n_prev;            /* preceding units added per selected unit (paper: 1) */
  int32_t n_recent_units;    /* N_r: the latest N_r units are recent, never scored (Eq. 4) */
  int32_t q_agg;             /* ss_q_agg: which question row(s) form the query */
  int32_t head_agg;          /* ss_head_agg: per-query-head lists or one list per layer */
  int32_t use_clusters;      /* 1: compressed windows are scored by their centroids */
} ss_retrieve_params;

/* Outputs of one retrieval, in caller-owned device buffers. A NULL member is placed in
 * the workspace instead (and is then overwritten by the next call). n_lists = P * Hq
 * for SS_H_PER_QHEAD, P for SS_H_MEAN. U_cap = max_frames / frames_per_unit. */
typedef struct {
  int32_t* topk_tok;         /* [n_lists][k] candidate ids sorted by (score desc, id asc);
                                token id p, or 0x40000000 + window * n_c + centroid for a
                                centroid; -1 past the number of candidates */
  float* topk_w;             /* [n_lists][k] normalised attention weight of each entry
                                (SS_H_MEAN: the head-averaged weight alpha;
                                SS_Q_MEAN_SOFTMAX: the row-averaged weight) */
  float* list_stats;         /* [n_lists][2] softmax stats (M, L): M = max over candidates
                                of the log2-scaled score s * log2(e), L = sum 2^(s' - M)
                                (SS_H_MEAN, SS_Q_MEAN_SOFTMAX: M = max weight,
                                L = sum of the weights = 1) */
  int32_t* unit_votes;       /* [U_cap] votes of each history unit */
  float* unit_mass;          /* [U_cap] attention mass of each history unit */
  int32_t* pool;             /* [pool_mult * K] vote-ranked pool, best first */
  int32_t* sel_units;        /* [K] max-min picks in selection order (required) */
  int32_t* exp_units;        /* [K * (1 + n_prev)] picks plus predecessors, ascending
                                (required) */
  int32_t* frames;           /* [K * (1 + n_prev) * frames_per_unit] frames of exp_units,
                                ascending (required) */
  int32_t* counts;           /* [4] n_pool, n_sel, n_exp, n_frames (required) */
  uint32_t* status;          /* [1] device status word, 0 = ok (required) */
} ss_result;

/* Host-side outputs of ss_retrieve_host (plain host arrays, pinned or not). */
typedef struct {
  int32_t* sel_units;        /* [K] */
  int32_t* exp_units;        /* [K * (1 + n_prev)] */
  int32_t* frames;           /* [K * (1 + n_prev) * frames_per_unit] */
  int32_t* counts;           /* [4] as in ss_result */
} ss_host_result;

/* Device outputs of one shard of a retrieval over an index split by token range (see
 * ss_retrieve_shard). n_lists = P * Hq; Uh = the shard's history units. */
typedef struct {
  int32_t* topk_tok;         /* [n_lists][k] the shard's top-k tokens per list, stream token
                                ids (shard unit u is stream unit unit_begin + u), sorted by
                                (score desc, id asc); -1 past the shard's tokens */
  float* topk_s;             /* [n_lists][k] their log2-scaled scores s * log2(e);
                                -infinity past the shard's tokens */
  float* list_stats;         /* [n_lists][2] (M, L) over the shard's history tokens, as in
                                ss_result */
  float* unit_stats;         /* [n_lists][Uh][2] (m, l) over each history unit's tokens:
                                m = max s * log2(e), l = sum 2^(s * log2(e) - m) */
  uint32_t* status;          /* [1] device status word (required) */
} ss_shard_result;

/* One shard's payload as the merge reads it (host arrays). */
typedef struct {
  int64_t unit_begin;        /* stream unit of the shard's first history unit */
  int32_t n_units;           /* the shard's history units */
  const int32_t* topk_tok;   /* [n_lists][k] as ss_shard_result */
  const float* topk_s;       /* [n_lists][k] */
  const float* list_stats;   /* [n_lists][2] */
  const float* unit_stats;   /* [n_lists][n_units][2] */
  const float* desc;         /* [n_units][desc_dim] the units' descriptors (Eq. 3) */
} ss_shard;

/* Host outputs of ss_merge_shards; sizes as ss_result's with U = the stream's history
 * units (the shards' n_units summed). All required. */
typedef struct {
  int32_t* topk_tok;         /* [n_lists][k] */
  float* topk_w;             /* [n_lists][k] */
  float* list_stats;         /* [n_lists][2] */
  int32_t* unit_votes;       /* [U] */
  float* unit_mass;          /* [U] */
  int32_t* pool;             /* [min(pool_mult * K, U)] */
  int32_t* sel_units;        /* [K] */
  int32_t* exp_units;        /* [K * (1 + n_prev)] */
  int32_t* frames;           /* [K * (1 + n_prev) * frames_per_unit] */
  int32_t* counts;           /* [4] n_pool, n_sel, n_exp, n_frames */
} ss_merge_result;

/* The question's forward through the shallow layers (ss_question_forward). */
typedef struct {
  int32_t intermediate;      /* I, the MLP width: a positive multiple of 128 */
  float rms_eps;             /* RMSNorm epsilon, > 0 */
  float rope_theta;          /* RoPE base theta, > 1 */
  int64_t pos0;              /* position of question row 0; < 0: the stored token count
                                (the question follows the retained history) */
} ss_forward_params;

/* One shallow layer's weights: device bf16, row-major, 16-byte aligned. D = Hq * d. */
typedef struct {
  const void* ln1;           /* [D] RMSNorm weight before attention */
  const void* wqkv;          /* [(Hq + 2 Hkv) d][D]: q rows (head-major), k rows, v rows */
  const void* bqkv;          /* [(Hq + 2 Hkv) d] projection bias, or NULL for none */
  const void* wo;            /* [D][Hq d] output projection */
  const void* ln2;           /* [D] RMSNorm weight before the MLP */
  const void* wgu;           /* [2 I][D]: gate rows, then up rows */
  const void* wd;            /* [D][I] down projection */
} ss_layer_weights;

/* Optional instrumentation: cudaEvent_t handles recorded on the call's stream
 * immediately before and after the key-scoring kernel. NULL members are skipped. */
typedef struct {
  void* score_begin;
  void* score_end;
} ss_trace;

/* --------------------------------------------------------------------------- */

/* Human-readable name of a status code (static storage). */
const char* ss_status_string(ss_status s);

/* Message of the last failed call on this host thread (static, thread-local). */
const char* ss_last_error(void);

/* Library version string. */
const char* ss_version(void);

/* Creates an empty index (Eq. 2 with T = 0) on the current CUDA device. Allocates
 * the key slabs bf16 [P][Hkv][max_frames * T_f][d] and descriptors fp32
 * [U_cap][Hkv * d] from `alloc` (NULL: cudaMalloc). `stream` is passed to alloc.
 * Errors: INVALID_ARG (NULL out/config, non-positive sizes, Hq % Hkv != 0,
 * max_frames % frames_per_unit != 0), UNSUPPORTED (head_dim != 128, Hq / Hkv > 8,
 * Hkv > 8), ALLOC, CUDA. *out is NULL on failure. */
ss_status ss_index_create(const ss_index_config* config, const ss_allocator* alloc,
                          void* stream, ss_index** out);

/* Frees the index's device memory through its allocator and the handle. The caller
 * must make sure no queued work still uses the index. NULL is accepted. */
ss_status ss_index_destroy(ss_index* index);

/* Appends n_frames frames of shallow keys (Eq. 1-2: the keys K^i_t of each new unit at
 * every shallow layer). `keys` is device bf16 laid out [P][Hkv][S][d] where S =
 * slab_stride_tokens (0 means n_frames * T_f) and the first n_frames * T_f tokens of
 * every (layer, key head) slab are appended in order. Computes the Eq. 3 descriptor of
 * every unit that this call completes. Asynchronous on `stream`; `keys` must stay valid
 * until the stream passes this call. Errors: INVALID_ARG (NULL keys with n_frames > 0,
 * negative n_frames, stride < n_frames * T_f, keys not 16-byte aligned), CAPACITY
 * (would exceed max_frames), CUDA. n_frames == 0 is a no-op. */
ss_status ss_index_append(ss_index* index, const void* keys, int32_t n_frames,
                          int64_t slab_stride_tokens, void* stream);

/* Fills *view with the index's current state. Device arrays are owned by the index. */
ss_status ss_index_get_view(const ss_index* index, ss_index_view* view);

/* Stores the values that the shallow layers produced for the next n_frames frames
 * whose keys are already stored (the layer-i KV cache C^i_T of Eq. 10 holds keys and
 * values; only the question's forward reads the values). `values` is device bf16
 * [P][Hkv][slab_stride_tokens][d], the key layout of ss_index_append (stride 0 =
 * n_frames * T_f). The first call allocates [P][Hkv][N_cap][d] from the index's
 * allocator. Errors: INVALID_ARG, STATE (values past the stored keys), ALLOC, CUDA. */
ss_status ss_index_append_values(ss_index* index, const void* values, int32_t n_frames,
                                 int64_t slab_stride_tokens, void* stream);

/* Bytes of device workspace ss_question_forward needs for this index, row count and
 * parameters (depends on the stored token count through the attention's chunking: take
 * it again after appends). Errors as ss_question_forward's argument checks. */
ss_status ss_forward_workspace_size(const ss_index* index, int32_t n_rows,
                                    const ss_forward_params* params, size_t* bytes);

/* The question's forward through the shallow layers (Sec. 4.2, Eq. 10): the question's
 * R embedded rows `h_in` (device bf16 [R][D], D = Hq * d) pass through layers [0, P),
 * each a pre-norm GQA decoder layer with the caller's weights `layers` [P]:
 *   x = bf16(RMSNorm(H) * ln1);  [q; k; v] = x Wqkv^T + bqkv
 *   q, k = bf16(RoPE(q, k)) at positions pos0 + r (rotate-half pairs (j, j + d/2),
 *          angle pos * theta^(-2j/d), computed in fp64), v = bf16(v)
 *   o = softmax(q k^T / sqrt(d)) v over the layer's stored tokens (their keys and values
 *       as stored) and the question's rows 0..r, query head h reading key head h / G
 *   H += bf16(o) Wo^T;  x2 = bf16(RMSNorm(H) * ln2);  H += bf16(silu(x2 Wg^T) * (x2 Wu^T)) Wd^T
 * Outputs: q_out (device bf16 [P][R][Hq][d]) = each layer's post-RoPE query rows Q^i,
 * the retrieval's input layout (ss_retrieve's q); h_out (device fp32 [R][D], or NULL) =
 * the hidden states after layer P - 1. H is carried in fp32; products run on the tensor
 * cores in bf16 with fp32 accumulation; attention weights are rounded to bf16 for the
 * tensor cores and normalised by the sum of the rounded weights. `status` (device word,
 * or NULL for one in the workspace) records SS_ERR_TIMEOUT as in ss_status_sync.
 * Needs R <= 64, (Hq / Hkv) * (R rounded up to 16) <= 256, values stored for every
 * stored frame, and an index without compressed windows or clusters.
 * Errors: INVALID_ARG (NULL, misaligned, bad parameters), UNSUPPORTED, STATE (values
 * missing, compressed index), CAPACITY (workspace too small), CUDA. */
ss_status ss_question_forward(ss_index* index, const ss_layer_weights* layers,
                              const ss_forward_params* params, const void* h_in,
                              int32_t n_rows, void* q_out, float* h_out, uint32_t* status,
                              void* workspace, size_t workspace_bytes, void* stream);

/* The index's shape (as given to ss_index_create). Host-only. */
ss_status ss_index_get_config(const ss_index* index, ss_index_config* config);

/* Checkpoint of an index: writes its host metadata and every device array (keys, values,
 * descriptors, compressed windows, unit clusters, at their full capacity) to the host file
 * `path`, through a page-locked staging buffer on `stream` (the call returns when the file
 * is written). The file is for this library version and a machine of the same byte order.
 * Errors: INVALID_ARG (NULL, the file cannot be written), ALLOC, CUDA. */
ss_status ss_index_save(const ss_index* index, const char* path, void* stream);

/* Recreates an index from a file of ss_index_save on the current device, its device memory
 * from `alloc` (NULL: cudaMalloc); the loaded index behaves as the saved one (appends,
 * compression, retrieval continue from its state). Errors: INVALID_ARG (not such a file,
 * truncated or inconsistent), ALLOC (nothing is kept), CUDA. */
ss_status ss_index_load(const char* path, const ss_allocator* alloc, void* stream,
                        ss_index** out);

/* k-means compression of already appended frames (the cluster-compressed variant;
 * closest paper text Sec. 4.1 Eq. 5-7). For every window of `window_frames` frames in
 * [first_frame, first_frame + n_frames) and every (layer, key head): X = the window's
 * keys, C0 = X's first n_centroids tokens, then `iters` Lloyd rounds (assign each key
 * to the nearest centroid by squared L2, lowest id on ties; move each centroid to the
 * fp32 mean of its members, empty ones unchanged). Stores the last round's centroids
 * (bf16, nearest-even) and memberships. Distances are compared as ||c||^2 - 2 x . c in
 * fp32 (x . c on the tensor cores with c split into two bf16 parts), so a key whose two
 * nearest centroids are within that rounding of each other may take either; the sums
 * of the update run in a fixed order (results repeat bit for bit). The first call fixes
 * window_frames and
 * n_centroids (later calls must match, with windows after those already compressed)
 * and allocates the cluster arrays from the index's allocator.
 * With n_centroids <= 64 and windows of <= 16384 tokens the rounds run on the tcgen05
 * tensor cores (one read of the window's keys per round; member sums accumulated by the
 * tensor cores in a fixed order), otherwise on mma.sync tensor cores. A device-side wait
 * of the compression that gives up (SS_ERR_TIMEOUT) is reported in the status word of
 * every later retrieval on the index.
 * Errors: INVALID_ARG (misaligned ranges, frames not yet appended, overlap with a
 * compressed window), UNSUPPORTED (n_centroids > 128 or > window tokens, windows of more
 * than 65536 tokens), ALLOC (nothing is kept; the call can be repeated), CUDA. */
ss_status ss_index_compress(ss_index* index, const ss_compress_params* params,
                            void* stream);

/* The paper's long-history compression (Sec. 4.1, Eq. 6-7): the next n_units oldest
 * detailed units leave the detailed window, in order. A leaving unit t joins the latest
 * cluster C_j when its descriptor k_t (Eq. 3) satisfies k_t . c_j >= tau, and then
 * c_j <- Norm((n_j c_j + k_t) / (n_j + 1)); otherwise it starts the next cluster with
 * c = k_t (the first unit to leave starts cluster 0). Each cluster keeps representative
 * keys, the running average (n K + K_t) / (n + 1) of its members' keys at every (layer,
 * key head, token slot of a unit, dim), in fp32. Retrieval then scores only the detailed
 * units (the clustered ones get no votes and no mass; a selected unit's predecessor is
 * added only if it is detailed), and ss_select_clusters gives the cluster evidence.
 * Decisions use fp32 dot products reduced in a fixed order, so repeated calls give the
 * same clusters. The first call fixes max_clusters (1..16384, at most the unit capacity)
 * and allocates fp32 [max_clusters][P][Hkv][T_u][d] for the representatives. More
 * clusters than that raise SS_ERR_INTERNAL in the status of later retrievals.
 * Errors: INVALID_ARG (n_units beyond the complete detailed units, NaN tau, another
 * max_clusters), STATE (the index has k-means windows), ALLOC, CUDA. */
ss_status ss_index_cluster_units(ss_index* index, int64_t n_units, float tau,
                                 int32_t max_clusters, void* stream);

/* Eq. 5 as a budget on the detailed units' keys: *n_units = how many of the oldest
 * detailed units must leave the detailed window so that the detailed keys fit
 * budget_bytes, never taking units from the latest near_term_units (the near-term and
 * recent context). Host-only. */
ss_status ss_index_units_over_budget(const ss_index* index, int64_t budget_bytes,
                                     int64_t near_term_units, int64_t* n_units);

/* The cluster evidence of a question (Sec. 4.2, Eq. 13): every cluster's centroid scored
 * against the query state of the last shallow layer, score_j = (1/Hq) sum_h
 * q_h . c_j[h / G] / sqrt(d), with q_h the last question row (SS_Q_LAST) or the rows'
 * mean rounded to bf16 (the other readings), and c_j[g] the 128 entries of key head g;
 * then the first min(k_l, clusters) clusters by (score desc, id asc). Device outputs:
 * ids [k_l] (-1 past the count), scores [k_l], count [1]. Errors: INVALID_ARG, STATE (no
 * clusters), UNSUPPORTED (k_l outside [1, 1024]), CUDA. */
ss_status ss_select_clusters(ss_index* index, const void* q, int32_t n_rows, int32_t q_agg,
                             int32_t k_l, int32_t* ids, float* scores, int32_t* count,
                             void* stream);

/* Bytes of device workspace that ss_retrieve_batched needs for these indexes, row
 * counts and parameters (ss_retrieve: n = 1). Depends on the indexes' capacities, not
 * their current fill, so one workspace serves every later call with the same params. */
ss_status ss_retrieve_workspace_size(const ss_index* const* indexes, int32_t n,
                                     const int32_t* n_rows,
                                     const ss_retrieve_params* params, size_t* bytes);

/* One question against one index (Sec. 4.2, Eq. 10-12; the retrieval gate of Eq. 9 is
 * taken as open). `q` is device bf16 [P][R][Hq][d], the question's post-RoPE query rows
 * at each shallow layer (Eq. 10). History = units [0, U - n_recent_units) (Eq. 4). For
 * each list (layer i, query head h): s_p = q_eff . K^i_{h/G, p} / sqrt(d) over the
 * history tokens, w = softmax(s), the top-k tokens by (s desc, id asc) (Eq. 11). Unit
 * votes count (list, selected token) pairs per unit; the pool is the top
 * min(pool_mult * K, |history|) units by (votes desc, mass desc, id asc) where mass is
 * the summed weight of all the unit's tokens over all lists; max-min diversity over the
 * pool's descriptors (start at the pool's best, then repeatedly the unit farthest, by
 * 1 - cosine, from its nearest pick; ties to the better pool rank) picks min(K, pool)
 * units; each pick and its n_prev predecessors, deduplicated and ascending, form
 * exp_units and frames (Eq. 12). With SS_H_MEAN the lists are per layer, ranked by the
 * mean over query heads of the per-head weights. With SS_Q_MEAN_SOFTMAX every question
 * row attends on its own and a list ranks tokens by the mean of the rows' weights. With
 * use_clusters, compressed
 * windows contribute their centroids as candidates instead of their tokens (only with
 * SS_H_PER_QHEAD); a selected centroid votes once per member token and its weight is
 * shared among member units by member count. These two modes keep every candidate's
 * score in the workspace (P * Hq rows of N_cap floats) and rank dense rows; the
 * default mode keeps only a running superset of each list's top k.
 * Errors: INVALID_ARG (NULL, R < 1, bad enums, workspace too small or misaligned),
 * UNSUPPORTED (k > 4096, pool > 1024, history > 16384 units, head_agg with clusters),
 * STATE (use_clusters without compression), CUDA. Device-side failures are reported
 * in *result->status (read with ss_status_sync). */
ss_status ss_retrieve(ss_index* index, const void* q, int32_t n_rows,
                      const ss_retrieve_params* params, const ss_result* result,
                      void* workspace, size_t workspace_bytes, void* stream,
                      const ss_trace* trace);

/* n independent questions against n indexes (all on one device, same params) in one
 * launch per stage: q[j] has n_rows[j] rows for indexes[j], results[j] receives its
 * outputs. 1 <= n <= 32. Errors as ss_retrieve. */
ss_status ss_retrieve_batched(ss_index* const* indexes, const void* const* q,
                              const int32_t* n_rows, int32_t n,
                              const ss_retrieve_params* params, const ss_result* results,
                              void* workspace, size_t workspace_bytes, void* stream,
                              const ss_trace* trace);

/* ss_retrieve from host memory. `q_host` (bf16 [P][R][Hq][d]) in page-locked memory is
 * read by the kernels in place through the device's mapping of it (on GB300 over
 * NVLink-C2C; only the rows the query reading needs are read); pageable rows are first
 * copied into the workspace (under SS_Q_LAST only each layer's last row). The
 * selection, expansion, frames and counts are written by the kernels directly into
 * page-locked host memory that the library keeps per host thread (allocated with
 * cudaHostAlloc on the thread's first call, grown to the largest selection seen),
 * then unpacked into `out` once `stream` is synchronized. Returns the device status
 * as well (TIMEOUT or INTERNAL). Errors as ss_retrieve. */
ss_status ss_retrieve_host(ss_index* index, const void* q_host, int32_t n_rows,
                           const ss_retrieve_params* params, const ss_host_result* out,
                           void* workspace, size_t workspace_bytes, void* stream);

/* ss_retrieve with no allocation and no caller workspace (the paper has no
 * counterpart: this is a deployment entry point). For callers that cannot allocate
 * device memory at question time: a serving loop whose device memory is committed to
 * its KV cache pool, where a cudaMalloc can fail; a host linking only this library,
 * with no device allocator of its own; a latency-bound loop that cannot take cudaFree's
 * implicit device synchronisation. The workspace is a fixed 64 MiB array in the
 * library's device memory (one per device, reserved when the library's device code is
 * loaded). The first call on each device looks up that array's address with the
 * device current (one-time set-up, repeated only if the device's context is destroyed
 * and made again, as cudaDeviceReset does); make that first call before any stream
 * capture.
 * Nothing in the scratch has to start at zero: the first kernel of every call resets
 * the counters that later kernels accumulate into. Every call on a device uses the same
 * scratch, so calls that overlap (other streams or host threads on that device, before
 * the previous call's kernels have finished) race and give wrong results: order them,
 * e.g. on one stream. Outputs as ss_retrieve; the result arrays are the caller's.
 * Errors as ss_retrieve, plus CAPACITY when the call's workspace (the size
 * ss_retrieve_workspace_size reports for n = 1) exceeds 64 MiB, and UNSUPPORTED on a
 * device ordinal >= 64. */
ss_status ss_retrieve_static(ss_index* index, const void* q, int32_t n_rows,
                             const ss_retrieve_params* params, const ss_result* result,
                             void* stream);

/* Sets how long the key-scoring kernel's waits for its key copies may take before
 * they give up: `polls` polls of the copy's barrier (each wait also gives up after about
 * one second), or -1 for the default (2^26 polls). A wait that gives up records
 * SS_ERR_TIMEOUT in the retrieval's status word, lets its copies in flight land and
 * ends its warp; the retrieval's later kernels then skip their work and leave the
 * counts at 0. 0 makes every such wait give up at once, which makes the failure path
 * testable without a fault. Process-wide; takes effect for retrievals issued after the
 * call. Errors: INVALID_ARG (polls < -1 or >= 2^32). */
ss_status ss_set_wait_limit(int64_t polls);

/* One shard of a retrieval over a stream whose history is split by unit range across
 * GPUs, each GPU holding the keys of its range in its own index (appended in order; its
 * unit 0 is stream unit unit_begin). The shard scores its own history keys exactly as
 * ss_retrieve does (Sec. 4.2) and stops after each list's top-k (Eq. 11), writing to
 * `out` its top-k tokens with their scores, its list statistics and its per-(list, unit)
 * statistics; with those, ss_merge_shards finishes the retrieval on one host. A token of
 * a list's global top-k is always in the top-k of its shard, and a list's (M, L) and a
 * unit's attention mass combine exactly from the shards' statistics, so the merged
 * result is the unsharded one (up to floating-point rounding). The shard's n_recent_units
 * counts its own latest units (0 except on the shard that holds the stream's latest
 * units). Only per-query-head lists over tokens (head_agg SS_H_PER_QHEAD, use_clusters 0)
 * are supported. `workspace` as ss_retrieve's (same size). Errors as ss_retrieve, plus
 * UNSUPPORTED for other list kinds. */
ss_status ss_retrieve_shard(ss_index* index, const void* q, int32_t n_rows,
                            const ss_retrieve_params* params, int64_t unit_begin,
                            const ss_shard_result* out, void* workspace,
                            size_t workspace_bytes, void* stream);

/* Merges the payloads of n_shards shards (host arrays, shards in stream order, their
 * history unit ranges tiling [0, U)) into the retrieval of the whole stream, on the host:
 * per list the first k of the shards' candidates by (score desc, id asc) and their
 * weights under the list's combined softmax statistics (M, L), the unit votes, the units'
 * attention mass (each unit's per-list statistics under the list's combined (M, L)), the
 * vote-ranked pool, max-min diversity over the descriptors and the expansion, with the
 * same rules as ss_retrieve (Sec. 4.2, Eq. 11-12). The merge's arithmetic is fp64.
 * Errors: INVALID_ARG (NULL, shards not tiling the history in order, a token outside its
 * shard), UNSUPPORTED (head_agg or use_clusters set). Runs on the calling thread; needs
 * no GPU. */
ss_status ss_merge_shards(const ss_shard* shards, int32_t n_shards, int32_t n_lists,
                          int32_t tokens_per_unit, int32_t frames_per_unit, int32_t desc_dim,
                          const ss_retrieve_params* params, const ss_merge_result* out);

/* Synchronizes `stream` and returns the status recorded in the device word `status`
 * by earlier retrievals on it (SS_OK, SS_ERR_TIMEOUT or SS_ERR_INTERNAL). */
ss_status ss_status_sync(const uint32_t* status, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SHALLOWSTREAM_H */
