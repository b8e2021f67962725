/*
 * mpcache.h - C ABI of the GB300 (sm_103a) MPCache decode path.
 *
 * MPCache (arXiv 2501.06807) shrinks the attention of LLM decoding in four
 * steps; each step is one call of this library:
 *
 *   mpc_static_evict        look-once static eviction at prefill (Sec. 3.2,
 *                           Alg. 2 Step 1)
 *   mpc_build_clusters      token gathering of the kept set into a
 *                           cluster-major cache plus the hierarchical cluster
 *                           summaries r_max, r_min and the reordered
 *                           representative of Eq. 3 (Sec. 3.3)
 *   mpc_select              per decode step: MPC-friendly similarity (Eq. 3)
 *                           and hierarchical top-k over the clusters, for the
 *                           leader layer of a cross-layer sharing group
 *                           (Sec. 3.3-3.4, Alg. 2 Step 2)
 *   mpc_sparse_decode_attn  per decode step: append the new k, v, then
 *                           softmax(q K'^T / sqrt(d)) V' over the selected
 *                           clusters and the tail (Alg. 1)
 *
 * mpc_decode_step runs the last two for every layer of one decode step in
 * one call (two launches, or one fused kernel; mpc_decode_step_plan says
 * which).  mpc_layer_refs lays out the cross-layer sharing groups (Sec. 3.4),
 * mpc_commonality measures the commonality of per-layer selections (Sec. 2,
 * Observation 3) and mpc_choose_share_every turns it into a group size.
 *
 * Conventions shared by every call
 * --------------------------------
 * - Pointers named "device" are CUDA device pointers owned by the caller; the
 *   library never allocates, frees or retains them past the call.  Scratch
 *   space is the caller's too: `*_workspace_size` reports how many bytes a
 *   call needs and the call receives them as `workspace`.  A workspace must
 *   be 16-byte aligned and zero-filled once before its first use; the calls
 *   that keep counters in it leave them zero, so it can be reused as is,
 *   except after a call whose bounded wait gave up (flag 1 of
 *   mpc_device_status): zero-fill the workspace again before reusing it.
 * - Every call is asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *   default stream) and returns once its kernels are queued.  Arguments are
 *   validated on the host before anything is launched.
 * - Tensors are row-major with the head dimension d innermost.  `dtype` is
 *   MPC_F32 or MPC_BF16 and applies to queries, keys, values and the
 *   cluster-major cache; summaries, scores and outputs are float32.
 * - One call may process several layers.  `refs[i]` names, for the i-th
 *   processed layer, its index along every per-layer tensor of the call
 *   (`layer`, scaled by that tensor's layer stride), its index along every
 *   per-group tensor (`group`: kept sets, summaries, selections) and whether
 *   it leads the group (`leader`, Sec. 3.4: the leader computes the shared
 *   indices, the other layers of the group reuse them).
 * - Ratios are integers in parts per million.  A count derived from a ratio
 *   r over N items is min(N, max(1, ceil(N r / 1e6))), 0 when N = 0.
 * - Return value: MPC_OK, or a negative MPC_ERR_* code; mpc_last_error()
 *   gives a thread-local message for the last failing call of the thread.
 *
 * Cluster-major cache (output of mpc_build_clusters, read and appended to
 * by mpc_sparse_decode_attn): per (layer, sequence, kv head) `cap_tokens`
 * rows of d elements.  Row i is the i-th kept token in position order,
 * followed by the tokens appended by decode steps.  Cluster c (finest level)
 * is rows [c s, (c + 1) s); the rows after the last full cluster form the
 * tail.  Inside a row the 16-byte chunks are permuted: logical chunk j of
 * row i is stored at chunk j ^ (i & 7).  The permutation keeps the
 * decode kernel's shared-memory reads free of bank conflicts.
 *
 * Summary pyramid (per group, sequence, kv head): `summary_rows` rows of d
 * float32.  Level 1 (clusters of s tokens) starts at row 0 and has
 * cap_1 = cap_tokens / s rows; level l + 1 starts after level l and has
 * cap_{l+1} = ceil(cap_l / fanout[l]) rows.  Three such arrays hold r_max,
 * r_min and rep = alpha r_max + (1 - alpha) r_min.
 */
#ifndef MPCACHE_H
#define MPCACHE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define MPC_API __attribute__((visibility("default")))

#define MPC_ABI_VERSION 7
#define MPC_MAX_LEVELS 4
#define MPC_MAX_REFS 128

enum mpc_status {
  MPC_OK = 0,
  MPC_ERR_INVALID_ARG = -1,   /* NULL pointer, bad enum, struct_size mismatch */
  MPC_ERR_BAD_SHAPE = -2,     /* a size or ratio outside the supported range */
  MPC_ERR_WORKSPACE = -3,     /* workspace NULL or smaller than reported */
  MPC_ERR_CUDA = -4           /* a CUDA launch or attribute call failed */
};

enum mpc_dtype { MPC_F32 = 0, MPC_BF16 = 1 };

/* Cluster similarity of mpc_select. */
enum mpc_sim_metric { MPC_SIM_EQ3 = 0, MPC_SIM_BOUND = 1, MPC_SIM_MEAN = 2, MPC_SIM_FXP = 3 };

typedef struct {
  int32_t layer;   /* index along per-layer tensors */
  int32_t group;   /* index along per-group tensors */
  int32_t leader;  /* nonzero if this layer computes the group's indices */
} mpc_layer_ref;

/* Prompt K or V of the processed layers, dense or paged.  Element
 * (layer l, sequence b, kv head h, position t, channel c) lives at
 *   dense: data + l*layer_stride + ((b*n_kv_heads + h)*t_max + t)*d + c
 *   paged: data + l*layer_stride
 *               + ((page_table[b*max_pages + t/page_size]*n_kv_heads + h)
 *                  *page_size + t%page_size)*d + c
 * (offsets in elements of the call's dtype). */
typedef struct {
  const void* data;            /* device */
  int64_t layer_stride;        /* elements between consecutive layers */
  const int32_t* page_table;   /* device [batch][max_pages], NULL = dense */
  int32_t page_size;           /* tokens per page (paged only) */
  int32_t max_pages;           /* page-table row length (paged only) */
} mpc_kv_tensor;

/* ---- mpc_static_evict ----------------------------------------------------
 * Look-once static eviction (Sec. 3.2; Alg. 2 Step 1; App. E "Static
 * eviction").  For every leader ref, sequence b and kv head h:
 *   w_b     = ceil(T_b * rho_w), rho_w = long_window_ppm if T_b >
 *             long_prompt_threshold else window_ppm (20% / 10% above 24k)
 *   score_j = sum over the group's query heads g and window rows i of
 *             softmax_{j' <= p_i}(q_{g,i} . k_{j'} * scale)_j,
 *             p_i = T_b - w_b + i (causal attention map of the last rows)
 *   kept    = the n_keep_b = count(T_b, keep_ppm) positions of highest score
 *             (equal scores: lower position first), in ascending order.
 * Outputs: out_scores[group][b][h][t_max] (positions >= T_b undefined),
 * out_kept[group][b][h][keep_cap] (entries >= n_keep_b are -1) and
 * out_n_keep[b].  Refs must all be leaders.  Workspace: the window rows'
 * statistics and, for paged bf16 keys, a dense copy of the refs' keys
 * (n_refs * batch * n_kv_heads * t_max * d * 2 bytes) gathered before the
 * tensor-core passes. */
typedef struct {
  uint32_t struct_size;        /* sizeof(mpc_static_args) */
  int32_t n_refs;
  const mpc_layer_ref* refs;   /* host [n_refs] */
  int32_t batch, n_q_heads, n_kv_heads, head_dim, dtype;
  int32_t t_max;               /* prompt capacity, >= every T_b */
  const int32_t* prompt_lens;  /* device [batch], 1 <= T_b <= t_max */
  const void* q_win;           /* device [layer][batch][n_q_heads][win_rows][d];
                                  row r is prompt position T_b - win_rows + r */
  int64_t q_win_layer_stride;  /* elements */
  int32_t win_rows;            /* >= every w_b */
  mpc_kv_tensor k;             /* device memory: host memory is refused (INVALID_ARG) */
  int32_t window_ppm, long_window_ppm, long_prompt_threshold;
  int32_t keep_ppm;
  float scale;                 /* 0 selects 1/sqrt(d) */
  int32_t keep_cap;            /* >= every n_keep_b */
  float* out_scores;           /* device */
  int32_t* out_kept;           /* device */
  int32_t* out_n_keep;         /* device [batch] */
} mpc_static_args;

/* ---- mpc_build_clusters --------------------------------------------------
 * Token gathering of the kept set (Alg. 2 Step 1, token_gather) into the
 * cluster-major cache, and the summary pyramid of the leaders (Sec. 3.3:
 * r_max / r_min of each cluster, the Eq. 3 representative; hierarchical
 * clustering: level l + 1 groups fanout[l] consecutive level-l clusters and
 * its r_max / r_min are taken over all member tokens).  Only the
 * floor(n_keep_b / s) full clusters get summaries; the remaining rows are the
 * tail.  For every ref: rows [0, n_keep_b) of its cache are written from the
 * kept positions of its group; leaders also write their group's pyramid.
 * out_n_tok[b] = n_keep_b starts the decode counter. */
typedef struct {
  uint32_t struct_size;        /* sizeof(mpc_cluster_args) */
  int32_t n_refs;
  const mpc_layer_ref* refs;   /* host [n_refs] */
  int32_t batch, n_kv_heads, head_dim, dtype;
  int32_t t_max;
  mpc_kv_tensor k, v;          /* prompt keys and values; data may also be pinned
                                  host memory (device-accessible under unified
                                  addressing): only the kept rows are read */
  const int32_t* kept;         /* device [group][batch][n_kv_heads][keep_cap] */
  int32_t keep_cap;
  const int32_t* n_keep;       /* device [batch] */
  void* kc;                    /* device cluster-major keys [layer][batch][n_kv_heads][cap_tokens][d] */
  void* vc;                    /* device cluster-major values, same layout */
  int64_t cache_layer_stride;  /* elements between layers of kc / vc */
  int32_t cap_tokens;          /* multiple of cluster_size, >= n_keep_b + decode steps */
  float* r_max;                /* device [group][batch][n_kv_heads][summary_rows][d] */
  float* r_min;
  float* rep;
  int32_t summary_rows;
  int32_t cluster_size;        /* s */
  int32_t n_levels;            /* 1 .. MPC_MAX_LEVELS */
  int32_t fanout[MPC_MAX_LEVELS]; /* fanout[l] >= 2 for l < n_levels - 1 */
  float alpha;                 /* Eq. 3 weight, default 0.6 */
  int32_t* out_n_tok;          /* device [batch] */
  float* mean;                 /* optional device pyramid like rep: the mean member key of
                                  every cluster (the average-key baseline); NULL skips it */
} mpc_cluster_args;

/* ---- mpc_select ----------------------------------------------------------
 * Dynamic selection of one decode step for leader layers (Sec. 3.3-3.4; Alg.
 * 2 Step 2, Sim + topk).  With C_1 = floor(n_tok_b / s) sealed clusters and
 * C_{l+1} = ceil(C_l / fanout[l]), for every ref, sequence b and kv head h,
 * with q = the sum of the group's query heads:
 *   metric MPC_SIM_EQ3:   sim(c) = q . rep_c                          (Eq. 3)
 *   metric MPC_SIM_BOUND: sim(c) = sum_i max(q_i r_max_ci, q_i r_min_ci) (Eq. 2)
 *   metric MPC_SIM_MEAN:  sim(c) = q . mean_c, the mean member key (App. G baseline)
 *   metric MPC_SIM_FXP:   Eq. 3 evaluated in the fixed-point ring Z_{2^64} of
 *     the MPC runtime (App. B), emulated on plaintext values: with f =
 *     frac_bits, enc(x) = rint(x 2^f) (ties to even) as a two's-complement
 *     int64, tr(y) = floor(y / 2^f) (arithmetic shift), sums and products
 *     modulo 2^64:
 *       q_i   = sum_g enc(q_gi)
 *       rep_i = tr(enc(alpha) enc(r_max_ci)) + tr(enc(1 - alpha) enc(r_min_ci))
 *       sim   = tr(sum_i q_i rep_i), saturated to int32 and ranked as an integer
 *     (1 - alpha taken in double precision from the float alpha; every
 *     |value| must stay below 2^(62 - f), as an encoding needs)
 *   the coarsest level ranks all of its clusters; every finer level ranks
 *   the children of the clusters its parent level kept; level l keeps
 *   k_l = count(C_l, level_keep_ppm[l]) (at most its candidates); equal
 *   similarities rank the lower id first.
 * out_sel[group][b][h][sel_cap] gets the kept finest-level ids ascending
 * (entries >= out_n_sel[b] are -1).  n_tok is read-only here. */
typedef struct {
  uint32_t struct_size;        /* sizeof(mpc_select_args) */
  int32_t n_refs;
  const mpc_layer_ref* refs;   /* host [n_refs], all leaders */
  int32_t batch, n_q_heads, n_kv_heads, head_dim, dtype;
  const void* q;               /* device [layer][batch][n_q_heads][d] */
  int64_t q_layer_stride;      /* elements */
  const float* rep;            /* device [group][batch][n_kv_heads][summary_rows][d] */
  int32_t summary_rows;
  int32_t cap_tokens;
  const int32_t* n_tok;        /* device [batch] cache rows before this step's append */
  int32_t cluster_size, n_levels;
  int32_t fanout[MPC_MAX_LEVELS];
  int32_t level_keep_ppm[MPC_MAX_LEVELS]; /* finest level first */
  int32_t sel_cap;             /* >= every k_1 */
  int32_t* out_sel;            /* device */
  int32_t* out_n_sel;          /* device [batch] */
  int32_t metric;              /* MPC_SIM_EQ3 (0), _BOUND (1), _MEAN (2) or _FXP (3) */
  const float* r_max;          /* device, laid out like rep; read for MPC_SIM_BOUND / _FXP */
  const float* r_min;          /* device, laid out like rep; read for MPC_SIM_BOUND / _FXP */
  const float* mean;           /* device, laid out like rep; read for MPC_SIM_MEAN only */
  float alpha;                 /* MPC_SIM_FXP: Eq. 3 weight in [0, 1] */
  int32_t frac_bits;           /* MPC_SIM_FXP: fractional bits f in [1, 24] */
} mpc_select_args;

/* ---- mpc_sparse_decode_attn ----------------------------------------------
 * One decode step of attention for every ref (Alg. 1; Alg. 2 Step 2,
 * gather + sparse attention; App. A decode append).  With n = n_tok_b and
 * C_1 = floor(n / s):
 *   1. k_new, v_new are written to row n of the layer's cache (append);
 *   2. o_g = softmax(q_g K'^T * scale) V' over the rows of the selected
 *      clusters of the ref's group (sel, n_sel) and the tail rows
 *      [C_1 s, n] (which include the appended row);
 *   3. if the tail now holds s rows it is sealed as cluster C_1: leaders
 *      write its r_max / r_min / rep and merge it into the coarser levels;
 *   4. if `advance` is nonzero, n_tok[b] += 1 once all refs are done.
 * A sequence with no row left for the append (n + 1 > cap_tokens) is
 * skipped on the device: nothing is written, n_tok[b] stays, and the device
 * status word gets flag 2 (see mpc_device_status).
 * Outputs o[layer][b][n_q_heads][d] float32. */
typedef struct {
  uint32_t struct_size;        /* sizeof(mpc_attn_args) */
  int32_t n_refs;
  const mpc_layer_ref* refs;   /* host [n_refs] */
  int32_t batch, n_q_heads, n_kv_heads, head_dim, dtype;
  const void* q;               /* device [layer][batch][n_q_heads][d] */
  const void* k_new;           /* device [layer][batch][n_kv_heads][d] */
  const void* v_new;
  int64_t q_layer_stride, kv_new_layer_stride;   /* elements */
  void* kc;                    /* device cluster-major cache (in/out) */
  void* vc;
  int64_t cache_layer_stride;
  int32_t cap_tokens;
  const int32_t* sel;          /* device [group][batch][n_kv_heads][sel_cap] */
  const int32_t* n_sel;        /* device [batch] */
  int32_t sel_cap;
  float* r_max;                /* device pyramid (in/out, leaders only); */
  float* r_min;                /* may be NULL when no ref is a leader    */
  float* rep;
  int32_t summary_rows;
  int32_t cluster_size, n_levels;
  int32_t fanout[MPC_MAX_LEVELS];
  float alpha;
  int32_t* n_tok;              /* device [batch] */
  int32_t advance;
  float scale;                 /* 0 selects 1/sqrt(d) */
  float* out;                  /* device [layer][batch][n_q_heads][d] */
  int64_t out_layer_stride;    /* elements */
  float* mean;                 /* optional mean pyramid (in/out) kept current when a tail is
                                  sealed; NULL skips it */
} mpc_attn_args;

/* Workspace byte counts (0 is a valid answer).  Same validation as the
 * calls; the pointer fields of `args` may be NULL here. */
MPC_API int mpc_static_evict_workspace_size(const mpc_static_args* args, size_t* bytes);
MPC_API int mpc_build_clusters_workspace_size(const mpc_cluster_args* args, size_t* bytes);
MPC_API int mpc_select_workspace_size(const mpc_select_args* args, size_t* bytes);
MPC_API int mpc_sparse_decode_attn_workspace_size(const mpc_attn_args* args, size_t* bytes);

MPC_API int mpc_static_evict(const mpc_static_args* args, void* workspace,
                             size_t workspace_bytes, void* stream);
MPC_API int mpc_build_clusters(const mpc_cluster_args* args, void* workspace,
                               size_t workspace_bytes, void* stream);
MPC_API int mpc_select(const mpc_select_args* args, void* workspace,
                       size_t workspace_bytes, void* stream);
MPC_API int mpc_sparse_decode_attn(const mpc_attn_args* args, void* workspace,
                                   size_t workspace_bytes, void* stream);

/* ---- mpc_decode_step -----------------------------------------------------
 * One whole decode step (Alg. 2 Step 2) in one call: for every leader ref the
 * hierarchical selection of mpc_select, then for every ref the append and
 * sparse attention of mpc_sparse_decode_attn over the selection of its group
 * (Sec. 3.4: the leader computes the indices, the other layers of the group
 * reuse them).  The selections and outputs are those of mpc_select followed
 * by mpc_sparse_decode_attn with the same arguments: the same similarity
 * arithmetic and ranking, so the same ids; the attention sums the same rows
 * in another order, so o agrees to fp32 rounding.
 * - attn: the arguments of mpc_sparse_decode_attn (attn.struct_size =
 *   sizeof(mpc_attn_args)); attn.sel / attn.n_sel are OUTPUTS here, written
 *   like mpc_select's out_sel / out_n_sel for every group of the call.  Every
 *   ref's group must have its leader among the refs (one leader per group),
 *   and the summary pyramid the metric reads must be given (rep for
 *   MPC_SIM_EQ3, mean for MPC_SIM_MEAN, r_max / r_min for MPC_SIM_BOUND and
 *   MPC_SIM_FXP; r_max, r_min and rep are also updated by the seal).
 * - level_keep_ppm, metric, frac_bits: as in mpc_select_args (alpha is
 *   attn.alpha).
 * - speculate: -1 automatic, 0 or 1: whether the selection's first round
 *   also scores every cluster of the level below the coarsest (one
 *   dependent round fewer, more rows read); both forms of the step.
 * - static_ppm, slice_tiles: the attention's tile list is cut into one
 *   contiguous range per warp for its first static_ppm parts per million,
 *   the rest into slices of slice_tiles tiles that warps claim once their
 *   range is done (a balance for SMs that stream slower); 1e6 keeps every
 *   tile static; 0 picks either.  (Fused kernel only.)
 * - fuse: 0: two launches, mpc_select's kernel followed by
 *   mpc_sparse_decode_attn's (with programmatic stream serialization, so the
 *   attention kernel becomes resident while the selection runs); 1: one
 *   persistent kernel for the whole step where it applies (bf16 caches, the
 *   EQ3 / BOUND / MEAN metrics, at most 1024 candidates at a level), else
 *   the two launches; -1 (automatic): the fused kernel for 305 to 1216
 *   selection units (leader refs x batch x kv heads), the two launches
 *   otherwise.  Measured on GB300 (us per step, two launches / fused): 8k
 *   GQA, 80 units, 23.2 / 25.3; 32k GQA, 80 units, 31.7 / 35.2; 2k MHA, 544
 *   units, 32.1 / 31.2; paged batch 1, 544 units, 42.4 / 39.5; batch 4,
 *   2176 units, 90.5 / 96.2; batch 32, 17408 units, 693 / 700.
 *   mpc_decode_step_plan reports which form a call takes.
 * In the fused kernel, selection teams publish each unit's ids in the
 * workspace (each word tagged with the call) and the attention warps wait
 * for them (bounded, 1 s; a wait that gives up sets flag 1 of
 * mpc_device_status and the call's outputs are undefined).
 * Workspace: mpc_decode_step_workspace_size bytes, zero-filled once; the
 * call leaves it ready for the next call, except after a wait that gave up
 * (flag 1 of mpc_device_status): zero-fill it again before the next call. */
typedef struct {
  uint32_t struct_size;        /* sizeof(mpc_decode_args) */
  mpc_attn_args attn;
  int32_t level_keep_ppm[MPC_MAX_LEVELS]; /* finest level first */
  int32_t metric;              /* MPC_SIM_EQ3, _BOUND, _MEAN or _FXP */
  int32_t frac_bits;           /* MPC_SIM_FXP only */
  int32_t speculate;           /* -1 = automatic */
  int32_t static_ppm;          /* share of the attention tiles in static warp ranges; 0 = automatic */
  int32_t slice_tiles;         /* tiles per dynamically claimed slice of the rest; 0 = automatic */
  int32_t fuse;                /* 1 = one fused kernel, 0 = selection + attention launches, -1 = automatic */
} mpc_decode_args;

MPC_API int mpc_decode_step_workspace_size(const mpc_decode_args* args, size_t* bytes);
/* Validates like mpc_decode_step and writes the kernel launches the call
 * makes (1: the fused kernel, 2: selection then attention); host only. */
MPC_API int mpc_decode_step_plan(const mpc_decode_args* args, int32_t* launches);
MPC_API int mpc_decode_step(const mpc_decode_args* args, void* workspace, size_t workspace_bytes,
                            void* stream);

/* ---- mpc_sparse_decode_attn_static_scratch --------------------------------
 * The same decode step as mpc_sparse_decode_attn, for callers that cannot
 * allocate device memory (a runtime that forbids raw cudaMalloc, a plugin
 * that only receives fixed input/output buffers, a path that must not
 * allocate after start-up).  The paper has no counterpart: it is a property
 * of this library's interface, not of the method.
 * - Scratch is a 4 MiB array inside the library's device image, held by every
 *   GPU that loads the library until the process exits.  A call whose
 *   workspace (mpc_sparse_decode_attn_workspace_size) exceeds 4 MiB is
 *   rejected with MPC_ERR_WORKSPACE and nothing is launched.
 * - Every call looks up the array's device address in the current device's
 *   context (cudaGetSymbolAddress), clears the counters it keeps in the
 *   array (an asynchronous memset on `stream`) and then runs the regular
 *   kernels.  Every call shares the one array: calls that overlap on the GPU
 *   (different streams, no ordering between them) race and corrupt each
 *   other's results.
 * - Allocates nothing (no cudaMalloc / cudaFree). */
MPC_API int mpc_sparse_decode_attn_static_scratch(const mpc_attn_args* args, void* stream);

/* ---- mpc_commonality --------------------------------------------------------
 * Commonality of the selected clusters across adjacent layers (Sec. 2,
 * Observation 3), the statistic that motivates cross-layer index sharing: for
 * the first k entries S_l of the selection lists of n_layers consecutive
 * layers (each its own leader), per (sequence b, kv head h)
 *   out_total[b][h] = sum over l < n_layers - m of |S_l n ... n S_{l+m}|
 *   out_score[b][h] = out_total[b][h] / (k (n_layers - m))
 * 1 means the layers selected the same clusters.  sel entries are cluster ids
 * < n_clusters or -1 (padding, ignored); an id >= n_clusters sets status bit 4.
 *
 * Token positions (kept != NULL).  Layers that lead their own groups also ran
 * their own static eviction, so one cluster id names different tokens in
 * different layers.  With kept set, every selected cluster c stands for the
 * positions of its cluster_size cache rows r = c s .. c s + s - 1: kept[r]
 * for a kept prompt row (r < n_keep[b]), prompt_len[b] + r - n_keep[b] for a
 * row appended while decoding; the sets S_l are then these k s positions, the
 * score divides by k s (n_layers - m), and n_clusters bounds the positions
 * instead (every position < n_clusters; a larger one, or a kept row r >=
 * kept_cap, sets status bit 4 and is skipped).
 * Read-only on its inputs; asynchronous on stream. */
typedef struct {
  uint32_t struct_size;        /* sizeof(mpc_commonality_args) */
  int32_t n_layers;            /* >= 2 */
  int32_t batch, n_kv_heads;
  const int32_t* sel;          /* device [n_layers][batch][n_kv_heads][sel_cap] */
  int64_t sel_layer_stride;    /* elements between layers */
  int32_t sel_cap;
  int32_t n_clusters;          /* every id < n_clusters (bitmap size) */
  int32_t k;                   /* entries compared per list, 1 .. sel_cap */
  int32_t m;                   /* windows of m + 1 layers, 1 .. n_layers - 1 */
  int32_t* out_total;          /* device [batch][n_kv_heads] */
  float* out_score;            /* device [batch][n_kv_heads] */
  /* optional: compare token positions instead of cluster ids */
  const int32_t* kept;         /* NULL, or device [n_layers][batch][n_kv_heads][kept_cap]: each layer's kept positions */
  int64_t kept_layer_stride;   /* elements between layers of kept */
  int32_t kept_cap;
  int32_t cluster_size;        /* s (>= 1 when kept is set) */
  const int32_t* n_keep;       /* device [batch], kept prompt rows (required with kept) */
  const int32_t* prompt_len;   /* device [batch], prompt lengths (required with kept) */
} mpc_commonality_args;

MPC_API int mpc_commonality(const mpc_commonality_args* args, void* stream);

/* ---- mpc_layer_refs ---------------------------------------------------------
 * Cross-layer index sharing (Sec. 3.4): the refs of a call over layers
 * 0 .. n_layers - 1.  The first two layers are left unshared (each leads
 * itself); from layer 2 on, consecutive groups of share_every layers reuse
 * the indices of the group's first layer, so layer l's leader is
 * 2 + share_every * floor((l - 2) / share_every).  share_every = 1: every
 * layer leads.  out_refs[l] = {layer l, the group of its leader (groups
 * numbered in layer order from 0), 1 if l leads its group}.
 * Host only: writes n_layers entries of out_refs (host memory) and returns
 * the number of groups, or MPC_ERR_INVALID_ARG (out_refs NULL, n_layers not
 * in 1 .. MPC_MAX_REFS, share_every < 1). */
MPC_API int mpc_layer_refs(int32_t n_layers, int32_t share_every, mpc_layer_ref* out_refs);

/* ---- mpc_choose_share_every --------------------------------------------------
 * The adaptive sharing-group size (Sec. 2, Observation 3; Sec. 3.4): score[m - 1]
 * is the commonality score of windows of m + 1 adjacent layers
 * (mpc_commonality's out_score for that m, e.g. averaged over sequences and
 * kv heads), for m = 1 .. n.  Returns the largest m + 1 whose score reaches
 * `threshold` (groups of that many layers selected nearly the same clusters,
 * so one leader can serve them), else 1 (no sharing).  Host only; returns
 * MPC_ERR_INVALID_ARG for score NULL, n < 1 or a threshold outside [0, 1]. */
MPC_API int mpc_choose_share_every(int32_t n, const float* score, float threshold);

/* Rows of the summary pyramid for a cache of cap_tokens rows (the sum of the
 * level capacities above), or a negative MPC_ERR_* code. */
MPC_API int64_t mpc_summary_rows(int32_t cap_tokens, int32_t cluster_size,
                                 int32_t n_levels, const int32_t* fanout);

/* Thread-local description of the last error of this thread ("" if none). */
MPC_API const char* mpc_last_error(void);

/* Device status word of the current device: flag 1 once a kernel of this
 * library gave up a bounded wait (for a bulk copy, or for a split unit's
 * pieces, that did not arrive); such a kernel skips the work that needed
 * the wait (an attention unit whose pieces did not all arrive keeps its
 * previous output, no partial o is written) and returns; the call's outputs
 * are then undefined and its workspace must be zero-filled again.  Flag 2:
 * a decode step found no cache row left (the sequence is skipped, its token
 * count kept); flag 4: an index out of range was reported and skipped.
 * Blocks on the device (cudaDeviceSynchronize), returns the flags and
 * clears them. */
MPC_API int mpc_device_status(int* flags);

/* Failure-path self-test: launches one kernel whose wait is never
 * satisfied (kind 0: an mbarrier nothing completes; kind 1: the device int
 * never_set, which the caller keeps 0, polled with acquire loads) and gives
 * up after limit_us microseconds (1 .. 1e6), setting flag 1 of the device
 * status word; the context stays usable.  Asynchronous on `stream`. */
MPC_API int mpc_selftest_wait(int32_t kind, int32_t limit_us, const int32_t* never_set, void* stream);

/* MPC_ABI_VERSION of the loaded library. */
MPC_API int mpc_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* MPCACHE_H */
