// Kernel parameter blocks and launchers of the MPCache library.
#pragma once

#include <cuda.h>

#include "common.cuh"

namespace mpc {

// RAII NVTX range: one named range over each ABI call
struct NvtxRange {
  explicit NvtxRange(const char* name);
  ~NvtxRange();
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

struct AttnParams {
  RefTable refs;
  int n_refs, B, Hq, Hkv, G;
  const void* q;
  const void* k_new;
  const void* v_new;
  int64_t q_ls, kvn_ls;
  void* kc;
  void* vc;
  int64_t cache_ls;
  int cap_tokens;
  const int* sel;
  const int* n_sel;
  int sel_cap;
  float* rmax;
  float* rmin;
  float* rep;
  float* mean;  // optional, kept current by the seal
  Pyramid pyr;
  float alpha;
  int* n_tok;
  int advance;
  float scale_log2;  // softmax scale times log2(e)
  float* out;
  int64_t out_ls;
  int n_split, tiles_per_split;  // split grid (fp32)
  int n_stages;                  // ring depth per warp (persistent bf16 kernel)
  float* part;        // fp32: [unit][split][G][D + 4]; bf16: [2 * warps][G][D + 4]
  int* unit_counter;  // [unit]
  int* grid_counter;  // [1]
};

// Fused decode step: the leaders' hierarchical selection and every ref's
// append + sparse attention in one persistent launch (decode_step.cu).
struct StepParams {
  AttnParams a;                // attention part; a.part holds two records per warp slot
  int* sel_out;                // written by the in-call selection (the same array as a.sel)
  int* n_sel_out;              // [B]
  int n_sel_units;             // leader refs x B x Hkv; 0 = attention only (selections are inputs)
  int16_t lead_ref[kMaxRefs];  // ref index of the i-th leader ref
  int16_t lead_of[kMaxRefs];   // for each ref: index among the leader refs of its group's leader
  int keep_ppm[kMaxLevels];
  int metric;                  // MPC_SIM_EQ3, _BOUND or _MEAN
  const float* src0;           // staged summary rows: rep (Eq. 3), mean, or r_max (Eq. 2)
  const float* src1;           // r_min (Eq. 2)
  int n_src;
  int max_cand;                // power of two, capacity of a team's candidate arrays
  int row_buf;                 // summary rows a team stages at once
  int spec;                    // the first round also stages the level below the coarsest
  int team_warps;              // warps per selection team (divides the CTA's warps)
  int static_ppm;              // share of the tile list cut into static warp ranges
  int slice_tiles;             // tiles per dynamic slice of the rest (0: all static)
  int rec_slots;               // range slots the partial-record arrays hold
  unsigned* sel_pub;           // [n_sel_units][1 + sel_cap]: count, then ids, each tagged with the call
  int* ctl;                    // [8]: claim counter, grid ticket, call counter, abort flag
};

struct SelectParams {
  RefTable refs;
  int n_refs, B, Hq, Hkv, G;
  const void* q;
  int64_t q_ls;
  const float* rep;
  Pyramid pyr;
  const int* n_tok;
  int keep_ppm[kMaxLevels];
  int sel_cap;
  int* out_sel;
  int* out_n_sel;
  int max_cand;  // power of two, capacity of the shared candidate arrays
  int row_buf;   // candidates whose summary rows are staged in shared memory at once
  int spec_first;  // the first round also scores the whole level below the coarsest
  int metric;      // MPC_SIM_EQ3: rep; MPC_SIM_BOUND / _FXP: r_max and r_min; MPC_SIM_MEAN: mean
  const float* rmax;
  const float* rmin;
  const float* mean;
  int frac_bits;           // MPC_SIM_FXP: fractional bits f
  long long fxp_a, fxp_b;  // MPC_SIM_FXP: enc(alpha), enc(1 - alpha)
};

struct StaticParams {
  RefTable refs;
  int n_refs, B, Hq, Hkv, G, t_max;
  const int* lens;
  const void* q_win;
  int64_t qw_ls;
  int win_rows;
  const void* k;
  int64_t k_ls;
  const int* page_table;
  int page_size, max_pages;
  int window_ppm, long_window_ppm, long_threshold, keep_ppm;
  float scale_log2;
  int keep_cap;
  float* scores;      // [group][b][Hkv][t_max]
  int* kept;          // [group][b][Hkv][keep_cap]
  int* n_keep;        // [b]
  float* stats;       // [ref][b][Hq][stats_ld]: -(m + log2 l) per window row (SIMT passes)
  int stats_ld;       // win_rows rounded up to 128
  void* aug;          // [ref][b][Hq][stats_ld][8] bf16: -(m + log2 l) / scale_log2 as the sum of
                      // three bf16 parts, then five zeros (tcgen05 passes)
  void* k_dense;      // paged bf16 keys gathered as [ref][b][Hkv][t_max][d] (tcgen05 passes)
};

// Window scoring on tcgen05 (bf16 queries and dense keys).
struct ScoreTcParams {
  CUtensorMap map_q;  // [layer][B*Hq*win_rows][d], 128 x 64 boxes, 128B swizzle
  CUtensorMap map_k;  // dense [layer or ref][B*Hkv*t_max][d] (128-row boxes)
  RefTable refs;
  int n_refs, B, Hq, Hkv, G, t_max, win_rows;
  const int* lens;
  const void* q_win;
  int64_t qw_ls;
  const void* k;
  int64_t k_ls;
  int window_ppm, long_window_ppm, long_threshold;
  float scale_log2;
  float* scores;
  float* stats;  // as StaticParams::stats
  int stats_ld;
  void* aug;     // as StaticParams::aug
  int k_by_ref;  // dense keys indexed by ref (a gathered copy) rather than by layer
  int items_per_cta;  // 1: one CTA per (unit, 128-block) item; > 1: consecutive items per CTA
};

struct KvSrc {
  const void* data;
  int64_t layer_stride;
  const int* page_table;
  int page_size, max_pages;
};

struct ClusterParams {
  RefTable refs;
  int n_refs, B, Hkv, t_max;
  KvSrc k, v;
  const int* kept;
  int keep_cap;
  const int* n_keep;
  void* kc;
  void* vc;
  int64_t cache_ls;
  int cap_tokens;
  float* rmax;
  float* rmin;
  float* rep;
  float* mean;  // optional mean member key per cluster
  Pyramid pyr;
  float alpha;
  int* out_n_tok;
};

// Summary rows staged per candidate by the select kernel: r_max and r_min for
// the metrics that read both, else one (rep or mean).
__host__ __device__ inline int select_n_src(int metric) {
  return metric == MPC_SIM_BOUND || metric == MPC_SIM_FXP ? 2 : 1;
}

// Sparse decode attention: bf16 caches on the persistent kernel (one CTA
// per SM, owner merges), fp32 caches on the split grid (last-CTA merge).
cudaError_t launch_attn(const AttnParams& p, int dtype, int D, int n_units, cudaStream_t st);
int attn_smem_bytes(int dtype, int D, int G, int B);
int attn_persist_ctas_max();
int attn_persist_batch_max();
cudaError_t launch_step(const StepParams& p, int D, cudaStream_t st);
int step_smem_bytes(int D, int G, int B);
// CTA shape of the fused step kernel: warps per CTA and ring stages per warp
void step_shape(int D, int G, int B, int* wpc, int* nst);
// Summary rows a selection team of team_warps warps stages at once (0 if
// its scratch cannot hold the candidate arrays).
int step_row_buf(int D, int G, int B, int team_warps, int max_cand, int n_src);
constexpr int kStepSelIds = 256;  // selected ids a warp of the step kernel stages per chunk
constexpr int kStepCtasMax = 152;
constexpr int kStepBatchMax = 512;  // sequences per call (the per-sequence table lives in shared memory)
int step_ctas();
int take_status_step();
cudaError_t launch_select(const SelectParams& p, int dtype, int D, int units, cudaStream_t st);
int select_smem_bytes(int D, int max_cand, int row_buf, int n_src);
int select_spec_first(int units);
int select_threads_of(int units);
cudaError_t launch_clusters(const ClusterParams& p, int dtype, int D, int n_units, int groups_x,
                            bool any_leader, bool host_src, cudaStream_t st);
cudaError_t launch_static(const StaticParams& p, int dtype, int D, int n_layer_span, cudaStream_t st);
cudaError_t launch_score_tc(ScoreTcParams& p, int D, int n_layer_span, cudaStream_t st);
// Bytes of the gathered dense copy of paged bf16 keys (0 when not needed).
size_t static_dense_bytes(const StaticParams& p, int dtype, int D);
int static_tile_smem(int D);

// The counters of mpc_sparse_decode_attn's workspace: the byte range that
// must be zero before a call.
int attn_counter_range(const mpc_attn_args* args, size_t* off, size_t* bytes);

// Records `msg` as this thread's last error (mpc_last_error) and returns code.
int set_error(int code, const char* msg);
int take_status_commonality();
int take_status_selftest();
cudaError_t launch_wait_selftest(int kind, const int* never_set, uint64_t limit_ns, cudaStream_t st);

// Device status word of each translation unit: read it and clear it.
int take_status_attn();
int take_status_select();
int take_status_clusters();
int take_status_static();
int take_status_score_tc();

}  // namespace mpc
