// C ABI of the MPCache library: argument validation (host only, before any
// CUDA call), workspace sizing, launch planning and kernel launches.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>

#include <nvtx3/nvToolsExt.h>

#include "kernels.cuh"

namespace mpc {

// NVTX range over one ABI call (a host-side marker for profilers and
// tracers; without an attached tool the push and pop return at once)
NvtxRange::NvtxRange(const char* name) { nvtxRangePushA(name); }
NvtxRange::~NvtxRange() { nvtxRangePop(); }

namespace {

thread_local std::string g_err;

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_err = buf;
  return code;
}

int ok() {
  g_err.clear();
  return MPC_OK;
}

#define MPC_TRY(expr)         \
  do {                        \
    const int _rc = (expr);   \
    if (_rc != MPC_OK) return _rc; \
  } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int esize(int dtype) { return dtype == MPC_BF16 ? 2 : 4; }

int check_common(int batch, int hq, int hkv, int d, int dtype) {
  if (dtype != MPC_F32 && dtype != MPC_BF16) return fail(MPC_ERR_INVALID_ARG, "dtype %d is not MPC_F32/MPC_BF16", dtype);
  if (batch < 1) return fail(MPC_ERR_BAD_SHAPE, "batch %d < 1", batch);
  if (hq < 1 || hkv < 1 || hq % hkv != 0)
    return fail(MPC_ERR_BAD_SHAPE, "n_q_heads %d must be a positive multiple of n_kv_heads %d", hq, hkv);
  if (d != 64 && d != 128) return fail(MPC_ERR_BAD_SHAPE, "head_dim %d not in {64, 128}", d);
  return MPC_OK;
}

int check_refs(int n, const mpc_layer_ref* refs, bool leaders_only, RefTable* t) {
  if (refs == nullptr) return fail(MPC_ERR_INVALID_ARG, "refs is NULL");
  if (n < 1 || n > kMaxRefs) return fail(MPC_ERR_BAD_SHAPE, "n_refs %d not in [1, %d]", n, kMaxRefs);
  for (int i = 0; i < n; ++i) {
    if (refs[i].layer < 0 || refs[i].group < 0)
      return fail(MPC_ERR_BAD_SHAPE, "refs[%d] has a negative index", i);
    if (leaders_only && !refs[i].leader) return fail(MPC_ERR_INVALID_ARG, "refs[%d] is not a leader", i);
    if (t) {
      t->layer[i] = refs[i].layer;
      t->group[i] = refs[i].group;
      t->leader[i] = refs[i].leader ? 1 : 0;
    }
  }
  return MPC_OK;
}

int check_ppm(int v, const char* name) {
  if (v < 1 || v > 1000000) return fail(MPC_ERR_BAD_SHAPE, "%s = %d ppm not in [1, 1e6]", name, v);
  return MPC_OK;
}

int make_pyramid(int cap_tokens, int s, int n_levels, const int32_t* fanout, int summary_rows, Pyramid* p,
                 bool need_rows) {
  if (s < 1 || s > 4096) return fail(MPC_ERR_BAD_SHAPE, "cluster_size %d not in [1, 4096]", s);
  if (n_levels < 1 || n_levels > kMaxLevels) return fail(MPC_ERR_BAD_SHAPE, "n_levels %d not in [1, %d]", n_levels, kMaxLevels);
  if (cap_tokens < 1 || cap_tokens % s != 0)
    return fail(MPC_ERR_BAD_SHAPE, "cap_tokens %d must be a positive multiple of cluster_size %d", cap_tokens, s);
  memset(p, 0, sizeof(*p));
  p->n_levels = n_levels;
  p->s = s;
  int rows = 0;
  int cap = cap_tokens / s;
  for (int l = 0; l < n_levels; ++l) {
    if (l > 0) {
      const int f = fanout[l - 1];
      if (f < 2 || f > 4096) return fail(MPC_ERR_BAD_SHAPE, "fanout[%d] = %d not in [2, 4096]", l - 1, f);
      p->fanout[l - 1] = f;
      cap = (cap + f - 1) / f;
    }
    p->cap[l] = cap;
    p->off[l] = rows;
    rows += cap;
  }
  p->rows = rows;
  if (need_rows && summary_rows < rows)
    return fail(MPC_ERR_BAD_SHAPE, "summary_rows %d < %d rows the pyramid needs", summary_rows, rows);
  if (need_rows) p->rows = summary_rows;
  return MPC_OK;
}

int window_bound(int t_max, int wppm, int lppm, int thr) {
  const int a = count_from_ppm(t_max < thr ? t_max : thr, wppm);
  const int b = t_max > thr ? count_from_ppm(t_max, lppm) : 0;
  return a > b ? a : b;
}

// The split of the attention tile list (static warp ranges, then dynamic
// slices) and the range slots the partial-record arrays need, for a call of
// `units` units of at most ntm tiles each.
void step_balance(int units, long long ntm, int wpc, int static_ppm, int slice_tiles, StepParams* sp) {
  // measured: slices of 2-8 tiles after a 30-80% static share were 12-50%
  // slower than all-static ranges on the 2k, 8k and 32k workloads (each slice
  // drains and refills its warp's ring and merges through a fenced ticket)
  sp->static_ppm = static_ppm > 0 ? static_ppm : 1000000;
  sp->slice_tiles = slice_tiles > 0 ? slice_tiles : 4;
  if (sp->static_ppm >= 1000000) sp->slice_tiles = 0;  // all static
  const long long tiles = (long long)units * ntm;
  const long long nb = sp->slice_tiles > 0 ? (tiles + sp->slice_tiles - 1) / sp->slice_tiles + 1 : 0;
  sp->rec_slots = (int)((long long)kStepCtasMax * wpc + nb);
}

// -------------------------------------------------------------- static ----
int validate_static(const mpc_static_args* a, StaticParams* p) {
  if (a == nullptr) return fail(MPC_ERR_INVALID_ARG, "args is NULL");
  if (a->struct_size != sizeof(mpc_static_args))
    return fail(MPC_ERR_INVALID_ARG, "struct_size %u != %zu", a->struct_size, sizeof(mpc_static_args));
  MPC_TRY(check_common(a->batch, a->n_q_heads, a->n_kv_heads, a->head_dim, a->dtype));
  memset(p, 0, sizeof(*p));
  MPC_TRY(check_refs(a->n_refs, a->refs, true, &p->refs));
  MPC_TRY(check_ppm(a->window_ppm, "window_ppm"));
  MPC_TRY(check_ppm(a->long_window_ppm, "long_window_ppm"));
  MPC_TRY(check_ppm(a->keep_ppm, "keep_ppm"));
  if (a->t_max < 1 || a->t_max > 49152) return fail(MPC_ERR_BAD_SHAPE, "t_max %d not in [1, 49152]", a->t_max);
  if (a->long_prompt_threshold < 1) return fail(MPC_ERR_BAD_SHAPE, "long_prompt_threshold < 1");
  const int wb = window_bound(a->t_max, a->window_ppm, a->long_window_ppm, a->long_prompt_threshold);
  if (a->win_rows < wb) return fail(MPC_ERR_BAD_SHAPE, "win_rows %d < longest window %d", a->win_rows, wb);
  const int kb = count_from_ppm(a->t_max, a->keep_ppm);
  if (a->keep_cap < kb) return fail(MPC_ERR_BAD_SHAPE, "keep_cap %d < %d kept tokens at t_max", a->keep_cap, kb);
  if (a->scale < 0.f || !std::isfinite(a->scale)) return fail(MPC_ERR_BAD_SHAPE, "scale must be finite and >= 0");
  const mpc_kv_tensor& k = a->k;
  if (a->dtype == MPC_BF16 &&
      (!aligned16(a->q_win) || !aligned16(k.data) || (a->q_win_layer_stride * 2) % 16 || (k.layer_stride * 2) % 16))
    return fail(MPC_ERR_INVALID_ARG, "bf16 q_win / k and their layer strides must be 16-byte aligned");
  if (k.page_table != nullptr && (k.page_size < 1 || k.max_pages < 1 ||
                                  (int64_t)k.page_size * k.max_pages < a->t_max))
    return fail(MPC_ERR_BAD_SHAPE, "paged keys: page_size * max_pages must cover t_max");
  if (a->n_kv_heads * a->batch * a->n_refs > 65535 || a->n_q_heads * a->batch * a->n_refs > 65535)
    return fail(MPC_ERR_BAD_SHAPE, "too many (ref, sequence, head) units for one call");
  p->n_refs = a->n_refs;
  p->B = a->batch;
  p->Hq = a->n_q_heads;
  p->Hkv = a->n_kv_heads;
  p->G = a->n_q_heads / a->n_kv_heads;
  p->t_max = a->t_max;
  p->lens = a->prompt_lens;
  p->q_win = a->q_win;
  p->qw_ls = a->q_win_layer_stride;
  p->win_rows = a->win_rows;
  p->k = k.data;
  p->k_ls = k.layer_stride;
  p->page_table = k.page_table;
  p->page_size = k.page_size;
  p->max_pages = k.max_pages;
  p->window_ppm = a->window_ppm;
  p->long_window_ppm = a->long_window_ppm;
  p->long_threshold = a->long_prompt_threshold;
  p->keep_ppm = a->keep_ppm;
  const float scale = a->scale > 0.f ? a->scale : 1.0f / sqrtf((float)a->head_dim);
  p->scale_log2 = scale * 1.4426950408889634f;
  p->keep_cap = a->keep_cap;
  p->scores = a->out_scores;
  p->kept = a->out_kept;
  p->n_keep = a->out_n_keep;
  return MPC_OK;
}

// Row statistics (m, 1/l) of every window row.
// Row statistics of the window, per (ref, b, query head), rows padded to a
// multiple of 128 (one bulk copy per row tile): -(m + log2 l) as fp32 for
// the SIMT passes, then the same value over the log2 scale as three bf16
// parts in a 16-byte row for the tcgen05 passes.
int stats_ld_of(int win_rows) { return (win_rows + 127) / 128 * 128; }
size_t static_stats_bytes(const StaticParams& p) {
  return (size_t)p.n_refs * p.B * p.Hq * stats_ld_of(p.win_rows) * (sizeof(float) + 16);
}
// the statistics, then (paged bf16 keys) their gathered dense copy
size_t static_ws(const StaticParams& p, int dtype, int D) {
  return static_stats_bytes(p) + static_dense_bytes(p, dtype, D);
}

// ------------------------------------------------------------ clusters ----
int validate_clusters(const mpc_cluster_args* a, ClusterParams* p) {
  if (a == nullptr) return fail(MPC_ERR_INVALID_ARG, "args is NULL");
  if (a->struct_size != sizeof(mpc_cluster_args))
    return fail(MPC_ERR_INVALID_ARG, "struct_size %u != %zu", a->struct_size, sizeof(mpc_cluster_args));
  MPC_TRY(check_common(a->batch, a->n_kv_heads, a->n_kv_heads, a->head_dim, a->dtype));
  memset(p, 0, sizeof(*p));
  MPC_TRY(check_refs(a->n_refs, a->refs, false, &p->refs));
  MPC_TRY(make_pyramid(a->cap_tokens, a->cluster_size, a->n_levels, a->fanout, a->summary_rows, &p->pyr, true));
  if (a->t_max < 1) return fail(MPC_ERR_BAD_SHAPE, "t_max < 1");
  if (a->keep_cap < 1) return fail(MPC_ERR_BAD_SHAPE, "keep_cap < 1");
  if (a->alpha < 0.f || a->alpha > 1.f) return fail(MPC_ERR_BAD_SHAPE, "alpha %g not in [0, 1]", a->alpha);
  const int es = esize(a->dtype);
  if (!aligned16(a->kc) || !aligned16(a->vc) || (a->cache_layer_stride * es) % 16 != 0)
    return fail(MPC_ERR_INVALID_ARG, "kc / vc and their layer stride must be 16-byte aligned");
  if (!aligned16(a->k.data) || !aligned16(a->v.data) || (a->k.layer_stride * es) % 16 || (a->v.layer_stride * es) % 16)
    return fail(MPC_ERR_INVALID_ARG, "prompt K / V and their layer strides must be 16-byte aligned");
  if (a->n_kv_heads * a->batch * a->n_refs > 65535) return fail(MPC_ERR_BAD_SHAPE, "too many units for one call");
  bool any_leader = false;
  for (int i = 0; i < a->n_refs; ++i) any_leader |= a->refs[i].leader != 0;
  if (any_leader && a->n_levels >= 1)
    if (a->r_max == nullptr || a->r_min == nullptr || a->rep == nullptr)
      return fail(MPC_ERR_INVALID_ARG, "a leader ref needs r_max, r_min and rep");
  p->n_refs = a->n_refs;
  p->B = a->batch;
  p->Hkv = a->n_kv_heads;
  p->t_max = a->t_max;
  p->k = KvSrc{a->k.data, a->k.layer_stride, a->k.page_table, a->k.page_size, a->k.max_pages};
  p->v = KvSrc{a->v.data, a->v.layer_stride, a->v.page_table, a->v.page_size, a->v.max_pages};
  p->kept = a->kept;
  p->keep_cap = a->keep_cap;
  p->n_keep = a->n_keep;
  p->kc = a->kc;
  p->vc = a->vc;
  p->cache_ls = a->cache_layer_stride;
  p->cap_tokens = a->cap_tokens;
  p->rmax = a->r_max;
  p->rmin = a->r_min;
  p->rep = a->rep;
  p->mean = a->mean;
  p->alpha = a->alpha;
  p->out_n_tok = a->out_n_tok;
  return MPC_OK;
}

// -------------------------------------------------------------- select ----
int validate_select(const mpc_select_args* a, SelectParams* p) {
  if (a == nullptr) return fail(MPC_ERR_INVALID_ARG, "args is NULL");
  if (a->struct_size != sizeof(mpc_select_args))
    return fail(MPC_ERR_INVALID_ARG, "struct_size %u != %zu", a->struct_size, sizeof(mpc_select_args));
  MPC_TRY(check_common(a->batch, a->n_q_heads, a->n_kv_heads, a->head_dim, a->dtype));
  memset(p, 0, sizeof(*p));
  MPC_TRY(check_refs(a->n_refs, a->refs, true, &p->refs));
  MPC_TRY(make_pyramid(a->cap_tokens, a->cluster_size, a->n_levels, a->fanout, a->summary_rows, &p->pyr, true));
  for (int l = 0; l < a->n_levels; ++l) MPC_TRY(check_ppm(a->level_keep_ppm[l], "level_keep_ppm"));
  if (!aligned16(a->rep)) return fail(MPC_ERR_INVALID_ARG, "rep must be 16-byte aligned");
  if (a->metric != MPC_SIM_EQ3 && a->metric != MPC_SIM_BOUND && a->metric != MPC_SIM_MEAN &&
      a->metric != MPC_SIM_FXP)
    return fail(MPC_ERR_INVALID_ARG, "metric %d is not MPC_SIM_EQ3, _BOUND, _MEAN or _FXP", a->metric);
  if (a->metric == MPC_SIM_FXP) {
    if (!(a->alpha >= 0.f && a->alpha <= 1.f)) return fail(MPC_ERR_BAD_SHAPE, "alpha %g not in [0, 1]", a->alpha);
    if (a->frac_bits < 1 || a->frac_bits > 24)
      return fail(MPC_ERR_BAD_SHAPE, "frac_bits %d not in [1, 24]", a->frac_bits);
  }
  if (select_n_src(a->metric) == 2 && (!aligned16(a->r_max) || !aligned16(a->r_min)))
    return fail(MPC_ERR_INVALID_ARG, "r_max / r_min must be 16-byte aligned");
  if (a->metric == MPC_SIM_MEAN && !aligned16(a->mean)) return fail(MPC_ERR_INVALID_ARG, "mean must be 16-byte aligned");
  // bound on the candidates of any level
  int kmax[kMaxLevels] = {0};
  long long mc = 0;
  for (int l = a->n_levels - 1; l >= 0; --l) {
    long long cand = p->pyr.cap[l];
    if (l < a->n_levels - 1) {
      const long long ch = (long long)p->pyr.fanout[l] * kmax[l + 1];
      if (ch < cand) cand = ch;
    }
    kmax[l] = count_from_ppm(p->pyr.cap[l], a->level_keep_ppm[l]);
    if (cand > mc) mc = cand;
  }
  if (mc > 8192) return fail(MPC_ERR_BAD_SHAPE, "up to %lld candidates at one level exceed 8192", mc);
  int P = 1;
  while (P < mc) P <<= 1;
  if (a->sel_cap < kmax[0]) return fail(MPC_ERR_BAD_SHAPE, "sel_cap %d < %d selected clusters", a->sel_cap, kmax[0]);
  if (a->n_kv_heads * a->batch * a->n_refs > 65535) return fail(MPC_ERR_BAD_SHAPE, "too many units for one call");
  p->n_refs = a->n_refs;
  p->B = a->batch;
  p->Hq = a->n_q_heads;
  p->Hkv = a->n_kv_heads;
  p->G = a->n_q_heads / a->n_kv_heads;
  p->q = a->q;
  p->q_ls = a->q_layer_stride;
  p->rep = a->rep;
  p->mean = a->mean;
  p->n_tok = a->n_tok;
  for (int l = 0; l < a->n_levels; ++l) p->keep_ppm[l] = a->level_keep_ppm[l];
  p->sel_cap = a->sel_cap;
  p->out_sel = a->out_sel;
  p->out_n_sel = a->out_n_sel;
  p->max_cand = P;
  // rows staged in shared memory at once: the first round (the coarsest
  // level, plus the level below it when the units are few) and each later
  // round (the children of a level's kept clusters), capped by what shared
  // memory holds
  const int top = a->n_levels - 1;
  p->spec_first = select_spec_first(a->n_refs * a->batch * a->n_kv_heads);
  const bool spec = p->spec_first && top > 0;
  long long need = (long long)p->pyr.cap[top] + (spec ? p->pyr.cap[top - 1] : 0);
  for (int l = spec ? top - 2 : top - 1; l >= 0; --l) {
    long long r = (long long)p->pyr.fanout[l] * kmax[l + 1];
    if (r > p->pyr.cap[l]) r = p->pyr.cap[l];
    if (r > need) need = r;
  }
  const int n_src = select_n_src(a->metric);  // summary rows per candidate
  p->metric = a->metric;
  p->rmax = a->r_max;
  p->rmin = a->r_min;
  if (a->metric == MPC_SIM_FXP) {
    // public constants enc(alpha), enc(1 - alpha): x 2^f is exact in double,
    // nearbyint rounds ties to even
    p->frac_bits = a->frac_bits;
    p->fxp_a = (long long)std::nearbyint(std::ldexp((double)a->alpha, a->frac_bits));
    p->fxp_b = (long long)std::nearbyint(std::ldexp(1.0 - (double)a->alpha, a->frac_bits));
  }
  const long long budget = (kSmemOptin - 256 - (long long)select_smem_bytes(a->head_dim, P, 0, n_src)) /
                           ((long long)a->head_dim * 4 * n_src + 4);
  if (budget < 1) return fail(MPC_ERR_BAD_SHAPE, "%d candidates leave no shared memory to stage representatives", P);
  long long rb = need < budget ? need : budget;
  // the 4-warp form (many units) runs six CTAs per SM: their shared memory
  // (each plus the 1 KB the SM reserves per CTA) within the SM's 228 KB
  if (select_threads_of(a->n_refs * a->batch * a->n_kv_heads) == 128) {
    const long long b6 = ((233472 / 6 - 1024) - 256 - (long long)select_smem_bytes(a->head_dim, P, 0, n_src)) /
                         ((long long)a->head_dim * 4 * n_src + 4);
    if (b6 >= 16 && rb > b6) rb = b6;
  }
  p->row_buf = (int)rb;
  return MPC_OK;
}

// ---------------------------------------------------------- attention ----
struct AttnPlan {
  int units, n_split, tps;
  size_t part_off, ucnt_off, gcnt_off, bytes;
};

int validate_attn(const mpc_attn_args* a, AttnParams* p, AttnPlan* plan) {
  if (a == nullptr) return fail(MPC_ERR_INVALID_ARG, "args is NULL");
  if (a->struct_size != sizeof(mpc_attn_args))
    return fail(MPC_ERR_INVALID_ARG, "struct_size %u != %zu", a->struct_size, sizeof(mpc_attn_args));
  MPC_TRY(check_common(a->batch, a->n_q_heads, a->n_kv_heads, a->head_dim, a->dtype));
  memset(p, 0, sizeof(*p));
  MPC_TRY(check_refs(a->n_refs, a->refs, false, &p->refs));
  MPC_TRY(make_pyramid(a->cap_tokens, a->cluster_size, a->n_levels, a->fanout, a->summary_rows, &p->pyr, false));
  const int G = a->n_q_heads / a->n_kv_heads;
  if (G > (a->dtype == MPC_BF16 ? 16 : 8))
    return fail(MPC_ERR_BAD_SHAPE, "%d query heads per kv head exceed %d", G, a->dtype == MPC_BF16 ? 16 : 8);
  if (a->sel_cap < 0) return fail(MPC_ERR_BAD_SHAPE, "sel_cap < 0");
  if (a->alpha < 0.f || a->alpha > 1.f) return fail(MPC_ERR_BAD_SHAPE, "alpha %g not in [0, 1]", a->alpha);
  if (a->scale < 0.f || !std::isfinite(a->scale)) return fail(MPC_ERR_BAD_SHAPE, "scale must be finite and >= 0");
  const int es = esize(a->dtype);
  if (!aligned16(a->kc) || !aligned16(a->vc) || (a->cache_layer_stride * es) % 16 != 0)
    return fail(MPC_ERR_INVALID_ARG, "kc / vc and their layer stride must be 16-byte aligned");
  if (!aligned16(a->q) || !aligned16(a->k_new) || !aligned16(a->v_new) || (a->q_layer_stride * es) % 16 ||
      (a->kv_new_layer_stride * es) % 16)
    return fail(MPC_ERR_INVALID_ARG, "q / k_new / v_new and their layer strides must be 16-byte aligned");
  bool any_leader = false;
  for (int i = 0; i < a->n_refs; ++i) any_leader |= a->refs[i].leader != 0;
  if (any_leader && a->r_max != nullptr) {
    if (a->r_min == nullptr || a->rep == nullptr) return fail(MPC_ERR_INVALID_ARG, "r_max given without r_min / rep");
    if (a->summary_rows < p->pyr.rows)
      return fail(MPC_ERR_BAD_SHAPE, "summary_rows %d < %d rows the pyramid needs", a->summary_rows, p->pyr.rows);
  }
  p->pyr.rows = a->summary_rows > p->pyr.rows ? a->summary_rows : p->pyr.rows;

  const int units = a->n_refs * a->batch * a->n_kv_heads;
  if (units > 65535) return fail(MPC_ERR_BAD_SHAPE, "too many (ref, sequence, kv head) units for one call");
  // tiles of the longest list: sel_cap clusters plus a tail of at most s rows
  const long long rows_max = (long long)a->sel_cap * a->cluster_size + a->cluster_size;
  const int tiles_max = (int)((rows_max + 15) / 16);
  int n_split = (1024 + units - 1) / units;
  if (n_split > 64) n_split = 64;
  if (n_split > tiles_max) n_split = tiles_max;
  if (n_split < 1) n_split = 1;
  int tps = (tiles_max + n_split - 1) / n_split;
  n_split = (tiles_max + tps - 1) / tps;
  plan->units = units;
  plan->n_split = n_split;
  plan->tps = tps;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += (bytes + 255) & ~size_t(255);
    return o;
  };
  if (a->dtype == MPC_BF16) {
    // persistent kernel: two partial records per warp of the grid
    // persistent kernel: one partial record per warp slot (at most eight
    // warps per CTA, so 2 x 4 x G records cover a CTA's slots)
    if (a->batch > attn_persist_batch_max())
      return fail(MPC_ERR_BAD_SHAPE, "batch %d > %d sequences per call", a->batch, attn_persist_batch_max());
    plan->part_off = take((size_t)2 * attn_persist_ctas_max() * 4 * G * (a->head_dim + 4) * sizeof(float));
  } else {
    plan->part_off = take(n_split > 1 ? (size_t)units * n_split * G * (a->head_dim + 4) * sizeof(float) : 0);
  }
  plan->ucnt_off = take((size_t)units * sizeof(int));
  plan->gcnt_off = take(sizeof(int));
  plan->bytes = off;

  p->n_refs = a->n_refs;
  p->B = a->batch;
  p->Hq = a->n_q_heads;
  p->Hkv = a->n_kv_heads;
  p->G = G;
  p->q = a->q;
  p->k_new = a->k_new;
  p->v_new = a->v_new;
  p->q_ls = a->q_layer_stride;
  p->kvn_ls = a->kv_new_layer_stride;
  p->kc = a->kc;
  p->vc = a->vc;
  p->cache_ls = a->cache_layer_stride;
  p->cap_tokens = a->cap_tokens;
  p->sel = a->sel;
  p->n_sel = a->n_sel;
  p->sel_cap = a->sel_cap;
  if (any_leader && a->r_max != nullptr) {
    p->rmax = a->r_max;
    p->rmin = a->r_min;
    p->rep = a->rep;
    p->mean = a->mean;
  }
  p->alpha = a->alpha;
  p->n_tok = a->n_tok;
  p->advance = a->advance != 0;
  const float scale = a->scale > 0.f ? a->scale : 1.0f / sqrtf((float)a->head_dim);
  p->scale_log2 = scale * 1.4426950408889634f;
  p->out = a->out;
  p->out_ls = a->out_layer_stride;
  p->n_split = n_split;
  p->tiles_per_split = tps;
  return MPC_OK;
}

// --------------------------------------------------------- decode step ----
struct StepPlan {
  AttnPlan attn;   // the two-launch path (mpc_select's and mpc_sparse_decode_attn's kernels)
  bool fused;      // one decode_step_kernel launch
  int sel_units;
  size_t part_off, ucnt_off, pub_off, ctl_off, bytes;
};

int validate_step(const mpc_decode_args* a, StepParams* sp, SelectParams* sel, StepPlan* plan) {
  if (a == nullptr) return fail(MPC_ERR_INVALID_ARG, "args is NULL");
  if (a->struct_size != sizeof(mpc_decode_args))
    return fail(MPC_ERR_INVALID_ARG, "struct_size %u != %zu", a->struct_size, sizeof(mpc_decode_args));
  memset(sp, 0, sizeof(*sp));
  memset(plan, 0, sizeof(*plan));
  const mpc_attn_args& t = a->attn;
  MPC_TRY(validate_attn(&t, &sp->a, &plan->attn));
  // one leader per group, and every ref's group led in this call
  mpc_layer_ref lead[kMaxRefs];
  int nl = 0;
  for (int i = 0; i < t.n_refs; ++i) {
    if (!t.refs[i].leader) continue;
    for (int k = 0; k < nl; ++k)
      if (lead[k].group == t.refs[i].group)
        return fail(MPC_ERR_INVALID_ARG, "refs[%d] is a second leader of group %d", i, t.refs[i].group);
    sp->lead_ref[nl] = (int16_t)i;
    lead[nl++] = t.refs[i];
  }
  for (int i = 0; i < t.n_refs; ++i) {
    int k = 0;
    while (k < nl && lead[k].group != t.refs[i].group) ++k;
    if (k == nl)
      return fail(MPC_ERR_INVALID_ARG,
                  "the leader of refs[%d]'s group %d is not among the refs (use mpc_sparse_decode_attn)", i,
                  t.refs[i].group);
    sp->lead_of[i] = (int16_t)k;
  }
  mpc_select_args sa;
  memset(&sa, 0, sizeof(sa));
  sa.struct_size = sizeof(sa);
  sa.n_refs = nl;
  sa.refs = lead;
  sa.batch = t.batch;
  sa.n_q_heads = t.n_q_heads;
  sa.n_kv_heads = t.n_kv_heads;
  sa.head_dim = t.head_dim;
  sa.dtype = t.dtype;
  sa.q = t.q;
  sa.q_layer_stride = t.q_layer_stride;
  sa.rep = t.rep;
  sa.summary_rows = t.summary_rows;
  sa.cap_tokens = t.cap_tokens;
  sa.n_tok = t.n_tok;
  sa.cluster_size = t.cluster_size;
  sa.n_levels = t.n_levels;
  for (int l = 0; l < kMaxLevels; ++l) {
    sa.fanout[l] = t.fanout[l];
    sa.level_keep_ppm[l] = a->level_keep_ppm[l];
  }
  sa.sel_cap = t.sel_cap;
  sa.out_sel = const_cast<int32_t*>(t.sel);
  sa.out_n_sel = const_cast<int32_t*>(t.n_sel);
  sa.metric = a->metric;
  sa.r_max = t.r_max;
  sa.r_min = t.r_min;
  sa.mean = t.mean;
  sa.alpha = t.alpha;
  sa.frac_bits = a->frac_bits;
  MPC_TRY(validate_select(&sa, sel));
  if (a->speculate < -1 || a->speculate > 1) return fail(MPC_ERR_BAD_SHAPE, "speculate %d not in {-1, 0, 1}", a->speculate);
  if (a->fuse < -1 || a->fuse > 1) return fail(MPC_ERR_BAD_SHAPE, "fuse %d not in {-1, 0, 1}", a->fuse);
  // an explicit speculate applies to the selection kernel of the two-launch
  // path too (its first round then stages the level below only if it fits
  // the row buffer sized above)
  if (a->speculate >= 0) sel->spec_first = a->speculate;

  const int D = t.head_dim, G = sp->a.G, B = t.batch, s = t.cluster_size;
  const int units = plan->attn.units;
  plan->sel_units = nl * B * t.n_kv_heads;
  const int n_src = select_n_src(a->metric);
  int wpc = 0, nst = 0;
  step_shape(D, G, B, &wpc, &nst);
  // published ids and counts are 16-bit values.  Automatic: the fused kernel
  // for 305-1216 selection units (2-8 per SM, where the standalone
  // selection runs its 4-warp form and its latency shows: measured faster on
  // the 2k MHA and batch-1 paged workloads), two launches otherwise
  // (measured faster on the 8k and 32k GQA workloads and at batch 4-32)
  const bool want = a->fuse == 1 || (a->fuse == -1 && plan->sel_units > 2 * kStepCtasMax &&
                                     plan->sel_units <= 8 * kStepCtasMax);
  plan->fused = want && t.dtype == MPC_BF16 && a->metric != MPC_SIM_FXP && sel->max_cand <= 1024 &&
                step_smem_bytes(D, G, B) <= kSmemOptin && t.cap_tokens / s < 65535 && t.sel_cap < 65535;
  int tw = 1, rb = 0;
  if (plan->fused) {
    // the largest team (divisor of the CTA's warps) that still gives every
    // selection unit its own team, grown while its scratch stages few rows
    const int ctas = kStepCtasMax;
    for (int d = 1; d <= wpc; ++d)
      if (wpc % d == 0 && (long long)ctas * (wpc / d) >= plan->sel_units) tw = d;
    rb = step_row_buf(D, G, B, tw, sel->max_cand, n_src);
    for (int d = tw + 1; d <= wpc && rb < 32; ++d)
      if (wpc % d == 0) {
        tw = d;
        rb = step_row_buf(D, G, B, tw, sel->max_cand, n_src);
      }
    if (rb < 8) plan->fused = false;
  }
  if (!plan->fused) {
    plan->bytes = plan->attn.bytes;
    return MPC_OK;
  }
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += (bytes + 255) & ~size_t(255);
    return o;
  };
  // two partial records per range slot (a later piece's, an owner's)
  if (a->static_ppm < 0 || a->static_ppm > 1000000 || a->slice_tiles < 0 || a->slice_tiles > 64)
    return fail(MPC_ERR_BAD_SHAPE, "static_ppm %d / slice_tiles %d out of range", a->static_ppm, a->slice_tiles);
  const long long ntm = (s + 15) / 16 + ((long long)t.sel_cap * s + 15) / 16;
  step_balance(units, ntm, wpc, a->static_ppm, a->slice_tiles, sp);
  plan->part_off = take((size_t)2 * sp->rec_slots * G * (D + 4) * sizeof(float));
  plan->ucnt_off = take((size_t)units * sizeof(int));
  plan->pub_off = take((size_t)plan->sel_units * (1 + t.sel_cap) * sizeof(unsigned));
  plan->ctl_off = take(8 * sizeof(int));
  plan->bytes = off;

  sp->sel_out = const_cast<int*>(t.sel);
  sp->n_sel_out = const_cast<int*>(t.n_sel);
  sp->n_sel_units = plan->sel_units;
  for (int l = 0; l < kMaxLevels; ++l) sp->keep_ppm[l] = sel->keep_ppm[l];
  sp->metric = a->metric;
  sp->src0 = a->metric == MPC_SIM_MEAN ? t.mean : (n_src == 2 ? t.r_max : t.rep);
  sp->src1 = t.r_min;
  sp->n_src = n_src;
  sp->max_cand = sel->max_cand;
  sp->row_buf = rb;
  sp->spec = a->speculate < 0 ? select_spec_first(plan->sel_units) : a->speculate;
  sp->team_warps = tw;
  return MPC_OK;
}

int cuda_fail(cudaError_t e, const char* what) {
  return fail(MPC_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

}  // namespace

int set_error(int code, const char* msg) { return fail(code, "%s", msg); }

// Byte range [off, off + bytes) of the workspace of mpc_sparse_decode_attn
// that must be zero before a call (its counters); the rest is written before
// it is read.
int attn_counter_range(const mpc_attn_args* args, size_t* off, size_t* bytes) {
  AttnParams p;
  AttnPlan plan;
  MPC_TRY(validate_attn(args, &p, &plan));
  *off = plan.ucnt_off;
  *bytes = plan.bytes - plan.ucnt_off;
  return MPC_OK;
}


}  // namespace mpc

using namespace mpc;

extern "C" {

MPC_API int mpc_abi_version(void) { return MPC_ABI_VERSION; }

MPC_API const char* mpc_last_error(void) { return g_err.c_str(); }

MPC_API int mpc_layer_refs(int32_t n_layers, int32_t share_every, mpc_layer_ref* out_refs) {
  if (out_refs == nullptr) return fail(MPC_ERR_INVALID_ARG, "out_refs is NULL");
  if (n_layers < 1 || n_layers > kMaxRefs) return fail(MPC_ERR_INVALID_ARG, "n_layers %d not in [1, %d]", n_layers, kMaxRefs);
  if (share_every < 1) return fail(MPC_ERR_INVALID_ARG, "share_every %d < 1", share_every);
  int groups = 0;
  for (int l = 0; l < n_layers; ++l) {
    // the first two layers lead themselves; later layers form groups of share_every
    const int lead = (share_every == 1 || l < 2) ? l : 2 + share_every * ((l - 2) / share_every);
    if (lead == l) ++groups;
    out_refs[l].layer = l;
    out_refs[l].group = groups - 1;
    out_refs[l].leader = lead == l ? 1 : 0;
  }
  return groups;
}

MPC_API int mpc_choose_share_every(int32_t n, const float* score, float threshold) {
  if (score == nullptr) return fail(MPC_ERR_INVALID_ARG, "score is NULL");
  if (n < 1) return fail(MPC_ERR_INVALID_ARG, "n %d < 1", n);
  if (!(threshold >= 0.f && threshold <= 1.f)) return fail(MPC_ERR_INVALID_ARG, "threshold %g not in [0, 1]", threshold);
  int best = 1;
  for (int m = 1; m <= n; ++m)
    if (score[m - 1] >= threshold && m + 1 > best) best = m + 1;
  return best;
}

MPC_API int64_t mpc_summary_rows(int32_t cap_tokens, int32_t cluster_size, int32_t n_levels, const int32_t* fanout) {
  Pyramid p;
  int32_t none[kMaxLevels] = {0, 0, 0, 0};
  const int rc = make_pyramid(cap_tokens, cluster_size, n_levels, fanout ? fanout : none, 0, &p, false);
  if (rc != MPC_OK) return rc;
  return p.rows;
}

MPC_API int mpc_selftest_wait(int32_t kind, int32_t limit_us, const int32_t* never_set, void* stream) {
  if (kind != 0 && kind != 1) return fail(MPC_ERR_INVALID_ARG, "kind %d is not 0 (mbarrier) or 1 (flag)", kind);
  if (limit_us < 1 || limit_us > 1000000) return fail(MPC_ERR_BAD_SHAPE, "limit_us %d not in [1, 1e6]", limit_us);
  if (kind == 1 && never_set == nullptr) return fail(MPC_ERR_INVALID_ARG, "kind 1 needs never_set");
  const cudaError_t e = launch_wait_selftest(kind, never_set, (uint64_t)limit_us * 1000ull,
                                             static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "mpc_selftest_wait launch");
  return ok();
}

MPC_API int mpc_device_status(int* flags) {
  if (flags == nullptr) return fail(MPC_ERR_INVALID_ARG, "flags is NULL");
  const cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
  const int parts[8] = {take_status_attn(),   take_status_select(),   take_status_clusters(),
                        take_status_static(), take_status_score_tc(), take_status_commonality(),
                        take_status_selftest(), take_status_step()};
  int v = 0;
  for (int x : parts) {
    if (x < 0) return fail(MPC_ERR_CUDA, "reading the device status word failed");
    v |= x;
  }
  *flags = v;
  return ok();
}

// True for pinned host memory reached through unified addressing.
static bool is_host_memory(const void* ptr) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, ptr) != cudaSuccess) {
    (void)cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeHost;
}

MPC_API int mpc_static_evict_workspace_size(const mpc_static_args* args, size_t* bytes) {
  if (bytes == nullptr) return fail(MPC_ERR_INVALID_ARG, "bytes is NULL");
  StaticParams p;
  MPC_TRY(validate_static(args, &p));
  *bytes = static_ws(p, args->dtype, args->head_dim);
  return ok();
}

MPC_API int mpc_static_evict(const mpc_static_args* args, void* workspace, size_t workspace_bytes, void* stream) {
  NvtxRange nvtx("mpc_static_evict");
  StaticParams p;
  MPC_TRY(validate_static(args, &p));
  if (!args->q_win || !args->k.data || !args->prompt_lens || !args->out_scores || !args->out_kept || !args->out_n_keep)
    return fail(MPC_ERR_INVALID_ARG, "a required pointer is NULL");
  // the tensor-core passes read keys and window queries through TMA tensor maps
  if (is_host_memory(args->k.data) || is_host_memory(args->q_win))
    return fail(MPC_ERR_INVALID_ARG, "k and q_win must be device memory, not host memory");
  const size_t need = static_ws(p, args->dtype, args->head_dim);
  if (workspace == nullptr || workspace_bytes < need)
    return fail(MPC_ERR_WORKSPACE, "workspace of %zu bytes needed", need);
  if (!aligned16(workspace)) return fail(MPC_ERR_INVALID_ARG, "workspace must be 16-byte aligned");
  p.stats = static_cast<float*>(workspace);
  p.stats_ld = stats_ld_of(p.win_rows);
  p.aug = static_cast<uint8_t*>(workspace) + (size_t)p.n_refs * p.B * p.Hq * p.stats_ld * sizeof(float);
  p.k_dense = static_dense_bytes(p, args->dtype, args->head_dim) ? static_cast<uint8_t*>(workspace) +
                                                                       static_stats_bytes(p)
                                                                 : nullptr;
  int span = 0;
  for (int i = 0; i < args->n_refs; ++i) span = args->refs[i].layer + 1 > span ? args->refs[i].layer + 1 : span;
  const cudaError_t e = launch_static(p, args->dtype, args->head_dim, span, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "mpc_static_evict launch");
  return ok();
}

MPC_API int mpc_build_clusters_workspace_size(const mpc_cluster_args* args, size_t* bytes) {
  if (bytes == nullptr) return fail(MPC_ERR_INVALID_ARG, "bytes is NULL");
  ClusterParams p;
  MPC_TRY(validate_clusters(args, &p));
  *bytes = 0;
  return ok();
}

MPC_API int mpc_build_clusters(const mpc_cluster_args* args, void* workspace, size_t workspace_bytes, void* stream) {
  NvtxRange nvtx("mpc_build_clusters");
  (void)workspace;
  (void)workspace_bytes;
  ClusterParams p;
  MPC_TRY(validate_clusters(args, &p));
  if (!args->k.data || !args->v.data || !args->kept || !args->n_keep || !args->kc || !args->vc || !args->out_n_tok)
    return fail(MPC_ERR_INVALID_ARG, "a required pointer is NULL");
  const int units = args->n_refs * args->batch * args->n_kv_heads;
  const int clusters = (args->keep_cap + args->cluster_size - 1) / args->cluster_size;
  const int gx = (clusters + 3) / 4;
  bool any_leader = false;
  for (int i = 0; i < args->n_refs; ++i) any_leader |= args->refs[i].leader != 0;
  // sources in host memory take the grid-stride gather (few SMs, deep loads)
  const bool host_src = is_host_memory(args->k.data) || is_host_memory(args->v.data);
  const cudaError_t e = launch_clusters(p, args->dtype, args->head_dim, units, gx > 0 ? gx : 1, any_leader,
                                        host_src, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "mpc_build_clusters launch");
  return ok();
}

MPC_API int mpc_select_workspace_size(const mpc_select_args* args, size_t* bytes) {
  if (bytes == nullptr) return fail(MPC_ERR_INVALID_ARG, "bytes is NULL");
  SelectParams p;
  MPC_TRY(validate_select(args, &p));
  *bytes = 0;
  return ok();
}

MPC_API int mpc_select(const mpc_select_args* args, void* workspace, size_t workspace_bytes, void* stream) {
  NvtxRange nvtx("mpc_select");
  (void)workspace;
  (void)workspace_bytes;
  SelectParams p;
  MPC_TRY(validate_select(args, &p));
  if (!args->q || !args->rep || !args->n_tok || !args->out_sel || !args->out_n_sel)
    return fail(MPC_ERR_INVALID_ARG, "a required pointer is NULL");
  if (select_n_src(args->metric) == 2 && (!args->r_max || !args->r_min))
    return fail(MPC_ERR_INVALID_ARG, "MPC_SIM_BOUND and MPC_SIM_FXP need r_max and r_min");
  if (args->metric == MPC_SIM_MEAN && !args->mean) return fail(MPC_ERR_INVALID_ARG, "MPC_SIM_MEAN needs mean");
  const int units = args->n_refs * args->batch * args->n_kv_heads;
  const cudaError_t e = launch_select(p, args->dtype, args->head_dim, units, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "mpc_select launch");
  return ok();
}

MPC_API int mpc_sparse_decode_attn_workspace_size(const mpc_attn_args* args, size_t* bytes) {
  if (bytes == nullptr) return fail(MPC_ERR_INVALID_ARG, "bytes is NULL");
  AttnParams p;
  AttnPlan plan;
  MPC_TRY(validate_attn(args, &p, &plan));
  *bytes = plan.bytes;
  return ok();
}

MPC_API int mpc_sparse_decode_attn(const mpc_attn_args* args, void* workspace, size_t workspace_bytes, void* stream) {
  NvtxRange nvtx("mpc_sparse_decode_attn");
  AttnParams p;
  AttnPlan plan;
  MPC_TRY(validate_attn(args, &p, &plan));
  if (!args->q || !args->k_new || !args->v_new || !args->kc || !args->vc || !args->n_tok || !args->out ||
      (args->sel_cap > 0 && (!args->sel || !args->n_sel)))
    return fail(MPC_ERR_INVALID_ARG, "a required pointer is NULL");
  if (workspace == nullptr || workspace_bytes < plan.bytes)
    return fail(MPC_ERR_WORKSPACE, "workspace of %zu bytes needed", plan.bytes);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  p.part = reinterpret_cast<float*>(ws + plan.part_off);
  p.unit_counter = reinterpret_cast<int*>(ws + plan.ucnt_off);
  p.grid_counter = reinterpret_cast<int*>(ws + plan.gcnt_off);
  const cudaError_t e = launch_attn(p, args->dtype, args->head_dim, plan.units, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "mpc_sparse_decode_attn launch");
  return ok();
}

MPC_API int mpc_decode_step_workspace_size(const mpc_decode_args* args, size_t* bytes) {
  if (bytes == nullptr) return fail(MPC_ERR_INVALID_ARG, "bytes is NULL");
  StepParams sp;
  SelectParams sel;
  StepPlan plan;
  MPC_TRY(validate_step(args, &sp, &sel, &plan));
  *bytes = plan.bytes;
  return ok();
}

MPC_API int mpc_decode_step_plan(const mpc_decode_args* args, int32_t* launches) {
  if (launches == nullptr) return fail(MPC_ERR_INVALID_ARG, "launches is NULL");
  StepParams sp;
  SelectParams sel;
  StepPlan plan;
  MPC_TRY(validate_step(args, &sp, &sel, &plan));
  *launches = plan.fused ? 1 : 2;
  return ok();
}

MPC_API int mpc_decode_step(const mpc_decode_args* args, void* workspace, size_t workspace_bytes, void* stream) {
  NvtxRange nvtx("mpc_decode_step");
  StepParams sp;
  SelectParams sel;
  StepPlan plan;
  MPC_TRY(validate_step(args, &sp, &sel, &plan));
  const mpc_attn_args& t = args->attn;
  if (!t.q || !t.k_new || !t.v_new || !t.kc || !t.vc || !t.n_tok || !t.out || !t.sel || !t.n_sel)
    return fail(MPC_ERR_INVALID_ARG, "a required pointer is NULL");
  if (!t.rep || !t.r_max || !t.r_min) return fail(MPC_ERR_INVALID_ARG, "the summary pyramid (r_max, r_min, rep) is required");
  if (args->metric == MPC_SIM_MEAN && !t.mean) return fail(MPC_ERR_INVALID_ARG, "MPC_SIM_MEAN needs mean");
  if (workspace == nullptr || workspace_bytes < plan.bytes)
    return fail(MPC_ERR_WORKSPACE, "workspace of %zu bytes needed", plan.bytes);
  if (!aligned16(workspace)) return fail(MPC_ERR_INVALID_ARG, "workspace must be 16-byte aligned");
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (plan.fused) {
    sp.a.part = reinterpret_cast<float*>(ws + plan.part_off);
    sp.a.unit_counter = reinterpret_cast<int*>(ws + plan.ucnt_off);
    sp.sel_pub = reinterpret_cast<unsigned*>(ws + plan.pub_off);
    sp.ctl = reinterpret_cast<int*>(ws + plan.ctl_off);
    e = launch_step(sp, t.head_dim, st);
    if (e != cudaSuccess) return cuda_fail(e, "mpc_decode_step launch");
    return ok();
  }
  e = launch_select(sel, t.dtype, t.head_dim, plan.sel_units, st);
  if (e != cudaSuccess) return cuda_fail(e, "mpc_decode_step select launch");
  sp.a.part = reinterpret_cast<float*>(ws + plan.attn.part_off);
  sp.a.unit_counter = reinterpret_cast<int*>(ws + plan.attn.ucnt_off);
  sp.a.grid_counter = reinterpret_cast<int*>(ws + plan.attn.gcnt_off);
  e = launch_attn(sp.a, t.dtype, t.head_dim, plan.attn.units, st);
  if (e != cudaSuccess) return cuda_fail(e, "mpc_decode_step attention launch");
  return ok();
}

}  // extern "C"
