// Look-once static eviction (Sec. 3.2; Alg. 2 Step 1; App. E).
//
// The accumulated attention of key j is sum_i p_ij with p_ij the causal
// softmax of window row i.  Two passes over the window x prompt score
// matrix avoid storing it:
//   rowstats_kernel  per (ref, b, query head, 64-row block): m_i = max_j s_ij
//                    and l_i = sum_j 2^(s_ij - m_i) with s in log2 units
//                    (online, one key tile at a time);
//   colsum_kernel    per (ref, b, kv head, 64-key block): recomputes s_ij for
//                    every window row of every query head of the group and
//                    sums 2^(s_ij - m_i) / l_i = 2^(s_ij - (m_i + log2 l_i))
//                    per key in registers (the row statistic is stored as
//                    the single value -(m_i + log2 l_i));
//   budget_kernel    per (ref, b, kv head): exact top-n_keep of the scores by
//                    a 4-pass 8-bit radix select on orderable fp32 keys, ties
//                    to the lower position, then an order-preserving
//                    compaction that emits the kept positions ascending.
// The two score passes are register-tiled FFMA products: a 16 x 16 thread
// block computes a 64 x 64 tile, 4 x 4 outputs per thread.
#include <cstring>

#include "kernels.cuh"

namespace mpc {


__device__ __forceinline__ int window_rows(const StaticParams& p, int T) {
  return count_from_ppm(T, T > p.long_threshold ? p.long_window_ppm : p.window_ppm);
}

template <typename T, int D>
__device__ __forceinline__ const T* key_row(const StaticParams& p, int layer, int b, int h, int t) {
  const T* base = (const T*)p.k + layer * p.k_ls;
  if (p.page_table == nullptr) return base + ((int64_t)(b * p.Hkv + h) * p.t_max + t) * D;
  const int pg = p.page_table[(int64_t)b * p.max_pages + t / p.page_size];
  return base + (((int64_t)pg * p.Hkv + h) * p.page_size + (t % p.page_size)) * D;
}

constexpr int kTile = 64;
constexpr int kPad = kTile + 4;

// Loads rows [r0, r0 + 64) of a [rows][D] operand into sm[c][row] (fp32),
// rows outside [0, n) as zeros.  `row_ptr(i)` returns the row pointer.
template <typename T, int D, typename F>
__device__ __forceinline__ void load_tile_t(float* sm, int n, int r0, F row_ptr) {
  for (int i = threadIdx.x; i < kTile * D; i += blockDim.x) {
    const int r = i / D, c = i % D;
    const int gr = r0 + r;
    float v = 0.f;
    if (gr < n) v = to_float<T>(row_ptr(gr)[c]);
    sm[c * kPad + r] = v;
  }
}

template <typename T, int D>
__global__ void __launch_bounds__(256) rowstats_kernel(const __grid_constant__ StaticParams p) {
  extern __shared__ __align__(16) float sm[];
  float* Qs = sm;
  float* Ks = sm + D * kPad;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int unit = blockIdx.y;
  const int hq = unit % p.Hq, b = (unit / p.Hq) % p.B, ri = unit / (p.Hq * p.B);
  const int layer = p.refs.layer[ri];
  const int hk = hq / p.G;
  const int T_b = p.lens[b];
  if (T_b < 1 || T_b > p.t_max) {
    if (threadIdx.x == 0 && blockIdx.x == 0) atomicOr(&g_mpc_status, 4);
    return;
  }
  const int w = window_rows(p, T_b);
  const int row0 = blockIdx.x * kTile;
  if (row0 >= w || w > p.win_rows) return;
  const T* qbase = (const T*)p.q_win + layer * p.qw_ls + ((int64_t)b * p.Hq + hq) * p.win_rows * D;
  const int qoff = p.win_rows - w;  // window row i is q_win row qoff + i
  load_tile_t<T, D>(Qs, w, row0, [&](int i) { return qbase + (int64_t)(qoff + i) * D; });
  const int last_row = min(row0 + kTile, w) - 1;
  const int pos_last = T_b - w + last_row;
  float m[4], l[4];
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    m[r] = kNegInf;
    l[r] = 0.f;
  }
  for (int j0 = 0; j0 <= pos_last; j0 += kTile) {
    __syncthreads();
    load_tile_t<T, D>(Ks, T_b, j0, [&](int t) { return key_row<T, D>(p, layer, b, hk, t); });
    __syncthreads();
    float acc[4][4] = {};
#pragma unroll 8
    for (int c = 0; c < D; ++c) {
      const float4 a = *reinterpret_cast<const float4*>(Qs + c * kPad + ty * 4);
      const float4 k4 = *reinterpret_cast<const float4*>(Ks + c * kPad + tx * 4);
      const float av[4] = {a.x, a.y, a.z, a.w}, kv[4] = {k4.x, k4.y, k4.z, k4.w};
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[r][q] = fmaf(av[r], kv[q], acc[r][q]);
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int i = row0 + ty * 4 + r;
      const int pos = T_b - w + i;
      float x[4];
      float mx = kNegInf;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int j = j0 + tx * 4 + q;
        x[q] = (i < w && j <= pos) ? acc[r][q] * p.scale_log2 : kNegInf;
        mx = fmaxf(mx, x[q]);
      }
#pragma unroll
      for (int o = 1; o < 16; o <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      const float mn = fmaxf(m[r], mx);
      const bool any = mn != kNegInf;  // row sees a key so far
      const float base = any ? mn : 0.f;
      float sum = 0.f;
#pragma unroll
      for (int q = 0; q < 4; ++q) sum += fast_exp2(x[q] - base);
#pragma unroll
      for (int o = 1; o < 16; o <<= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      if (any) {
        l[r] = (m[r] == kNegInf) ? sum : l[r] * fast_exp2(m[r] - mn) + sum;
        m[r] = mn;
      }
    }
  }
  if (tx == 0) {
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int i = row0 + ty * 4 + r;
      if (i < w) p.stats[(((int64_t)ri * p.B + b) * p.Hq + hq) * p.stats_ld + i] = -(m[r] + log2f(l[r]));
    }
  }
}

template <typename T, int D>
__global__ void __launch_bounds__(256) colsum_kernel(const __grid_constant__ StaticParams p) {
  extern __shared__ __align__(16) float sm[];
  float* Ks = sm;
  float* Qs = sm + D * kPad;
  float* st = Qs + D * kPad;  // -(m + log2 l) of the tile's rows
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;  // ty: keys, tx: rows
  const int unit = blockIdx.y;
  const int hk = unit % p.Hkv, b = (unit / p.Hkv) % p.B, ri = unit / (p.Hkv * p.B);
  const int layer = p.refs.layer[ri], group = p.refs.group[ri];
  const int T_b = p.lens[b];
  if (T_b < 1 || T_b > p.t_max) return;
  const int w = window_rows(p, T_b);
  const int j0 = blockIdx.x * kTile;
  if (j0 >= T_b || w > p.win_rows) return;
  load_tile_t<T, D>(Ks, T_b, j0, [&](int t) { return key_row<T, D>(p, layer, b, hk, t); });
  const int qoff = p.win_rows - w;
  // rows whose position reaches this key block: pos_i = T_b - w + i >= j0
  const int i_first = max(0, j0 - (T_b - w));
  const int i_start = (i_first / kTile) * kTile;
  float col[4] = {0.f, 0.f, 0.f, 0.f};
  for (int g = 0; g < p.G; ++g) {
    const int hq = hk * p.G + g;
    const T* qbase = (const T*)p.q_win + layer * p.qw_ls + ((int64_t)b * p.Hq + hq) * p.win_rows * D;
    const float* stats = p.stats + (((int64_t)ri * p.B + b) * p.Hq + hq) * p.stats_ld;
    for (int i0 = i_start; i0 < w; i0 += kTile) {
      __syncthreads();
      load_tile_t<T, D>(Qs, w, i0, [&](int i) { return qbase + (int64_t)(qoff + i) * D; });
      for (int i = threadIdx.x; i < kTile; i += blockDim.x)
        st[i] = (i0 + i < w) ? stats[i0 + i] : kNegInf;
      __syncthreads();
      float acc[4][4] = {};
#pragma unroll 8
      for (int c = 0; c < D; ++c) {
        const float4 k4 = *reinterpret_cast<const float4*>(Ks + c * kPad + ty * 4);
        const float4 a = *reinterpret_cast<const float4*>(Qs + c * kPad + tx * 4);
        const float kv[4] = {k4.x, k4.y, k4.z, k4.w}, av[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
        for (int q = 0; q < 4; ++q)
#pragma unroll
          for (int r = 0; r < 4; ++r) acc[q][r] = fmaf(kv[q], av[r], acc[q][r]);
      }
      float tile[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int i = i0 + tx * 4 + r;
        const int pos = T_b - w + i;
        const float nml = st[tx * 4 + r];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int j = j0 + ty * 4 + q;
          if (i < w && j <= pos) tile[q] += fast_exp2(acc[q][r] * p.scale_log2 + nml);
        }
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) col[q] += tile[q];
    }
  }
#pragma unroll
  for (int q = 0; q < 4; ++q)
#pragma unroll
    for (int o = 1; o < 16; o <<= 1) col[q] += __shfl_xor_sync(0xffffffffu, col[q], o);
  if (tx == 0) {
    float* out = p.scores + ((int64_t)(group * p.B + b) * p.Hkv + hk) * p.t_max;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int j = j0 + ty * 4 + q;
      if (j < T_b) out[j] = col[q];
    }
  }
}

constexpr int kBudgetThreads = 1024;

__device__ __forceinline__ int block_scan_1024(int v, int* wt, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wt[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int t = wt[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, t, o);
      if (lane >= o) t += y;
    }
    wt[lane] = t;
    if (lane == 31) *total = t;
  }
  __syncthreads();
  const int before = (warp > 0 ? wt[warp - 1] : 0) + x - v;
  __syncthreads();
  return before;
}

__global__ void __launch_bounds__(kBudgetThreads) budget_kernel(const __grid_constant__ StaticParams p) {
  extern __shared__ __align__(16) uint32_t keys[];
  __shared__ int hist[256];
  __shared__ int wt[32];
  __shared__ int s_total, s_digit, s_above;
  const int unit = blockIdx.x;
  const int hk = unit % p.Hkv, b = (unit / p.Hkv) % p.B, ri = unit / (p.Hkv * p.B);
  const int group = p.refs.group[ri];
  const int T_b = min(max(p.lens[b], 0), p.t_max);
  const int nk = count_from_ppm(T_b, p.keep_ppm);
  const int64_t ub = (int64_t)(group * p.B + b) * p.Hkv + hk;
  const float* sc = p.scores + ub * p.t_max;
  int* out = p.kept + ub * p.keep_cap;
  for (int j = threadIdx.x; j < T_b; j += blockDim.x) keys[j] = orderable(sc[j]);
  if (threadIdx.x == 0 && ri == 0 && hk == 0) p.n_keep[b] = nk;
  uint32_t prefix = 0, mask = 0;
  int remaining = nk;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (int j = threadIdx.x; j < T_b; j += blockDim.x) {
      const uint32_t k = keys[j];
      if ((k & mask) == prefix) atomicAdd(&hist[(k >> shift) & 255u], 1);
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      // the largest digit d whose suffix count S[d] = sum_{d' >= d} hist[d']
      // reaches `remaining` (d = 0 if none above 0 does), and S[d + 1]:
      // lane l holds digits 8l .. 8l + 7, the suffix runs over the lanes
      const int lane = threadIdx.x;
      int h[8], local = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        h[i] = hist[lane * 8 + i];
        local += h[i];
      }
      int incl = local;  // sum over lanes >= lane
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_down_sync(0xffffffffu, incl, o);
        if (lane + o < 32) incl += y;
      }
      int run = incl - local, found = -1, above = 0;  // run = S[8 lane + 8]
#pragma unroll
      for (int i = 7; i >= 0; --i) {
        if (found < 0 && lane * 8 + i > 0 && run + h[i] >= remaining) {
          found = lane * 8 + i;
          above = run;
        }
        run += h[i];
      }
      const unsigned bal = __ballot_sync(0xffffffffu, found >= 0);
      if (bal != 0) {
        if (lane == 31 - __clz(bal)) {
          s_digit = found;
          s_above = above;
        }
      } else if (lane == 0) {
        s_digit = 0;
        s_above = incl - h[0];  // S[1]
      }
    }
    __syncthreads();
    remaining -= s_above;
    prefix |= (uint32_t)s_digit << shift;
    mask |= 255u << shift;
    __syncthreads();
  }
  // prefix is the n_keep-th largest key; `remaining` copies of it are kept,
  // the lowest positions first
  const int per = (T_b + kBudgetThreads - 1) / kBudgetThreads;
  const int j0 = threadIdx.x * per, j1 = min(T_b, j0 + per);
  int gt = 0, eq = 0;
  for (int j = j0; j < j1; ++j) {
    gt += keys[j] > prefix;
    eq += keys[j] == prefix;
  }
  const int eq_before = block_scan_1024(eq, wt, &s_total);
  const int take = max(0, min(eq, remaining - eq_before));
  const int off = block_scan_1024(gt + take, wt, &s_total);
  int o = off, taken = 0;
  for (int j = j0; j < j1; ++j) {
    const uint32_t k = keys[j];
    if (k > prefix || (k == prefix && taken < take)) {
      if (k == prefix) ++taken;
      out[o++] = j;
    }
  }
  for (int j = nk + threadIdx.x; j < p.keep_cap; j += blockDim.x) out[j] = -1;
}

int static_tile_smem(int D) { return (2 * D * kPad) * 4 + kTile * 8; }

template <typename K>
static cudaError_t set_smem(K kernel, int bytes) {
  return ensure_dyn_smem((const void*)kernel, bytes);
}

// Gathers the paged keys of every (ref, sequence, kv head) into a dense
// [ref][b][Hkv][t_max][d] copy (rows [0, T_b)), so that the tensor-core
// passes stream 128-key tiles with two TMA boxes rather than one per page
// and half.  Page ids outside the pool are reported and their rows skipped.
template <int D>
__global__ void __launch_bounds__(256) densify_kernel(const __grid_constant__ StaticParams p) {
  constexpr int CH = D * 2 / 16;  // 16-byte chunks per bf16 row
  const int unit = blockIdx.y;
  const int h = unit % p.Hkv, b = (unit / p.Hkv) % p.B, ri = unit / (p.Hkv * p.B);
  const int layer = p.refs.layer[ri];
  const int T_b = p.lens[b];
  const int r0 = blockIdx.x * 128;
  if (T_b < 1 || T_b > p.t_max || r0 >= T_b) return;
  const int64_t pool_pages = p.k_ls / ((int64_t)p.Hkv * p.page_size * D);
  const bf16* pool = (const bf16*)p.k + layer * p.k_ls;
  bf16* dst = (bf16*)p.k_dense + (((int64_t)ri * p.B + b) * p.Hkv + h) * p.t_max * D;
  for (int i = threadIdx.x; i < 128 * CH; i += blockDim.x) {
    const int r = r0 + i / CH, c = i % CH;
    if (r >= T_b) break;
    const int pg = p.page_table[(int64_t)b * p.max_pages + r / p.page_size];
    if (pg < 0 || pg >= pool_pages) {
      atomicOr(&g_mpc_status, 4);
      continue;
    }
    const bf16* src = pool + (((int64_t)pg * p.Hkv + h) * p.page_size + r % p.page_size) * D;
    reinterpret_cast<uint4*>(dst + (int64_t)r * D)[c] = reinterpret_cast<const uint4*>(src)[c];
  }
}

size_t static_dense_bytes(const StaticParams& p, int dtype, int D) {
  if (dtype != MPC_BF16 || p.page_table == nullptr) return 0;
  return (size_t)p.n_refs * p.B * p.Hkv * p.t_max * D * 2;
}

cudaError_t launch_static(const StaticParams& p, int dtype, int D, int n_layer_span, cudaStream_t st) {
  cudaError_t e = cudaSuccess;
  if (dtype == MPC_BF16) {
    // both score passes on the tensor cores; paged keys are first gathered
    // into the dense copy in the workspace
    const bool paged = p.page_table != nullptr;
    if (paged) {
      const dim3 gd((p.t_max + 127) / 128, p.n_refs * p.B * p.Hkv);
      if (D == 64) densify_kernel<64><<<gd, 256, 0, st>>>(p);
      else densify_kernel<128><<<gd, 256, 0, st>>>(p);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    ScoreTcParams t;
    memset(&t, 0, sizeof(t));
    t.refs = p.refs;
    t.n_refs = p.n_refs;
    t.B = p.B;
    t.Hq = p.Hq;
    t.Hkv = p.Hkv;
    t.G = p.G;
    t.t_max = p.t_max;
    t.win_rows = p.win_rows;
    t.lens = p.lens;
    t.q_win = p.q_win;
    t.qw_ls = p.qw_ls;
    t.k = paged ? p.k_dense : p.k;
    t.k_ls = paged ? (int64_t)p.B * p.Hkv * p.t_max * D : p.k_ls;
    t.k_by_ref = paged ? 1 : 0;
    t.window_ppm = p.window_ppm;
    t.long_window_ppm = p.long_window_ppm;
    t.long_threshold = p.long_threshold;
    t.scale_log2 = p.scale_log2;
    t.scores = p.scores;
    t.stats = p.stats;
    t.stats_ld = p.stats_ld;
    t.aug = p.aug;
    if ((e = launch_score_tc(t, D, n_layer_span, st)) != cudaSuccess) return e;
  } else {
    const int smem = static_tile_smem(D);
    const dim3 g1((p.win_rows + kTile - 1) / kTile, p.n_refs * p.B * p.Hq);
    const dim3 g2((p.t_max + kTile - 1) / kTile, p.n_refs * p.B * p.Hkv);
#define MPC_STATIC_CASE(TT, DD)                                                        \
  if ((e = set_smem(rowstats_kernel<TT, DD>, smem)) != cudaSuccess) return e;          \
  if ((e = set_smem(colsum_kernel<TT, DD>, smem)) != cudaSuccess) return e;            \
  rowstats_kernel<TT, DD><<<g1, 256, smem, st>>>(p);                                   \
  if ((e = cudaGetLastError()) != cudaSuccess) return e;                               \
  colsum_kernel<TT, DD><<<g2, 256, smem, st>>>(p);                                     \
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (dtype == MPC_BF16 && D == 64) { MPC_STATIC_CASE(bf16, 64) }
    else if (dtype == MPC_BF16) { MPC_STATIC_CASE(bf16, 128) }
    else if (D == 64) { MPC_STATIC_CASE(float, 64) }
    else { MPC_STATIC_CASE(float, 128) }
#undef MPC_STATIC_CASE
  }
  const int bsmem = p.t_max * 4;
  if ((e = set_smem(budget_kernel, bsmem)) != cudaSuccess) return e;
  budget_kernel<<<p.n_refs * p.B * p.Hkv, kBudgetThreads, bsmem, st>>>(p);
  return cudaGetLastError();
}

int take_status_static() { return take_status(); }

}  // namespace mpc
