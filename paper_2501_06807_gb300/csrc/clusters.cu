// Token gathering of the kept set into the cluster-major cache and the
// summary pyramid (Alg. 2 Step 1 token_gather; Sec. 3.3: r_max, r_min, the
// Eq. 3 representative and the hierarchical levels).
//
// gather_kernel: one warp per finest cluster (s consecutive kept rows; the
// last, partial one is the tail).  Lanes own 16-byte chunks of a row, so a
// warp moves whole rows with coalesced 16-byte loads and stores, writing each
// chunk to its swizzled slot, and leaders fold the chunk into a running
// channel max / min (and sum, for the optional mean key).  coarse_kernel: one
// CTA per (ref, b, h) builds the coarser levels from the level below
// (element-wise max / min of children; means weighted by their finest
// clusters).
#include "kernels.cuh"

namespace mpc {

// CTAs of the grid-stride gather (host sources): 4 warps each, U x 2 x 512
// bytes in flight per warp (about 2.5 MB in all, ample for the host link);
// half the SMs, measured best beside a concurrent scoring kernel.
constexpr int kHostGatherCtas = 76;
// Row steps loaded at once by the one-warp-per-cluster gather (device
// sources: occupancy hides the latency).
constexpr int kDeviceGatherSteps = 1;

template <typename T, int D>
__device__ __forceinline__ const T* kv_row(const KvSrc& src, int layer, int b, int h, int t, int Hkv,
                                           int t_max) {
  const T* base = (const T*)src.data + layer * src.layer_stride;
  if (src.page_table == nullptr) return base + ((int64_t)(b * Hkv + h) * t_max + t) * D;
  const int pg = src.page_table[(int64_t)b * src.max_pages + t / src.page_size];
  return base + (((int64_t)pg * Hkv + h) * src.page_size + (t % src.page_size)) * D;
}

// Gathers finest cluster c of unit (ref, b, h) with one warp.  The rows'
// chunks are loaded U row-steps at a time before any is used, so a warp keeps
// U x 2 x 512 bytes in flight (U > 1 for sources across the host link).
template <typename T, int D, int U>
__device__ __forceinline__ void gather_cluster(const ClusterParams& p, int unit, int c, int lane) {
  constexpr int E = 16 / (int)sizeof(T);  // elements per chunk
  constexpr int CH = D / E;               // chunks per row
  constexpr int RPW = 32 / CH;            // rows per warp step
  const int h = unit % p.Hkv, b = (unit / p.Hkv) % p.B, ri = unit / (p.Hkv * p.B);
  const int layer = p.refs.layer[ri], group = p.refs.group[ri];
  const bool leader = p.refs.leader[ri];
  const int s = p.pyr.s;
  const int nk = p.n_keep[b];
  if (c == 0 && lane == 0 && ri == 0 && h == 0) p.out_n_tok[b] = nk;
  const int r0 = c * s;
  if (r0 >= nk) return;
  const int r1 = min(r0 + s, nk);
  const bool full = (r1 - r0) == s;
  if (nk > p.cap_tokens || nk > p.keep_cap) {
    if (lane == 0) atomicOr(&g_mpc_status, 2);
    return;
  }
  const int* kept = p.kept + ((int64_t)(group * p.B + b) * p.Hkv + h) * p.keep_cap;
  T* kc = (T*)p.kc + layer * p.cache_ls + (int64_t)(b * p.Hkv + h) * p.cap_tokens * D;
  T* vc = (T*)p.vc + layer * p.cache_ls + (int64_t)(b * p.Hkv + h) * p.cap_tokens * D;
  const int ch = lane % CH, ro = lane / CH;
  float mx[E], mn[E], sm[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    mx[e] = kNegInf;
    mn[e] = kPosInf;
    sm[e] = 0.f;
  }
  for (int rb = r0 + ro; rb < r1; rb += U * RPW) {
    uint4 kv[U], vv[U];
    bool ok[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int r = rb + u * RPW;
      const int t = r < r1 ? kept[r] : 0;
      ok[u] = r < r1 && t >= 0 && t < p.t_max;
      if (r < r1 && !ok[u]) atomicOr(&g_mpc_status, 4);  // corrupt kept set: report, skip the row
      if (ok[u]) {
        kv[u] = reinterpret_cast<const uint4*>(kv_row<T, D>(p.k, layer, b, h, t, p.Hkv, p.t_max))[ch];
        vv[u] = reinterpret_cast<const uint4*>(kv_row<T, D>(p.v, layer, b, h, t, p.Hkv, p.t_max))[ch];
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (!ok[u]) continue;
      const int r = rb + u * RPW;
      const int pch = ch ^ (r & 7);
      reinterpret_cast<uint4*>(kc + (int64_t)r * D)[pch] = kv[u];
      reinterpret_cast<uint4*>(vc + (int64_t)r * D)[pch] = vv[u];
      if (leader && full) {
        const T* el = reinterpret_cast<const T*>(&kv[u]);
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const float x = to_float<T>(el[e]);
          mx[e] = fmaxf(mx[e], x);
          mn[e] = fminf(mn[e], x);
          sm[e] += x;
        }
      }
    }
  }
  if (!(leader && full)) return;
#pragma unroll
  for (int o = CH; o < 32; o <<= 1)
#pragma unroll
    for (int e = 0; e < E; ++e) {
      mx[e] = fmaxf(mx[e], __shfl_xor_sync(0xffffffffu, mx[e], o));
      mn[e] = fminf(mn[e], __shfl_xor_sync(0xffffffffu, mn[e], o));
      sm[e] += __shfl_xor_sync(0xffffffffu, sm[e], o);
    }
  if (ro != 0) return;
  if (c >= p.pyr.cap[0]) {
    atomicOr(&g_mpc_status, 2);
    return;
  }
  const int64_t row = (((int64_t)(group * p.B + b) * p.Hkv + h) * p.pyr.rows + p.pyr.off[0] + c) * D;
  const float a = p.alpha, am = 1.f - p.alpha;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int cc = ch * E + e;
    p.rmax[row + cc] = mx[e];
    p.rmin[row + cc] = mn[e];
    p.rep[row + cc] = fmaf(a, mx[e], am * mn[e]);
    if (p.mean != nullptr) p.mean[row + cc] = sm[e] / (float)s;
  }
}

// One warp per finest cluster: blockIdx.y = unit, 4 clusters per CTA.
template <typename T, int D>
__global__ void __launch_bounds__(128) gather_kernel(const __grid_constant__ ClusterParams p) {
  gather_cluster<T, D, kDeviceGatherSteps>(p, blockIdx.y, blockIdx.x * 4 + (threadIdx.x >> 5), threadIdx.x & 31);
}

// Grid-stride form for sources in host memory: a few CTAs keep the host link
// busy (every warp holds U row-steps in flight) without spreading over every
// SM, so that concurrent kernels keep the rest of the GPU.
template <typename T, int D>
__global__ void __launch_bounds__(128) gather_stride_kernel(const __grid_constant__ ClusterParams p, int per_unit,
                                                            int n_items) {
  for (int w = blockIdx.x * 4 + (threadIdx.x >> 5); w < n_items; w += gridDim.x * 4) {
    __syncwarp();
    gather_cluster<T, D, 8>(p, w / per_unit, w % per_unit, threadIdx.x & 31);
  }
}

template <int D>
__global__ void __launch_bounds__(256) coarse_kernel(const __grid_constant__ ClusterParams p) {
  const int unit = blockIdx.x;
  const int h = unit % p.Hkv, b = (unit / p.Hkv) % p.B, ri = unit / (p.Hkv * p.B);
  if (!p.refs.leader[ri]) return;
  const int group = p.refs.group[ri];
  int C[kMaxLevels];
  level_counts(p.pyr, p.n_keep[b], C);
  if (C[0] > p.pyr.cap[0]) return;  // reported by gather_kernel
  const int64_t ubase = ((int64_t)(group * p.B + b) * p.Hkv + h) * p.pyr.rows;
  const float a = p.alpha, am = 1.f - p.alpha;
  int P = 1;  // finest clusters under one level l-1 cluster
  for (int l = 1; l < p.pyr.n_levels; ++l) {
    const int f = p.pyr.fanout[l - 1];
    const int nc = min(C[l], p.pyr.cap[l]);
    const float* cm = p.mean ? p.mean + (ubase + p.pyr.off[l - 1]) * D : nullptr;
    float* Rm = p.mean ? p.mean + (ubase + p.pyr.off[l]) * D : nullptr;
    const float* cx = p.rmax + (ubase + p.pyr.off[l - 1]) * D;
    const float* cn = p.rmin + (ubase + p.pyr.off[l - 1]) * D;
    float* Rx = p.rmax + (ubase + p.pyr.off[l]) * D;
    float* Rn = p.rmin + (ubase + p.pyr.off[l]) * D;
    float* Rp = p.rep + (ubase + p.pyr.off[l]) * D;
    for (int i = threadIdx.x; i < nc * D; i += blockDim.x) {
      const int node = i / D, cc = i % D;
      const int q0 = node * f, q1 = min(q0 + f, C[l - 1]);
      float x = kNegInf, n = kPosInf, wsum = 0.f;
      int cnt = 0;
      for (int q = q0; q < q1; ++q) {
        x = fmaxf(x, cx[(int64_t)q * D + cc]);
        n = fminf(n, cn[(int64_t)q * D + cc]);
        if (Rm) {  // children weighted by their finest clusters (the last may hold fewer)
          const int w = min((q + 1) * P, C[0]) - q * P;
          wsum = fmaf((float)w, cm[(int64_t)q * D + cc], wsum);
          cnt += w;
        }
      }
      Rx[i] = x;
      Rn[i] = n;
      Rp[i] = fmaf(a, x, am * n);
      if (Rm) Rm[i] = wsum / (float)cnt;
    }
    P *= f;
    __syncthreads();
  }
}

cudaError_t launch_clusters(const ClusterParams& p, int dtype, int D, int n_units, int groups_x,
                            bool any_leader, bool host_src, cudaStream_t st) {
  const dim3 grid(groups_x, n_units);
  const int per_unit = groups_x * 4;
  const long long items = (long long)per_unit * n_units;
  const int nb = (int)(items / 4 < kHostGatherCtas ? (items + 3) / 4 : kHostGatherCtas);
#define MPC_GATHER(TT, DD)                                                           \
  if (host_src) gather_stride_kernel<TT, DD><<<nb, 128, 0, st>>>(p, per_unit, (int)items); \
  else gather_kernel<TT, DD><<<grid, 128, 0, st>>>(p);
  if (dtype == MPC_BF16) {
    if (D == 64) { MPC_GATHER(bf16, 64) }
    else { MPC_GATHER(bf16, 128) }
  } else {
    if (D == 64) { MPC_GATHER(float, 64) }
    else { MPC_GATHER(float, 128) }
  }
#undef MPC_GATHER
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (p.pyr.n_levels > 1 && any_leader) {
    if (D == 64) coarse_kernel<64><<<n_units, 256, 0, st>>>(p);
    else coarse_kernel<128><<<n_units, 256, 0, st>>>(p);
    e = cudaGetLastError();
  }
  return e;
}

int take_status_clusters() { return take_status(); }

}  // namespace mpc
