// Hierarchical cluster selection of one decode step (Sec. 3.3-3.4, Eq. 3;
// Alg. 2 Step 2, Sim + topk) for the leader layer of each sharing group.
//
// One CTA per (ref, sequence b, kv head h).  The GQA group's queries are
// summed once (Eq. 3 is linear in q, so the sum scores the group), then the
// levels are walked from the coarsest down: a warp per candidate computes
// q_sum . rep over d channels (float4 loads of the fp32 representative), a
// block bitonic sort of 64-bit keys (orderable score, inverted id) finds the
// k-th key, and an order-preserving compaction keeps the candidates at or
// above it, so the kept ids stay ascending.  The children of the kept
// clusters are the next level's candidates.
#include "kernels.cuh"

namespace mpc {


constexpr int kSelThreads = 256;

__device__ __forceinline__ unsigned long long sel_key(float score, int id) {
  return ((unsigned long long)orderable(score) << 32) | (unsigned long long)(0xffffffffu - (uint32_t)id);
}

// Exclusive prefix sum over the block (blockDim.x == kSelThreads).
__device__ __forceinline__ int block_exclusive_scan(int v, int* warp_tot, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_tot[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int t = (lane < kSelThreads / 32) ? warp_tot[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, t, o);
      if (lane >= o) t += y;
    }
    if (lane < kSelThreads / 32) warp_tot[lane] = t;
    if (lane == kSelThreads / 32 - 1) *total = t;
  }
  __syncthreads();
  const int before = (warp > 0 ? warp_tot[warp - 1] : 0) + x - v;
  __syncthreads();
  return before;
}

template <typename T, int D>
__global__ void __launch_bounds__(kSelThreads) select_kernel(const __grid_constant__ SelectParams p) {
  extern __shared__ __align__(16) uint8_t smem[];
  const int MC = p.max_cand;
  float* qsum = reinterpret_cast<float*>(smem);
  unsigned long long* keys = reinterpret_cast<unsigned long long*>(qsum + D);
  int* cand = reinterpret_cast<int*>(keys + MC);
  float* score = reinterpret_cast<float*>(cand + MC);
  int* kept = reinterpret_cast<int*>(score + MC);
  __shared__ int warp_tot[32];
  __shared__ int s_total, s_ncand;
  __shared__ unsigned long long s_thr;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int unit = blockIdx.x;
  const int h = unit % p.Hkv, b = (unit / p.Hkv) % p.B, ri = unit / (p.Hkv * p.B);
  const int layer = p.refs.layer[ri], group = p.refs.group[ri];
  const int G = p.G;

  // q_sum = sum over the group's query heads (fixed order)
  const T* qp = (const T*)p.q + layer * p.q_ls + ((int64_t)b * p.Hq + h * G) * D;
  for (int c = tid; c < D; c += blockDim.x) {
    float acc = 0.f;
    for (int g = 0; g < G; ++g) acc += to_float<T>(qp[g * D + c]);
    qsum[c] = acc;
  }

  int C[kMaxLevels];
  level_counts(p.pyr, p.n_tok[b], C);
  const int64_t ubase = ((int64_t)(group * p.B + b) * p.Hkv + h) * p.pyr.rows;
  int* out = p.out_sel + ((int64_t)(group * p.B + b) * p.Hkv + h) * p.sel_cap;

  const int top = p.pyr.n_levels - 1;
  bool overflow = C[0] > p.pyr.cap[0];
  if (tid == 0) s_ncand = min(C[top], MC);
  if (C[top] > MC) overflow = true;
  for (int i = tid; i < min(C[top], MC); i += blockDim.x) cand[i] = i;
  __syncthreads();

  int nk = 0;
  for (int l = top; l >= 0 && !overflow; --l) {
    const int n_cand = s_ncand;
    // Eq. 3 similarity of every candidate: a warp takes 4 candidates at a
    // time so that four independent row loads are in flight per lane
    const float* rep = p.rep + (ubase + p.pyr.off[l]) * D;
    for (int i0 = warp * 4; i0 < n_cand; i0 += (kSelThreads / 32) * 4) {
      float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int c4 = lane; c4 < D / 4; c4 += 32) {
        const float4 qv = *reinterpret_cast<const float4*>(qsum + 4 * c4);
        float4 r[4];
#pragma unroll
        for (int u = 0; u < 4; ++u)
          r[u] = (i0 + u < n_cand) ? __ldg(reinterpret_cast<const float4*>(rep + (int64_t)cand[i0 + u] * D) + c4)
                                   : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          acc[u] = fmaf(r[u].x, qv.x, acc[u]);
          acc[u] = fmaf(r[u].y, qv.y, acc[u]);
          acc[u] = fmaf(r[u].z, qv.z, acc[u]);
          acc[u] = fmaf(r[u].w, qv.w, acc[u]);
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) acc[u] = warp_sum(acc[u]);
      if (lane < 4 && i0 + lane < n_cand) {
        const float a = lane == 0 ? acc[0] : lane == 1 ? acc[1] : lane == 2 ? acc[2] : acc[3];
        score[i0 + lane] = a;
        keys[i0 + lane] = sel_key(a, cand[i0 + lane]);
      }
    }
    const int k = min(count_from_ppm(C[l], p.keep_ppm[l]), n_cand);
    __syncthreads();
    unsigned long long thr = 0ull;
    if (k < n_cand && n_cand <= 2 * kSelThreads) {
      // rank of each candidate = number of larger keys (keys are distinct);
      // the key of rank k - 1 is the k-th largest
      for (int i = tid; i < n_cand; i += blockDim.x) {
        const unsigned long long ki = keys[i];
        int rank = 0;
        for (int j = 0; j < n_cand; ++j) rank += keys[j] > ki;
        if (rank == k - 1) s_thr = ki;
      }
      __syncthreads();
      thr = s_thr;
    } else if (k < n_cand) {
      int P = 1;
      while (P < n_cand) P <<= 1;
      for (int i = n_cand + tid; i < P; i += blockDim.x) keys[i] = 0ull;
      __syncthreads();
      // bitonic sort, descending
      for (int kk = 2; kk <= P; kk <<= 1) {
        for (int j = kk >> 1; j > 0; j >>= 1) {
          for (int i = tid; i < P; i += blockDim.x) {
            const int ixj = i ^ j;
            if (ixj > i) {
              const unsigned long long a = keys[i], bb = keys[ixj];
              const bool desc = (i & kk) == 0;
              if (desc ? (a < bb) : (a > bb)) {
                keys[i] = bb;
                keys[ixj] = a;
              }
            }
          }
          __syncthreads();
        }
      }
      thr = keys[k - 1];
    }
    // order-preserving compaction of the kept candidates
    const int per = (n_cand + kSelThreads - 1) / kSelThreads;
    const int i0 = tid * per, i1 = min(n_cand, i0 + per);
    int cnt = 0;
    for (int i = i0; i < i1; ++i) cnt += (sel_key(score[i], cand[i]) >= thr);
    const int off = block_exclusive_scan(cnt, warp_tot, &s_total);
    for (int i = i0, o = off; i < i1; ++i)
      if (sel_key(score[i], cand[i]) >= thr) kept[o++] = cand[i];
    __syncthreads();
    nk = s_total;
    if (l == 0) break;
    // children of the kept clusters become the next candidates
    const int f = p.pyr.fanout[l - 1];
    const int n_child = C[l - 1];
    const int perk = (nk + kSelThreads - 1) / kSelThreads;
    const int k0 = tid * perk, k1 = min(nk, k0 + perk);
    int ccount = 0;
    for (int i = k0; i < k1; ++i) ccount += min(f, n_child - kept[i] * f);
    const int coff = block_exclusive_scan(ccount, warp_tot, &s_total);
    if (s_total > MC) {
      overflow = true;
      break;
    }
    for (int i = k0, o = coff; i < k1; ++i) {
      const int c0 = kept[i] * f, c1 = min(c0 + f, n_child);
      for (int c = c0; c < c1; ++c) cand[o++] = c;
    }
    if (tid == 0) s_ncand = s_total;
    __syncthreads();
  }
  if (overflow || nk > p.sel_cap) {
    if (tid == 0) atomicOr(&g_mpc_status, 4);
    nk = 0;
  }
  for (int i = tid; i < p.sel_cap; i += blockDim.x) out[i] = (i < nk) ? kept[i] : -1;
  if (tid == 0 && h == 0 && ri == 0) p.out_n_sel[b] = nk;
}

int select_smem_bytes(int D, int max_cand) {
  return D * 4 + max_cand * (8 + 4 + 4 + 4);
}

template <typename K>
static cudaError_t launch_sel(K kernel, int units, int smem, cudaStream_t st, const SelectParams& p) {
  cudaError_t e = ensure_dyn_smem((const void*)kernel, smem);
  if (e != cudaSuccess) return e;
  kernel<<<units, kSelThreads, smem, st>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_select(const SelectParams& p, int dtype, int D, int units, cudaStream_t st) {
  const int smem = select_smem_bytes(D, p.max_cand);
  if (dtype == MPC_BF16) {
    if (D == 64) return launch_sel(select_kernel<bf16, 64>, units, smem, st, p);
    return launch_sel(select_kernel<bf16, 128>, units, smem, st, p);
  }
  if (D == 64) return launch_sel(select_kernel<float, 64>, units, smem, st, p);
  return launch_sel(select_kernel<float, 128>, units, smem, st, p);
}

int take_status_select() { return take_status(); }

}  // namespace mpc
