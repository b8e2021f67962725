// Commonality of the selected clusters across adjacent layers (Sec. 2,
// Observation 3): for index sets S_0 .. S_{L-1} of consecutive layers,
//   score = sum over l < L - m of |S_l n S_{l+1} n ... n S_{l+m}| / (k (L - m)),
// the statistic behind cross-layer index sharing (Sec. 3.4).  One CTA per
// (sequence, kv head) marks each layer's selected ids in a shared-memory
// bitmap, then counts the ids present in every layer of each window of m + 1
// layers with 32-bit AND + popcount over the bitmap words.  With a kept map
// the marked ids are the token positions of the selected clusters' rows
// (the prompt position of a kept row, prompt_len + offset for an appended
// row), so layers with different kept sets compare the same tokens.
#include <cstdio>

#include "kernels.cuh"

namespace mpc {
namespace {

constexpr int kComThreads = 256;

struct PosMap {
  const int32_t* kept;  // NULL: compare cluster ids
  int64_t kls;
  int kept_cap, s;
  const int32_t* n_keep;
  const int32_t* plen;
};

__global__ void __launch_bounds__(kComThreads) commonality_kernel(const int32_t* sel, int64_t ls, int sel_cap,
                                                                   int k, int L, int m, int B, int Hkv, int words,
                                                                   PosMap pm, int32_t* out_total, float* out_score) {
  extern __shared__ uint32_t bits[];  // [L][words]
  const int b = blockIdx.x / Hkv, h = blockIdx.x % Hkv;
  for (int i = threadIdx.x; i < L * words; i += blockDim.x) bits[i] = 0u;
  __syncthreads();
  // the first k entries of every layer's list (ids ascending, -1 padded),
  // each as its s row positions when mapped
  const int S = pm.kept != nullptr ? pm.s : 1;
  const int nk = pm.kept != nullptr ? pm.n_keep[b] : 0;
  const int T = pm.kept != nullptr ? pm.plen[b] : 0;
  for (int i = threadIdx.x; i < L * k * S; i += blockDim.x) {
    const int l = i / (k * S), jt = i - l * (k * S), j = jt / S, t = jt - j * S;
    const int id = sel[l * ls + ((int64_t)b * Hkv + h) * sel_cap + j];
    if (id < 0) continue;
    int x = id;
    if (pm.kept != nullptr) {
      const long long r = (long long)id * S + t;  // cache row
      if (r < nk) {
        if (r >= pm.kept_cap) {
          atomicOr(&g_mpc_status, 4);
          continue;
        }
        x = pm.kept[l * pm.kls + ((int64_t)b * Hkv + h) * pm.kept_cap + r];
      } else {
        const long long p = T + (r - nk);
        x = p < (long long)words * 32 ? (int)p : words * 32;
      }
    }
    if (x >= 0 && x < words * 32) atomicOr(&bits[l * words + (x >> 5)], 1u << (x & 31));
    else atomicOr(&g_mpc_status, 4);
  }
  __syncthreads();
  __shared__ int s_total;
  if (threadIdx.x == 0) s_total = 0;
  __syncthreads();
  int cnt = 0;
  for (int i = threadIdx.x; i < (L - m) * words; i += blockDim.x) {
    const int l = i / words, wd = i - l * words;
    uint32_t x = bits[l * words + wd];
    for (int t = 1; t <= m; ++t) x &= bits[(l + t) * words + wd];
    cnt += __popc(x);
  }
  atomicAdd(&s_total, cnt);
  __syncthreads();
  if (threadIdx.x == 0) {
    out_total[blockIdx.x] = s_total;
    out_score[blockIdx.x] = (float)((double)s_total / ((double)k * S * (L - m)));
  }
}

}  // namespace

int take_status_commonality() { return take_status(); }

}  // namespace mpc

extern "C" MPC_API int mpc_commonality(const mpc_commonality_args* a, void* stream) {
  using namespace mpc;
  NvtxRange nvtx("mpc_commonality");
  if (a == nullptr) return set_error(MPC_ERR_INVALID_ARG, "args is NULL");
  if (a->struct_size != sizeof(mpc_commonality_args))
    return set_error(MPC_ERR_INVALID_ARG, "struct_size does not match sizeof(mpc_commonality_args)");
  if (a->n_layers < 2 || a->batch < 1 || a->n_kv_heads < 1 || a->sel_cap < 1)
    return set_error(MPC_ERR_BAD_SHAPE, "need n_layers >= 2, batch, n_kv_heads and sel_cap >= 1");
  if (a->m < 1 || a->m >= a->n_layers) return set_error(MPC_ERR_BAD_SHAPE, "m must be in [1, n_layers)");
  if (a->k < 1 || a->k > a->sel_cap) return set_error(MPC_ERR_BAD_SHAPE, "k must be in [1, sel_cap]");
  if (a->n_clusters < 1 || a->sel_layer_stride < (int64_t)a->batch * a->n_kv_heads * a->sel_cap)
    return set_error(MPC_ERR_BAD_SHAPE, "n_clusters >= 1 and a layer stride covering [batch][n_kv_heads][sel_cap]");
  const int words = (a->n_clusters + 31) / 32;
  const size_t smem = (size_t)a->n_layers * words * 4;
  if (smem > (size_t)kSmemOptin) return set_error(MPC_ERR_BAD_SHAPE, "n_layers x n_clusters bitmap exceeds shared memory");
  if (a->sel == nullptr || a->out_total == nullptr || a->out_score == nullptr)
    return set_error(MPC_ERR_INVALID_ARG, "a required pointer is NULL");
  if ((int64_t)a->batch * a->n_kv_heads > 65535 * 32) return set_error(MPC_ERR_BAD_SHAPE, "too many (b, h) units");
  PosMap pm{a->kept, a->kept_layer_stride, a->kept_cap, a->cluster_size, a->n_keep, a->prompt_len};
  if (pm.kept != nullptr) {
    if (pm.n_keep == nullptr || pm.plen == nullptr)
      return set_error(MPC_ERR_INVALID_ARG, "kept needs n_keep and prompt_len");
    if (pm.s < 1 || pm.kept_cap < 1 || pm.kls < (int64_t)a->batch * a->n_kv_heads * pm.kept_cap)
      return set_error(MPC_ERR_BAD_SHAPE, "cluster_size, kept_cap >= 1 and a kept layer stride covering [batch][n_kv_heads][kept_cap]");
    if ((int64_t)a->n_layers * a->k * pm.s > (int64_t)1 << 30)
      return set_error(MPC_ERR_BAD_SHAPE, "n_layers x k x cluster_size too large");
  }
  cudaError_t e = ensure_dyn_smem((const void*)commonality_kernel, (int)smem);
  if (e != cudaSuccess) return set_error(MPC_ERR_CUDA, cudaGetErrorString(e));
  commonality_kernel<<<a->batch * a->n_kv_heads, kComThreads, smem, static_cast<cudaStream_t>(stream)>>>(
      a->sel, a->sel_layer_stride, a->sel_cap, a->k, a->n_layers, a->m, a->batch, a->n_kv_heads, words, pm,
      a->out_total, a->out_score);
  e = cudaGetLastError();
  if (e != cudaSuccess) return set_error(MPC_ERR_CUDA, cudaGetErrorString(e));
  return MPC_OK;
}
