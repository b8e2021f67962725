// Commonality of the selected clusters across adjacent layers (Sec. 2,
// Observation 3): for index sets S_0 .. S_{L-1} of consecutive layers,
//   score = sum over l < L - m of |S_l n S_{l+1} n ... n S_{l+m}| / (k (L - m)),
// the statistic behind cross-layer index sharing (Sec. 3.4).  One CTA per
// (sequence, kv head) marks each layer's selected ids in a shared-memory
// bitmap, then counts the ids present in every layer of each window of m + 1
// layers with 32-bit AND + popcount over the bitmap words.
#include <cstdio>

#include "kernels.cuh"

namespace mpc {
namespace {

constexpr int kComThreads = 256;

__global__ void __launch_bounds__(kComThreads) commonality_kernel(const int32_t* sel, int64_t ls, int sel_cap,
                                                                   int k, int L, int m, int B, int Hkv, int words,
                                                                   int32_t* out_total, float* out_score) {
  extern __shared__ uint32_t bits[];  // [L][words]
  const int b = blockIdx.x / Hkv, h = blockIdx.x % Hkv;
  for (int i = threadIdx.x; i < L * words; i += blockDim.x) bits[i] = 0u;
  __syncthreads();
  // the first k entries of every layer's list (ids ascending, -1 padded)
  for (int i = threadIdx.x; i < L * k; i += blockDim.x) {
    const int l = i / k, j = i - l * k;
    const int id = sel[l * ls + ((int64_t)b * Hkv + h) * sel_cap + j];
    if (id >= 0 && id < words * 32) atomicOr(&bits[l * words + (id >> 5)], 1u << (id & 31));
    else if (id >= words * 32) atomicOr(&g_mpc_status, 4);
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
    out_score[blockIdx.x] = (float)s_total / ((float)k * (float)(L - m));
  }
}

}  // namespace

int take_status_commonality() { return take_status(); }

}  // namespace mpc

extern "C" MPC_API int mpc_commonality(const mpc_commonality_args* a, void* stream) {
  using namespace mpc;
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
  cudaError_t e = ensure_dyn_smem((const void*)commonality_kernel, (int)smem);
  if (e != cudaSuccess) return set_error(MPC_ERR_CUDA, cudaGetErrorString(e));
  commonality_kernel<<<a->batch * a->n_kv_heads, kComThreads, smem, static_cast<cudaStream_t>(stream)>>>(
      a->sel, a->sel_layer_stride, a->sel_cap, a->k, a->n_layers, a->m, a->batch, a->n_kv_heads, words,
      a->out_total, a->out_score);
  e = cudaGetLastError();
  if (e != cudaSuccess) return set_error(MPC_ERR_CUDA, cudaGetErrorString(e));
  return MPC_OK;
}
