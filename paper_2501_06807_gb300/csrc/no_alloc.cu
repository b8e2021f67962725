// Decode attention for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc at all: code that runs inside a
// memory-pool-managed runtime that forbids raw allocations, plugins handed
// only fixed input/output buffers by their host, or paths that must not
// allocate after start-up (allocation can block or fail).  The regular
// mpc_sparse_decode_attn asks its caller for a workspace; this entry point
// instead uses a fixed scratch array that lives in the library's own device
// image, so the caller passes only inputs and outputs.
//
// The array is a file-scope __device__ variable.  Host code cannot use its
// name as a device address, so every call looks the address up with
// cudaGetSymbolAddress in the current device's context.
#include "kernels.cuh"

namespace mpc {
namespace {

constexpr size_t kStaticScratchBytes = size_t(4) << 20;  // 4 MiB per device

static __device__ __align__(256) unsigned char g_attn_scratch[kStaticScratchBytes];

// Device address of g_attn_scratch in the current device's context, looked
// up on every call (a cached address would dangle after a device reset or a
// switch of context on the same ordinal).
int scratch_address(void** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_attn_scratch);
  if (e != cudaSuccess || p == nullptr)
    return set_error(MPC_ERR_CUDA, "cudaGetSymbolAddress of the static scratch array failed");
  *out = p;
  return MPC_OK;
}

}  // namespace
}  // namespace mpc

extern "C" MPC_API int mpc_sparse_decode_attn_static_scratch(const mpc_attn_args* args, void* stream) {
  mpc::NvtxRange nvtx("mpc_sparse_decode_attn_static_scratch");
  using namespace mpc;
  size_t need = 0;
  int rc = mpc_sparse_decode_attn_workspace_size(args, &need);
  if (rc != MPC_OK) return rc;
  if (need > kStaticScratchBytes)
    return set_error(MPC_ERR_WORKSPACE,
                     "this call needs more scratch than the 4 MiB static array holds; "
                     "use mpc_sparse_decode_attn with a caller workspace");
  void* ws = nullptr;
  rc = scratch_address(&ws);
  if (rc != MPC_OK) return rc;
  // the counters must start at zero; the array keeps the previous call's
  // contents, so clear them (the partial records are written before they
  // are read)
  size_t coff = 0, cbytes = 0;
  rc = attn_counter_range(args, &coff, &cbytes);
  if (rc != MPC_OK) return rc;
  const cudaError_t e = cudaMemsetAsync(static_cast<uint8_t*>(ws) + coff, 0, cbytes, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return set_error(MPC_ERR_CUDA, cudaGetErrorString(e));
  return mpc_sparse_decode_attn(args, ws, need, stream);
}
