// Device helpers shared by the MPCache kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <map>
#include <mutex>
#include <utility>

#include "../../include/mpcache.h"

namespace mpc {

typedef __nv_bfloat16 bf16;

constexpr int kMaxRefs = MPC_MAX_REFS;
constexpr int kMaxLevels = MPC_MAX_LEVELS;
constexpr int kSmemOptin = 232448;  // shared memory per CTA on sm_103a (227 KB)

constexpr float kPosInf = __builtin_huge_valf();
constexpr float kNegInf = -__builtin_huge_valf();

// Status bits of the device status word (mpc_device_status).
constexpr int kStatusWaitTimeout = 1;

// Per-call layer table, passed by value to every kernel.
struct RefTable {
  int32_t layer[kMaxRefs];
  int32_t group[kMaxRefs];
  int8_t leader[kMaxRefs];
};

// Geometry of a summary pyramid (levels indexed from 0 = finest).
struct Pyramid {
  int n_levels;
  int s;                     // tokens per finest cluster
  int fanout[kMaxLevels];    // fanout[l]: level-l clusters under one level-(l+1) cluster
  int cap[kMaxLevels];       // rows reserved per level
  int off[kMaxLevels];       // first row of each level
  int rows;                  // total rows
};

// Counts of clusters per level for n cache rows: level 0 has floor(n / s)
// full clusters, level l+1 has ceil(C_l / fanout[l]).
__device__ __forceinline__ void level_counts(const Pyramid& p, int n, int* C) {
  C[0] = n / p.s;
#pragma unroll
  for (int l = 1; l < kMaxLevels; ++l)
    C[l] = (l < p.n_levels) ? (C[l - 1] + p.fanout[l - 1] - 1) / p.fanout[l - 1] : 0;
}

// min(N, max(1, ceil(N * ppm / 1e6))), 0 for N = 0.
__host__ __device__ __forceinline__ int count_from_ppm(int n, int ppm) {
  if (n <= 0) return 0;
  long long k = ((long long)n * ppm + 999999LL) / 1000000LL;
  if (k < 1) k = 1;
  if (k > n) k = n;
  return (int)k;
}

// Total order on float scores as unsigned keys (larger float -> larger key).
__device__ __forceinline__ uint32_t orderable(float f) {
  uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Element offset of (row, col) inside the row-swizzled cluster-major cache:
// logical 16-byte chunk j of row i lives at chunk j ^ (i & 7).
template <typename T>
__host__ __device__ __forceinline__ int swz(int row, int col) {
  constexpr int E = 16 / (int)sizeof(T);
  return ((col / E) ^ (row & 7)) * E + (col % E);
}

template <typename T> __device__ __forceinline__ float to_float(T x);
template <> __device__ __forceinline__ float to_float<float>(float x) { return x; }
template <> __device__ __forceinline__ float to_float<bf16>(bf16 x) { return __bfloat162float(x); }

// ---------------------------------------------------------------- PTX ----

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// Orders this thread's generic-proxy shared-memory accesses before later
// async-proxy (bulk copy) accesses.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n"
      " mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Release reduction (orders this thread's earlier writes, and those ordered
// before it by a barrier, before the add) and acquire load, at gpu scope.
__device__ __forceinline__ void red_release_add(int* addr, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(addr), "r"(v) : "memory");
}
__device__ __forceinline__ int ld_acquire(const int* addr) {
  int v;
  asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(addr) : "memory");
  return v;
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// One status word per translation unit (internal linkage; no device linking
// needed).  Bits: 1 a bounded wait gave up, 2 a cache or pyramid capacity was
// too small for the device-side counts, 4 a selection or window exceeded the
// sizes the call was configured for.
static __device__ int g_mpc_status = 0;

static inline int take_status() {
  int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_mpc_status, sizeof(int)) != cudaSuccess) return -1;
  if (cudaMemcpyToSymbol(g_mpc_status, &z, sizeof(int)) != cudaSuccess) return -1;
  return v;
}

// Programmatic dependent launch.  The per-step kernels are launched with
// cudaLaunchAttributeProgrammaticStreamSerialization, so a kernel may become
// resident while the previous kernel of the stream is still running.  Every
// such kernel calls grid_dep_wait() before its first access to global memory
// that an earlier launch may write; grid_dep_wait() returns once all earlier
// grids have completed and their writes are visible (a no-op for a kernel
// launched without the attribute).  grid_dep_launch() lets the next kernel of
// the stream start its own launch early.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... P, typename... A>
inline cudaError_t launch_pdl(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              A&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<A>(args)...);
}

// launch_pdl for a kernel whose CTAs wait on one another: a cooperative
// launch, which starts the grid only when every CTA can be resident at once
// (and fails, with nothing launched, for a grid that could never be), so
// every such wait ends.
template <typename... P, typename... A>
inline cudaError_t launch_pdl_coop(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                                   A&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  at[1].id = cudaLaunchAttributeCooperative;
  at[1].val.cooperative = 1;
  cfg.attrs = at;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<A>(args)...);
}

// Raises a kernel's dynamic shared-memory limit once per (kernel, device), so
// later launches (including ones recorded into a CUDA graph) skip the call.
inline cudaError_t ensure_dyn_smem(const void* kernel, int bytes) {
  static std::mutex mu;
  static std::map<std::pair<const void*, int>, int> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lk(mu);
  const auto key = std::make_pair(kernel, dev);
  const auto it = done.find(key);
  if (it != done.end() && it->second >= bytes) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done[key] = bytes;
  return e;
}

// Waits for the phase of `bar` with parity `parity`, giving up after
// `limit_ns`.  On timeout sets the status word and returns false.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  uint64_t limit_ns = 1000000000ull) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > limit_ns) {
      atomicOr(&g_mpc_status, kStatusWaitTimeout);
      return false;
    }
  }
  return true;
}

// 16-byte asynchronous copy global -> shared (cached in L2 only), and its
// commit / wait-group pair.
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// 1-D bulk copy global -> shared (TMA engine), completion counted on `bar`.
// dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// D = A(16x16 bf16, row) * B(16x8 bf16, col) + D (fp32).
__device__ __forceinline__ void mma_bf16(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// ------------------------------------------------------- reductions ----

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

}  // namespace mpc
