// Read floor of one decode step's attention traffic (measurement for
// bench.py --report read-floor; not part of the library).
//
// The sparse attention of a decode step reads, for every (layer, kv head)
// unit, the K and V rows of its selected clusters (16-row runs of 256-byte
// bf16 rows, one 4 KB K tile and one 4 KB V tile per cluster) and its tail,
// scattered over that unit's cache.  This program reads the same pattern and
// nothing else: a persistent grid (one CTA per SM, W warps, NST cp.async ring
// stages of one K + V tile pair per warp, warp ranges cut from one list of
// all tiles like the attention kernel's), each lane folding what it loaded
// into one word so no load is dead.  It reports the time per launch (CUDA
// events, after warm-up, L2 flushed by a 512 MB write before every launch)
// at the step's size and at 2, 4, 8 and 16 times its tiles, so the fixed
// cost of a launch of this size shows against the copy rate; and at the
// step's size once more with the same tiles read again right before (no
// flush: the step's bytes then come from L2).
//
// usage: bench_floor <units> <clusters per unit> <selected per unit>
//                    <cache rows per unit> <warps per CTA> <stages> <seed>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <random>
#include <vector>

#define CK(x)                                                                            \
  do {                                                                                   \
    cudaError_t e_ = (x);                                                                \
    if (e_ != cudaSuccess) {                                                             \
      std::fprintf(stderr, "%s:%d %s\n", __FILE__, __LINE__, cudaGetErrorString(e_));   \
      std::exit(1);                                                                      \
    }                                                                                    \
  } while (0)

constexpr int kRowBytes = 256;             // one bf16 row of d = 128
constexpr int kTileBytes = 16 * kRowBytes;  // 16 rows

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void cp16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void wait_groups() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// tiles[i] = byte offset of tile i's K rows (its V rows sit at the same
// offset in the V buffer); warp w of the grid takes tiles [w NT / NW, ...).
template <int NST>
__global__ void floor_kernel(const uint8_t* __restrict__ kc, const uint8_t* __restrict__ vc,
                             const long long* __restrict__ tiles, long long n_tiles, uint32_t* sink) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int wpc = blockDim.x >> 5;
  const long long nw = (long long)gridDim.x * wpc;
  const long long gw = (long long)warp * gridDim.x + blockIdx.x;  // slots interleaved over the CTAs
  const long long x0 = n_tiles * gw / nw, x1 = n_tiles * (gw + 1) / nw;
  uint8_t* ring = smem + (size_t)warp * NST * 2 * kTileBytes;
  uint32_t acc = 0;
  auto issue = [&](long long x, int slot) {
    const long long off = tiles[x];
    uint8_t* sk = ring + (size_t)slot * 2 * kTileBytes;
    for (int c = lane; c < kTileBytes / 16; c += 32) {
      cp16(sk + c * 16, kc + off + c * 16);
      cp16(sk + kTileBytes + c * 16, vc + off + c * 16);
    }
  };
  const long long n = x1 - x0;
  for (int j = 0; j < NST; ++j) {
    if (j < n) issue(x0 + j, j);
    commit();
  }
  for (long long j = 0; j < n; ++j) {
    wait_groups<NST - 1>();
    __syncwarp();
    const uint8_t* s = ring + (size_t)(j % NST) * 2 * kTileBytes;
    for (int c = lane; c < 2 * kTileBytes / 16; c += 32) {
      const uint4 v = reinterpret_cast<const uint4*>(s)[c];
      acc ^= v.x ^ v.y ^ v.z ^ v.w;
    }
    __syncwarp();
    if (j + NST < n) issue(x0 + j + NST, (int)((j + NST) % NST));
    commit();
  }
  wait_groups<0>();
  if (acc == 0x9e3779b9u) sink[0] = acc;  // keeps the loads live
}

__global__ void flush_kernel(uint4* buf, size_t n) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x)
    buf[i] = make_uint4((uint32_t)i, 1u, 2u, 3u);
}

int main(int argc, char** argv) {
  if (argc != 8) {
    std::fprintf(stderr, "usage: %s units clusters selected cache_rows warps stages seed\n", argv[0]);
    return 2;
  }
  const int units = std::atoi(argv[1]), clusters = std::atoi(argv[2]), selected = std::atoi(argv[3]);
  const long long cache_rows = std::atoll(argv[4]);
  const int wpc = std::atoi(argv[5]), nst = std::atoi(argv[6]);
  const unsigned seed = (unsigned)std::atoi(argv[7]);
  if (units < 1 || clusters < 1 || selected < 1 || selected > clusters || cache_rows < 16LL * (clusters + 1) ||
      wpc < 1 || wpc > 16 || !(nst == 2 || nst == 3 || nst == 4 || nst == 5 || nst == 6 || nst == 8 || nst == 12)) {
    std::fprintf(stderr, "bad arguments\n");
    return 2;
  }
  int dev = 0, sms = 0;
  CK(cudaGetDevice(&dev));
  CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  const int max_rep = 16;
  const size_t unit_bytes = (size_t)cache_rows * kRowBytes;
  const size_t cache_bytes = unit_bytes * units * max_rep;  // a separate cache per repetition of the step
  uint8_t *kc = nullptr, *vc = nullptr;
  CK(cudaMalloc(&kc, cache_bytes));
  CK(cudaMalloc(&vc, cache_bytes));
  CK(cudaMemset(kc, 1, cache_bytes));
  CK(cudaMemset(vc, 2, cache_bytes));
  // the step's tiles: per unit `selected` distinct clusters (ascending, as
  // the selection lists them), then the tail tile after the last cluster
  std::mt19937 rng(seed);
  std::vector<long long> all;
  for (int r = 0; r < max_rep; ++r)
    for (int u = 0; u < units; ++u) {
      std::vector<int> ids(clusters);
      for (int i = 0; i < clusters; ++i) ids[i] = i;
      std::shuffle(ids.begin(), ids.end(), rng);
      ids.resize(selected);
      std::sort(ids.begin(), ids.end());
      const long long base = (long long)(r * units + u) * (long long)unit_bytes;
      for (int c : ids) all.push_back(base + (long long)c * kTileBytes);
      all.push_back(base + (long long)clusters * kTileBytes);
    }
  long long* d_tiles = nullptr;
  uint32_t* sink = nullptr;
  CK(cudaMalloc(&d_tiles, all.size() * sizeof(long long)));
  CK(cudaMemcpy(d_tiles, all.data(), all.size() * sizeof(long long), cudaMemcpyHostToDevice));
  CK(cudaMalloc(&sink, 16));
  const size_t flush_n = (512ull << 20) / sizeof(uint4);
  uint4* flush = nullptr;
  CK(cudaMalloc(&flush, flush_n * sizeof(uint4)));
  const int smem = wpc * nst * 2 * kTileBytes;
  if (smem > 227 * 1024) {
    std::fprintf(stderr, "%d warps x %d stages need %d bytes of shared memory (227 KB at most)\n", wpc, nst, smem);
    return 2;
  }
  auto kern = nst == 2 ? floor_kernel<2>
              : nst == 3 ? floor_kernel<3>
              : nst == 4 ? floor_kernel<4>
              : nst == 5 ? floor_kernel<5>
              : nst == 6 ? floor_kernel<6>
              : nst == 8 ? floor_kernel<8>
                         : floor_kernel<12>;
  CK(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
  const long long step_tiles = (long long)units * (selected + 1);
  cudaEvent_t a, b;
  CK(cudaEventCreate(&a));
  CK(cudaEventCreate(&b));
  std::printf("{\"units\": %d, \"tiles_per_unit\": %d, \"grid\": %d, \"warps\": %d, \"stages\": %d, \"runs\": [",
              units, selected + 1, sms, wpc, nst);
  const int mults[5] = {1, 2, 4, 8, 16};
  for (int mi = 0; mi < 5; ++mi) {
    const long long nt = step_tiles * mults[mi];
    std::vector<float> ms;
    for (int it = 0; it < 8; ++it) {
      flush_kernel<<<sms * 4, 256>>>(flush, flush_n);
      CK(cudaEventRecord(a));
      kern<<<sms, wpc * 32, smem>>>(kc, vc, d_tiles, nt, sink);
      CK(cudaEventRecord(b));
      CK(cudaEventSynchronize(b));
      float t = 0.f;
      CK(cudaEventElapsedTime(&t, a, b));
      if (it >= 3) ms.push_back(t);
    }
    CK(cudaGetLastError());
    std::sort(ms.begin(), ms.end());
    const double us = ms[ms.size() / 2] * 1e3;
    const double bytes = (double)nt * 2 * kTileBytes;
    std::printf("%s{\"tiles\": %lld, \"mbytes\": %.1f, \"us\": %.2f, \"gbs\": %.0f}", mi ? ", " : "", nt,
                bytes / 1e6, us, bytes / us / 1e3);
  }
  // warm: the step's tiles twice in a row, the second launch timed
  std::vector<float> wms;
  for (int it = 0; it < 8; ++it) {
    kern<<<sms, wpc * 32, smem>>>(kc, vc, d_tiles, step_tiles, sink);
    CK(cudaEventRecord(a));
    kern<<<sms, wpc * 32, smem>>>(kc, vc, d_tiles, step_tiles, sink);
    CK(cudaEventRecord(b));
    CK(cudaEventSynchronize(b));
    float t = 0.f;
    CK(cudaEventElapsedTime(&t, a, b));
    if (it >= 3) wms.push_back(t);
  }
  std::sort(wms.begin(), wms.end());
  std::printf("], \"warm_step_us\": %.2f}\n", wms[wms.size() / 2] * 1e3);
  CK(cudaDeviceSynchronize());
  return 0;
}
