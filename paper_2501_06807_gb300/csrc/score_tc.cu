// Window scoring of look-once static eviction on the 5th-generation tensor
// cores (Sec. 3.2; Alg. 2 Step 1): the two passes of the accumulated window
// attention for bf16 queries and dense keys (paged keys arrive as a dense
// copy gathered by the caller, indexed by ref).
//
//   pass 0 (row statistics): one CTA per (ref, sequence, query head, 128
//     window rows).  A = the 128 query rows (fixed), B = 128-key tiles
//     streamed over every key a row can see.  S = A B^T lands in TMEM with
//     one window row per TMEM lane, so each epilogue thread owns a row and
//     keeps its online max m and sum l of 2^(s - m) without any cross-thread
//     reduction.
//   pass 1 (column sums): one CTA per (ref, sequence, kv head, 128 keys).
//     A = the 128 key rows (fixed), B = 128-row tiles of window queries of
//     every query head of the GQA group.  S^T = A B^T puts one key per TMEM
//     lane, so each thread sums 2^(s_ij - m_i) / l_i over the rows i in its
//     own registers, in a fixed order (deterministic scores).  The row
//     statistic -(m_i + log2 l_i) enters through the MMA itself: one extra
//     K = 16 step multiplies a constant key-side operand (1, 1, 1, 0, ...)
//     with the row's statistic over the log2 scale, stored by pass 0 as three
//     bf16 parts, so the accumulator holds s_ij + that value and the
//     epilogue needs one multiply, one ex2 and one add per score and no
//     shared-memory loads (every lane would need every row's value, and
//     broadcast loads were this pass's bound).
//   An item is one such 128-row block.  When an item has fewer than 32
//   tiles (short prompts, one query head per group), score_tc_items_kernel
//   gives each CTA several consecutive items instead of one, so that setup
//   and the filling and draining of its pipeline are paid once per CTA.

// Roles: warp 0 issues TMA tile loads (128B-swizzled, K-major boxes of
// 128 rows x 64 channels), warp 1 allocates TMEM and issues tcgen05.mma
// (M = N = 128, K = 16, bf16 in, fp32 accumulate) into one of two 128-column
// accumulators, and eight epilogue warps drain the other accumulator with
// tcgen05.ld: two warps per 32-lane quarter, each taking half of the 128
// columns, combined through shared memory at the end.  The epilogue is the
// bound (one ex2 per score), so its inner loops use packed f32x2 FMA / add
// and a three-input max, and compare keys against rows only on the tiles
// that cross the causal diagonal.  Every wait is bounded; a timeout sets
// the device status word and an abort flag that stops the other roles, and
// TMEM is always released.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "kernels.cuh"

namespace mpc {
namespace {

constexpr int kTcEpiWarps = 8;
constexpr int kTcEpiThreads = 32 * kTcEpiWarps;
constexpr int kTcThreads = 64 + kTcEpiThreads;
constexpr int kStagesTc = 2;
constexpr int kStatSlots = 4;  // row-statistics ring of pass 1 (tiles in flight ahead of the epilogue)
constexpr int kBoxBytes = 128 * 128;  // 128 rows x 64 bf16 channels
constexpr int kTilesPerCta = 32;      // below this many tiles per item, a CTA takes several items

template <int D>
struct TcSmem {
  static constexpr int KH = D / 64;                 // 64-channel halves
  static constexpr int TILE = KH * kBoxBytes;       // one 128-row operand tile
  static constexpr int A_OFF = 0;
  static constexpr int B_OFF = TILE;
  static constexpr int STAGE = TILE;                // one streamed B tile
  static constexpr int AUG_OFF = B_OFF + kStagesTc * STAGE;    // pass 1: kStatSlots x 128 rows x 16 B
  static constexpr int ONE_OFF = AUG_OFF + kStatSlots * 2048;   // pass 1: constant K-side core matrices
  static constexpr int XCH_OFF = ONE_OFF + 256;                 // halves' partials, 2 x 128 x float2
  static constexpr int BAR_OFF = XCH_OFF + 2 * 128 * 8;
  static constexpr int USED = BAR_OFF + 256 + 1024;  // + alignment slack
  // at least 80 KB so that at most two CTAs (2 x 256 TMEM columns) share an SM
  static constexpr int TOTAL = USED > 80 * 1024 ? USED : 80 * 1024;
};

__device__ __forceinline__ void epilogue_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kTcEpiThreads) : "memory"); }

// Packed pairs of fp32 (one 64-bit register pair) and the sm_100 f32x2 ops.
__device__ __forceinline__ uint64_t pk2(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void upk2(uint64_t r, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(r));
}
__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.ftz.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t fadd2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.ftz.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
// two ex2.approx (MUFU)
__device__ __forceinline__ uint64_t exp2_mufu2(uint64_t x2) {
  float x0, x1;
  upk2(x2, x0, x1);
  return pk2(fast_exp2(x0), fast_exp2(x1));
}

// max of 32 values, two independent chains of three-input max
__device__ __forceinline__ float max32(const float* v) {
  float a = fmax3(v[0], v[1], v[2]), b = fmax3(v[3], v[4], v[5]);
#pragma unroll
  for (int k = 6; k < 30; k += 4) {
    a = fmax3(a, v[k], v[k + 1]);
    b = fmax3(b, v[k + 2], v[k + 3]);
  }
  return fmax3(a, b, fmaxf(v[30], v[31]));
}

// ----------------------------------------------------------------- PTX ----

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int c0, int c1, int c2,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, "
      "%4}], [%5];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tmem_alloc(uint32_t* dst, uint32_t cols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst)), "r"(cols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t cols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(cols) : "memory");
}

// D[tmem] (+)= A[smem desc] * B[smem desc]^T, bf16 x bf16 -> fp32.
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrives on `bar` once every tcgen05.mma issued so far by this thread is done.
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

// 32 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,"
      "%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups
// 1024 bytes apart (the layout a 128B-swizzled TMA box of 128-byte rows
// produces).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;            // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;  // stride byte offset: next 8-row group
  d |= (uint64_t)1 << 46;            // descriptor version of tcgen05
  d |= (uint64_t)2 << 61;            // 128-byte swizzle
  return d;
}

// Shared-memory matrix descriptor without swizzle (K-major): 8-row x 16-byte
// core matrices stored as 128 contiguous bytes; `lbo` is the byte step
// between the two core matrices of a 16-element K step, `sbo` the step
// between 8-row groups.
__device__ __forceinline__ uint64_t plain_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;  // descriptor version of tcgen05; layout 0 = no swizzle
  return d;
}
__device__ __forceinline__ uint32_t pack_bf16_pair(bf16 lo, bf16 hi) {
  return (uint32_t)__bfloat16_as_ushort(lo) | ((uint32_t)__bfloat16_as_ushort(hi) << 16);
}

// Instruction descriptor: bf16 A and B (K-major), fp32 D, M = N = 128.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((128u >> 3) << 17) | ((128u >> 4) << 24);

// Bounded wait that also gives up when another role has aborted.
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (*abort) return false;
    if (global_timer_ns() - t0 > 1000000000ull) {
      atomicOr(&g_mpc_status, kStatusWaitTimeout);
      *abort = 1;
      return false;
    }
  }
  return true;
}

__device__ __forceinline__ int win_rows_of(const ScoreTcParams& p, int T) {
  return count_from_ppm(T, T > p.long_threshold ? p.long_window_ppm : p.window_ppm);
}

template <int PASS, int D>
__global__ void __launch_bounds__(kTcThreads, 2) score_tc_kernel(const __grid_constant__ ScoreTcParams p) {
  using S = TcSmem<D>;
  constexpr int KH = S::KH;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::BAR_OFF);
  uint64_t* empty = full + kStagesTc;
  uint64_t* a_full = empty + kStagesTc;
  uint64_t* acc_full = a_full + 1;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* stats_full = acc_empty + 2;
  uint64_t* stats_empty = stats_full + kStatSlots;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(stats_empty + kStatSlots);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // ---- work unit
  const int HEADS = PASS == 0 ? p.Hq : p.Hkv;
  const int unit = blockIdx.y;
  const int head = unit % HEADS, b = (unit / HEADS) % p.B, ri = unit / (HEADS * p.B);
  const int layer = p.refs.layer[ri], group = p.refs.group[ri];
  const int T_b = p.lens[b];
  const bool valid_len = T_b >= 1 && T_b <= p.t_max;
  const int w = valid_len ? win_rows_of(p, T_b) : 0;
  const int qoff = p.win_rows - w;
  const int base = T_b - w;  // position of window row 0
  int n_tiles = 0, i0 = 0, j0 = 0, i_start = 0, tiles_per_g = 0;
  if (valid_len && w <= p.win_rows) {
    if (PASS == 0) {
      i0 = blockIdx.x * 128;  // window rows of this CTA
      if (i0 < w) {
        const int pos_last = base + min(i0 + 127, w - 1);
        n_tiles = pos_last / 128 + 1;  // key tiles 0 .. pos_last
      }
    } else {
      j0 = blockIdx.x * 128;  // keys of this CTA
      if (j0 < T_b) {
        const int i_first = max(0, j0 - base);  // first row that sees key j0
        i_start = (i_first / 128) * 128;
        tiles_per_g = (w - i_start + 127) / 128;
        n_tiles = p.G * tiles_per_g;
      }
    }
  }
  // a CTA past its sequence's window (pass 0) or keys (pass 1) has nothing
  // to compute or write: leave before the barriers and the TMEM allocation
  // (ragged batches launch many of them)
  if (n_tiles == 0) return;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStagesTc; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(a_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kTcEpiWarps);
    }
    for (int i = 0; i < kStatSlots; ++i) {
      mbar_init(&stats_full[i], 1);
      mbar_init(&stats_empty[i], 1);  // released by the MMA that read the slot
    }
    *abort = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 256);
    tmem_relinquish();
  }
  if (PASS == 1 && threadIdx.x >= 64 && threadIdx.x < 80) {
    // K-side operand of the statistic step: one 8-row core matrix whose rows
    // are (1, 1, 1, 0, 0, 0, 0, 0) (every 8-row group reuses it), then a zero
    // core matrix for channels 8..15
    const int i = threadIdx.x - 64;
    reinterpret_cast<uint4*>(smem + S::ONE_OFF)[i] =
        i < 8 ? make_uint4(0x3F803F80u, 0x00003F80u, 0u, 0u) : make_uint4(0u, 0u, 0u, 0u);
    fence_proxy_async_smem();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0 && lane == 0 && n_tiles > 0) {
    // ---------------------------------------------------- TMA producer
    int n_issued = 0, n_stats = 0;
    const int qrow0 = (b * p.Hq) * p.win_rows + qoff;       // + hq * win_rows + i
    const int krow0 = (b * p.Hkv) * p.t_max;                 // + hk * t_max + j
    // keys [kj, kj + 128) of kv head hk: one 128-row box per 64-channel half
    auto load_keys = [&](uint8_t* dst, int hk, int kj, uint64_t* bar) {
      mbar_arrive_expect_tx(bar, S::TILE);
      for (int kh = 0; kh < KH; ++kh)
        tma_load_3d(dst + kh * kBoxBytes, &p.map_k, kh * 64, krow0 + hk * p.t_max + kj, p.k_by_ref ? ri : layer,
                    bar);
    };
    if (PASS == 0) {
      mbar_arrive_expect_tx(a_full, S::TILE);
      for (int kh = 0; kh < KH; ++kh)
        tma_load_3d(smem + S::A_OFF + kh * kBoxBytes, &p.map_q, kh * 64, qrow0 + head * p.win_rows + i0, layer, a_full);
    } else {
      load_keys(smem + S::A_OFF, head, j0, a_full);
    }
    for (int t = 0; t < n_tiles; ++t) {
      const int s = t % kStagesTc;
      if (t >= kStagesTc && !wait_or_abort(&empty[s], ((t / kStagesTc) - 1) & 1, abort)) break;
      uint8_t* st = smem + S::B_OFF + s * S::STAGE;
      if (PASS == 0) {
        load_keys(st, head / p.G, t * 128, &full[s]);
      } else {
        const int g = t / tiles_per_g, it = i_start + (t % tiles_per_g) * 128;
        const int hq = head * p.G + g;
        mbar_arrive_expect_tx(&full[s], S::TILE);
        for (int kh = 0; kh < KH; ++kh)
          tma_load_3d(st + kh * kBoxBytes, &p.map_q, kh * 64, qrow0 + hq * p.win_rows + it, layer, &full[s]);
        n_issued = t + 1;
        // the rows' statistic (16 bytes per row) into their ring slot, once
        // the MMA that read the slot before has completed
        const int sb = t % kStatSlots;
        if (t >= kStatSlots && !wait_or_abort(&stats_empty[sb], ((t / kStatSlots) - 1) & 1, abort)) break;
        const uint8_t* src =
            static_cast<const uint8_t*>(p.aug) + ((((int64_t)ri * p.B + b) * p.Hq + hq) * p.stats_ld + it) * 16;
        mbar_arrive_expect_tx(&stats_full[sb], 2048);
        bulk_g2s(smem + S::AUG_OFF + sb * 2048, src, 2048, &stats_full[sb]);
        n_stats = t + 1;
      }
      n_issued = t + 1;
    }
    // leave no copy in flight: wait (bounded) for the last copies issued
    for (int t = n_issued > kStagesTc ? n_issued - kStagesTc : 0; t < n_issued; ++t) {
      int never = 0;
      wait_or_abort(&full[t % kStagesTc], (t / kStagesTc) & 1, &never);
    }
    for (int t = n_stats > kStatSlots ? n_stats - kStatSlots : 0; t < n_stats; ++t) {
      int never = 0;
      wait_or_abort(&stats_full[t % kStatSlots], (t / kStatSlots) & 1, &never);
    }
  } else if (warp == 1 && lane == 0 && n_tiles > 0) {
    // ---------------------------------------------------- MMA issuer
    int n_mma = 0;
    if (wait_or_abort(a_full, 0, abort)) {
      const uint32_t a_base = smem_u32(smem + S::A_OFF);
      for (int t = 0; t < n_tiles; ++t) {
        const int s = t % kStagesTc, buf = t & 1;
        if (!wait_or_abort(&full[s], (t / kStagesTc) & 1, abort)) break;
        if (t >= 2 && !wait_or_abort(&acc_empty[buf], ((t >> 1) - 1) & 1, abort)) break;
        if (PASS == 1 && !wait_or_abort(&stats_full[t % kStatSlots], (t / kStatSlots) & 1, abort)) break;
        tc_fence_after();
        const uint32_t b_base = smem_u32(smem + S::B_OFF + s * S::STAGE);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kBoxBytes + (kk & 3) * 32;
          umma_bf16(tmem + buf * 128, sw128_desc(a_base + off), sw128_desc(b_base + off), kIdesc, kk > 0);
        }
        if (PASS == 1) {
          // one more K step adds the rows' statistic: S^T + (x1 + x2 + x3)
          const int sb = t % kStatSlots;
          umma_bf16(tmem + buf * 128, plain_desc(smem_u32(smem + S::ONE_OFF), 128, 0),
                    plain_desc(smem_u32(smem + S::AUG_OFF + sb * 2048), 0, 128), kIdesc, 1);
          umma_commit(&stats_empty[sb]);
        }
        umma_commit(&empty[s]);
        umma_commit(&acc_full[buf]);
        n_mma = t + 1;
      }
    }
    // leave no MMA in flight before TMEM is released (bounded)
    if (n_mma > 0) {
      int never = 0;
      wait_or_abort(&acc_full[(n_mma - 1) & 1], ((n_mma - 1) >> 1) & 1, &never);
    }
  } else if (warp >= 2) {
    // ---------------------------------------------------- epilogue
    const int quarter = warp & 3;               // TMEM lanes 32*quarter ..
    const int half = (warp - 2) >> 2;           // columns 64*half .. +63
    const int col0 = half * 64;
    const int r = quarter * 32 + lane;          // this thread's TMEM lane
    const uint32_t lane_addr = tmem + ((uint32_t)(quarter * 32) << 16) + col0;
    const uint64_t sc2 = pk2(p.scale_log2, p.scale_log2);
    float m = kNegInf, l = 0.f, acc = 0.f;
    const int i_row = i0 + r;                   // pass 0: window row
    const int pos_row = base + i_row;
    const int j_key = j0 + r;                   // pass 1: key
    int t = 0;
    for (; t < n_tiles; ++t) {
      const int buf = t & 1;
      const bool ok = wait_or_abort(&acc_full[buf], (t >> 1) & 1, abort);
      // each epilogue warp goes on alone (its lanes agree); a warp that gave
      // up leaves the abort flag set, so the others stop at their next wait
      // and every warp still meets the exchange barrier after the loop (a
      // barrier of all epilogue warps per tile cost 3% of the pass)
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      if (PASS == 0) {
        const int kj = t * 128 + col0;                  // first key of this thread's columns
        const bool need_mask = kj + 63 > base + i0;     // crosses some row's diagonal
#pragma unroll 1
        for (int c = 0; c < 2; ++c) {
          float v[32];
          tmem_ld32(lane_addr + buf * 128 + c * 32, v);
          if (need_mask) {
#pragma unroll
            for (int k = 0; k < 32; ++k)
              if (kj + c * 32 + k > pos_row) v[k] = kNegInf;
          }
          const float mnew = fmaxf(m, max32(v) * p.scale_log2);
          if (mnew != kNegInf) {
            const uint64_t nm2 = pk2(-mnew, -mnew);
            uint64_t s2 = pk2(0.f, 0.f);
#pragma unroll
            for (int k = 0; k < 32; k += 2) {
              const uint64_t x2 = ffma2(pk2(v[k], v[k + 1]), sc2, nm2);
              s2 = fadd2(s2, exp2_mufu2(x2));
            }
            float s0, s1;
            upk2(s2, s0, s1);
            const float sum = s0 + s1;
            l = (m == kNegInf) ? sum : l * fast_exp2(m - mnew) + sum;
            m = mnew;
          }
        }
      } else {
        const int it = i_start + (t % tiles_per_g) * 128 + col0;  // first row of this thread's columns
        // the accumulator already holds s + statistic / scale_log2 (about
        // -3e38 past the window); row i sees key j when j <= base + i
        const bool need_mask = j0 + 127 > base + it;
        const uint64_t zero2 = pk2(0.f, 0.f);
        uint64_t s2 = pk2(0.f, 0.f);
#pragma unroll 1
        for (int c = 0; c < 2; ++c) {
          float v[32];
          tmem_ld32(lane_addr + buf * 128 + c * 32, v);
          if (need_mask) {
#pragma unroll
            for (int k = 0; k < 32; ++k)
              if (j_key > base + it + c * 32 + k) v[k] = kNegInf;
          }
#pragma unroll
          for (int k = 0; k < 32; k += 2) s2 = fadd2(s2, exp2_mufu2(ffma2(pk2(v[k], v[k + 1]), sc2, zero2)));
        }
        float s0, s1;
        upk2(s2, s0, s1);
        acc += s0 + s1;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[buf]);
    }
    // combine the two column halves of every lane (fixed order: half 0 + half 1)
    float2* xch = reinterpret_cast<float2*>(smem + S::XCH_OFF);
    if (half == 1) xch[r] = PASS == 0 ? make_float2(m, l) : make_float2(acc, 0.f);
    epilogue_sync();
    if (half == 0 && !*abort && t == n_tiles && n_tiles > 0) {
      const float2 o = xch[r];
      if (PASS == 0) {
        const float M = fmaxf(m, o.x);
        const float L = (m == kNegInf ? 0.f : l * fast_exp2(m - M)) + (o.x == kNegInf ? 0.f : o.y * fast_exp2(o.x - M));
        // the statistic over the log2 scale, split into three bf16 parts
        // (x1 + x2 + x3 = x to fp32 precision), so pass 1's extra MMA step
        // adds it to every score of the row.  Rows past the window get a
        // large finite negative value (ex2 of it is 0): -inf would meet the
        // zero channels of the step's other operand and give 0 x inf = NaN
        uint4* ar = reinterpret_cast<uint4*>(p.aug) + (((int64_t)ri * p.B + b) * p.Hq + head) * p.stats_ld + i_row;
        if (i_row < w) {
          const float x = -(M + log2f(L)) / p.scale_log2;
          const bf16 x1 = __float2bfloat16_rn(x);
          const float r1 = x - __bfloat162float(x1);
          const bf16 x2 = __float2bfloat16_rn(r1);
          const bf16 x3 = __float2bfloat16_rn(r1 - __bfloat162float(x2));
          *ar = make_uint4(pack_bf16_pair(x1, x2), pack_bf16_pair(x3, __float2bfloat16_rn(0.f)), 0u, 0u);
        } else if (i_row < (w + 127) / 128 * 128) {
          *ar = make_uint4(pack_bf16_pair(__float2bfloat16_rn(-3.0e38f), __float2bfloat16_rn(0.f)), 0u, 0u, 0u);
        }
      } else if (j_key < T_b) {
        p.scores[((int64_t)(group * p.B + b) * p.Hkv + head) * p.t_max + j_key] = acc + o.x;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
}

// Several consecutive items per CTA, for items of few tiles (short prompts,
// one query head per group), where the one-item kernel spends much of a
// CTA's life on setup and on filling and draining its pipeline.
template <int PASS, int D>
__global__ void __launch_bounds__(kTcThreads, 2) score_tc_items_kernel(const __grid_constant__ ScoreTcParams p) {
  using S = TcSmem<D>;
  constexpr int KH = S::KH;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::BAR_OFF);
  uint64_t* empty = full + kStagesTc;
  uint64_t* a_full = empty + kStagesTc;
  uint64_t* a_empty = a_full + 1;
  uint64_t* acc_full = a_empty + 1;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* stats_full = acc_empty + 2;
  uint64_t* stats_empty = stats_full + kStatSlots;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(stats_empty + kStatSlots);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // ---- work items: (unit, block) pairs.  CTA c takes the contiguous items
  // [c * per_cta, (c + 1) * per_cta) (consecutive blocks of one unit share
  // their other operand through L2); every role walks them in the same
  // order and skips the items with nothing to compute.  The stage ring, the two accumulators and the statistics ring
  // run on tile counters that continue across items, so TMEM and the
  // barriers are set up once per CTA.
  const int HEADS = PASS == 0 ? p.Hq : p.Hkv;
  const int n_blk = PASS == 0 ? (p.win_rows + 127) / 128 : (p.t_max + 127) / 128;
  const int64_t n_items = (int64_t)n_blk * p.n_refs * p.B * HEADS;
  const int64_t x_begin = (int64_t)blockIdx.x * p.items_per_cta;
  const int64_t x_end = min(n_items, x_begin + p.items_per_cta);
  struct Item {
    int head, b, ri, layer, group, T_b, w, qoff, base, i0, j0, i_start, tiles_per_g, n_tiles;
  };
  auto item_at = [&](int64_t x) {
    Item it;
    const int unit = (int)(x / n_blk), blk = (int)(x % n_blk);
    it.head = unit % HEADS;
    it.b = (unit / HEADS) % p.B;
    it.ri = unit / (HEADS * p.B);
    it.layer = p.refs.layer[it.ri];
    it.group = p.refs.group[it.ri];
    it.T_b = p.lens[it.b];
    const bool valid_len = it.T_b >= 1 && it.T_b <= p.t_max;
    it.w = valid_len ? win_rows_of(p, it.T_b) : 0;
    it.qoff = p.win_rows - it.w;
    it.base = it.T_b - it.w;  // position of window row 0
    it.n_tiles = it.i0 = it.j0 = it.i_start = it.tiles_per_g = 0;
    if (valid_len && it.w <= p.win_rows) {
      if (PASS == 0) {
        it.i0 = blk * 128;  // window rows of this item
        if (it.i0 < it.w) {
          const int pos_last = it.base + min(it.i0 + 127, it.w - 1);
          it.n_tiles = pos_last / 128 + 1;  // key tiles 0 .. pos_last
        }
      } else {
        it.j0 = blk * 128;  // keys of this item
        if (it.j0 < it.T_b) {
          const int i_first = max(0, it.j0 - it.base);  // first row that sees key j0
          it.i_start = (i_first / 128) * 128;
          it.tiles_per_g = (it.w - it.i_start + 127) / 128;
          it.n_tiles = p.G * it.tiles_per_g;
        }
      }
    }
    return it;
  };
  // the first item is worked out once, before the setup, and reused by
  // every role; a CTA whose items are all empty (past its sequences'
  // windows or keys) leaves before the barriers and the TMEM allocation
  const Item first = item_at(x_begin);
  {
    bool any = first.n_tiles > 0;
    for (int64_t x = x_begin + 1; x < x_end && !any; ++x) any = item_at(x).n_tiles > 0;
    if (!any) return;
  }
  auto item_of = [&](int64_t x) { return x == x_begin ? first : item_at(x); };

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStagesTc; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(a_full, 1);
    mbar_init(a_empty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kTcEpiWarps);
    }
    for (int i = 0; i < kStatSlots; ++i) {
      mbar_init(&stats_full[i], 1);
      mbar_init(&stats_empty[i], 1);  // released by the MMA that read the slot
    }
    *abort = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 256);
    tmem_relinquish();
  }
  if (PASS == 1 && threadIdx.x >= 64 && threadIdx.x < 80) {
    // K-side operand of the statistic step: one 8-row core matrix whose rows
    // are (1, 1, 1, 0, 0, 0, 0, 0) (every 8-row group reuses it), then a zero
    // core matrix for channels 8..15
    const int i = threadIdx.x - 64;
    reinterpret_cast<uint4*>(smem + S::ONE_OFF)[i] =
        i < 8 ? make_uint4(0x3F803F80u, 0x00003F80u, 0u, 0u) : make_uint4(0u, 0u, 0u, 0u);
    fence_proxy_async_smem();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0 && lane == 0) {
    // ---------------------------------------------------- TMA producer
    int64_t gt = 0;  // B tiles issued (all items)
    int n_a = 0;     // A tiles issued
    for (int64_t x = x_begin; x < x_end && !*abort; ++x) {
      const Item it = item_of(x);
      if (it.n_tiles == 0) continue;
      const int qrow0 = (it.b * p.Hq) * p.win_rows + it.qoff;  // + hq * win_rows + i
      const int krow0 = (it.b * p.Hkv) * p.t_max;              // + hk * t_max + j
      const int kcoord = p.k_by_ref ? it.ri : it.layer;
      // A: once the previous item's MMAs have read it
      if (n_a > 0 && !wait_or_abort(a_empty, (n_a - 1) & 1, abort)) break;
      mbar_arrive_expect_tx(a_full, S::TILE);
      for (int kh = 0; kh < KH; ++kh) {
        if (PASS == 0)
          tma_load_3d(smem + S::A_OFF + kh * kBoxBytes, &p.map_q, kh * 64, qrow0 + it.head * p.win_rows + it.i0,
                      it.layer, a_full);
        else  // keys [j0, j0 + 128) of this kv head: one 128-row box per 64-channel half
          tma_load_3d(smem + S::A_OFF + kh * kBoxBytes, &p.map_k, kh * 64, krow0 + it.head * p.t_max + it.j0,
                      kcoord, a_full);
      }
      ++n_a;
      for (int t = 0; t < it.n_tiles; ++t, ++gt) {
        const int s = (int)(gt % kStagesTc);
        if (gt >= kStagesTc && !wait_or_abort(&empty[s], (int)((gt / kStagesTc) - 1) & 1, abort)) break;
        uint8_t* st = smem + S::B_OFF + s * S::STAGE;
        mbar_arrive_expect_tx(&full[s], S::TILE);
        if (PASS == 0) {
          for (int kh = 0; kh < KH; ++kh)
            tma_load_3d(st + kh * kBoxBytes, &p.map_k, kh * 64, krow0 + (it.head / p.G) * p.t_max + t * 128, kcoord,
                        &full[s]);
        } else {
          const int g = t / it.tiles_per_g, ir = it.i_start + (t % it.tiles_per_g) * 128;
          const int hq = it.head * p.G + g;
          for (int kh = 0; kh < KH; ++kh)
            tma_load_3d(st + kh * kBoxBytes, &p.map_q, kh * 64, qrow0 + hq * p.win_rows + ir, it.layer, &full[s]);
          // the rows' statistic (16 bytes per row) into its ring slot, once
          // the MMA that read the slot before has completed
          const int sb = (int)(gt % kStatSlots);
          if (gt >= kStatSlots && !wait_or_abort(&stats_empty[sb], (int)((gt / kStatSlots) - 1) & 1, abort)) {
            ++gt;
            break;
          }
          const uint8_t* src = static_cast<const uint8_t*>(p.aug) +
                               ((((int64_t)it.ri * p.B + it.b) * p.Hq + hq) * p.stats_ld + ir) * 16;
          mbar_arrive_expect_tx(&stats_full[sb], 2048);
          bulk_g2s(smem + S::AUG_OFF + sb * 2048, src, 2048, &stats_full[sb]);
        }
      }
    }
    // leave no copy in flight: wait (bounded) for the last copies issued
    for (int64_t t = gt > kStagesTc ? gt - kStagesTc : 0; t < gt; ++t) {
      int never = 0;
      wait_or_abort(&full[t % kStagesTc], (int)(t / kStagesTc) & 1, &never);
    }
    if (PASS == 1)
      for (int64_t t = gt > kStatSlots ? gt - kStatSlots : 0; t < gt; ++t) {
        int never = 0;
        wait_or_abort(&stats_full[t % kStatSlots], (int)(t / kStatSlots) & 1, &never);
      }
    if (n_a > 0) {
      int never = 0;
      wait_or_abort(a_full, (n_a - 1) & 1, &never);
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------------------------------------------- MMA issuer
    int64_t gt = 0;  // B tiles consumed (all items)
    int n_a = 0;
    bool any = false;
    for (int64_t x = x_begin; x < x_end && !*abort; ++x) {
      const Item it = item_of(x);
      if (it.n_tiles == 0) continue;
      if (!wait_or_abort(a_full, n_a & 1, abort)) break;
      ++n_a;
      const uint32_t a_base = smem_u32(smem + S::A_OFF);
      bool ok = true;
      for (int t = 0; t < it.n_tiles; ++t, ++gt) {
        const int s = (int)(gt % kStagesTc), buf = (int)(gt & 1);
        if (!wait_or_abort(&full[s], (int)(gt / kStagesTc) & 1, abort) ||
            (gt >= 2 && !wait_or_abort(&acc_empty[buf], (int)((gt >> 1) - 1) & 1, abort)) ||
            (PASS == 1 && !wait_or_abort(&stats_full[gt % kStatSlots], (int)(gt / kStatSlots) & 1, abort))) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t b_base = smem_u32(smem + S::B_OFF + s * S::STAGE);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kBoxBytes + (kk & 3) * 32;
          umma_bf16(tmem + buf * 128, sw128_desc(a_base + off), sw128_desc(b_base + off), kIdesc, kk > 0);
        }
        if (PASS == 1) {
          // one more K step adds the rows' statistic: S^T + (x1 + x2 + x3)
          const int sb = (int)(gt % kStatSlots);
          umma_bf16(tmem + buf * 128, plain_desc(smem_u32(smem + S::ONE_OFF), 128, 0),
                    plain_desc(smem_u32(smem + S::AUG_OFF + sb * 2048), 0, 128), kIdesc, 1);
          umma_commit(&stats_empty[sb]);
        }
        umma_commit(&empty[s]);
        umma_commit(&acc_full[buf]);
        any = true;
      }
      umma_commit(a_empty);  // A is free once this item's MMAs are done
      if (!ok) break;
    }
    // leave no MMA in flight before TMEM is released (bounded)
    if (any) {
      int never = 0;
      wait_or_abort(&acc_full[(gt - 1) & 1], (int)((gt - 1) >> 1) & 1, &never);
    }
  } else if (warp >= 2) {
    // ---------------------------------------------------- epilogue
    const int quarter = warp & 3;               // TMEM lanes 32*quarter ..
    const int half = (warp - 2) >> 2;           // columns 64*half .. +63
    const int col0 = half * 64;
    const int r = quarter * 32 + lane;          // this thread's TMEM lane
    const uint32_t lane_addr = tmem + ((uint32_t)(quarter * 32) << 16) + col0;
    const uint64_t sc2 = pk2(p.scale_log2, p.scale_log2);
    int64_t gt = 0;
    int n_done = 0;
    for (int64_t x = x_begin; x < x_end; ++x) {
      const Item it = item_of(x);
      if (it.n_tiles == 0) continue;
      float m = kNegInf, l = 0.f, acc = 0.f;
      const int i_row = it.i0 + r;                // pass 0: window row
      const int pos_row = it.base + i_row;
      const int j_key = it.j0 + r;                // pass 1: key
      int t = 0;
      for (; t < it.n_tiles; ++t, ++gt) {
        const int buf = (int)(gt & 1);
        const bool ok = wait_or_abort(&acc_full[buf], (int)(gt >> 1) & 1, abort);
        if (!__all_sync(0xffffffffu, ok)) break;  // per warp, as in score_tc_kernel
        tc_fence_after();
        if (PASS == 0) {
          const int kj = t * 128 + col0;                     // first key of this thread's columns
          const bool need_mask = kj + 63 > it.base + it.i0;  // crosses some row's diagonal
#pragma unroll 1
          for (int c = 0; c < 2; ++c) {
            float v[32];
            tmem_ld32(lane_addr + buf * 128 + c * 32, v);
            if (need_mask) {
#pragma unroll
              for (int k = 0; k < 32; ++k)
                if (kj + c * 32 + k > pos_row) v[k] = kNegInf;
            }
            const float mnew = fmaxf(m, max32(v) * p.scale_log2);
            if (mnew != kNegInf) {
              const uint64_t nm2 = pk2(-mnew, -mnew);
              uint64_t s2 = pk2(0.f, 0.f);
#pragma unroll
              for (int k = 0; k < 32; k += 2) {
                const uint64_t x2 = ffma2(pk2(v[k], v[k + 1]), sc2, nm2);
                s2 = fadd2(s2, exp2_mufu2(x2));
              }
              float s0, s1;
              upk2(s2, s0, s1);
              const float sum = s0 + s1;
              l = (m == kNegInf) ? sum : l * fast_exp2(m - mnew) + sum;
              m = mnew;
            }
          }
        } else {
          const int ir = it.i_start + (t % it.tiles_per_g) * 128 + col0;  // first row of this thread's columns
          // the accumulator already holds s + statistic / scale_log2 (about
          // -3e38 past the window); row i sees key j when j <= base + i
          const bool need_mask = it.j0 + 127 > it.base + ir;
          const uint64_t zero2 = pk2(0.f, 0.f);
          uint64_t s2 = pk2(0.f, 0.f);
#pragma unroll 1
          for (int c = 0; c < 2; ++c) {
            float v[32];
            tmem_ld32(lane_addr + buf * 128 + c * 32, v);
            if (need_mask) {
#pragma unroll
              for (int k = 0; k < 32; ++k)
                if (j_key > it.base + ir + c * 32 + k) v[k] = kNegInf;
            }
#pragma unroll
            for (int k = 0; k < 32; k += 2) s2 = fadd2(s2, exp2_mufu2(ffma2(pk2(v[k], v[k + 1]), sc2, zero2)));
          }
          float s0, s1;
          upk2(s2, s0, s1);
          acc += s0 + s1;
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[buf]);
      }
      if (t < it.n_tiles) break;  // aborted (every epilogue warp takes this branch)
      // combine the two column halves of every lane (fixed order: half 0 +
      // half 1), through a buffer that alternates between items
      float2* xch = reinterpret_cast<float2*>(smem + S::XCH_OFF) + (n_done & 1) * 128;
      if (half == 1) xch[r] = PASS == 0 ? make_float2(m, l) : make_float2(acc, 0.f);
      epilogue_sync();
      if (half == 0 && !*abort) {
        const float2 o = xch[r];
        if (PASS == 0) {
          const float M = fmaxf(m, o.x);
          const float L =
              (m == kNegInf ? 0.f : l * fast_exp2(m - M)) + (o.x == kNegInf ? 0.f : o.y * fast_exp2(o.x - M));
          // the statistic over the log2 scale, split into three bf16 parts
          // (x1 + x2 + x3 = x to fp32 precision), so pass 1's extra MMA step
          // adds it to every score of the row.  Rows past the window get a
          // large finite negative value (ex2 of it is 0): -inf would meet
          // the zero channels of the step's other operand and give
          // 0 x inf = NaN
          uint4* ar = reinterpret_cast<uint4*>(p.aug) +
                      (((int64_t)it.ri * p.B + it.b) * p.Hq + it.head) * p.stats_ld + i_row;
          if (i_row < it.w) {
            const float xv = -(M + log2f(L)) / p.scale_log2;
            const bf16 x1 = __float2bfloat16_rn(xv);
            const float r1 = xv - __bfloat162float(x1);
            const bf16 x2 = __float2bfloat16_rn(r1);
            const bf16 x3 = __float2bfloat16_rn(r1 - __bfloat162float(x2));
            *ar = make_uint4(pack_bf16_pair(x1, x2), pack_bf16_pair(x3, __float2bfloat16_rn(0.f)), 0u, 0u);
          } else if (i_row < (it.w + 127) / 128 * 128) {
            *ar = make_uint4(pack_bf16_pair(__float2bfloat16_rn(-3.0e38f), __float2bfloat16_rn(0.f)), 0u, 0u, 0u);
          }
        } else if (j_key < it.T_b) {
          p.scores[((int64_t)(it.group * p.B + it.b) * p.Hkv + it.head) * p.t_max + j_key] = acc + o.x;
        }
      }
      ++n_done;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
}

// ------------------------------------------------------------- host side ----

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static std::mutex mu;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::lock_guard<std::mutex> lk(mu);
  if (fn == nullptr) {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  }
  return fn;
}

// 3-D map over [layers][rows][d] bf16 with 128-row x 64-channel boxes.
bool make_map(CUtensorMap* map, const void* base, int d, int64_t rows, int layers, int64_t layer_stride_elems) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)rows, (cuuint64_t)layers};
  const cuuint64_t strides[2] = {(cuuint64_t)d * 2, (cuuint64_t)layer_stride_elems * 2};
  const cuuint32_t box[3] = {64, 128, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int PASS, int D>
cudaError_t launch_pass(const ScoreTcParams& p, dim3 grid, cudaStream_t st) {
  const int smem = TcSmem<D>::TOTAL;
  if (p.items_per_cta > 1) {
    cudaError_t e = ensure_dyn_smem((const void*)score_tc_items_kernel<PASS, D>, smem);
    if (e != cudaSuccess) return e;
    score_tc_items_kernel<PASS, D><<<grid, kTcThreads, smem, st>>>(p);
    return cudaGetLastError();
  }
  cudaError_t e = ensure_dyn_smem((const void*)score_tc_kernel<PASS, D>, smem);
  if (e != cudaSuccess) return e;
  score_tc_kernel<PASS, D><<<grid, kTcThreads, smem, st>>>(p);
  return cudaGetLastError();
}

// Items per CTA of a pass: one while an item has kTilesPerCta tiles or more
// (the one-item kernel, one CTA per item on a 2-D grid), else enough items
// for about that many tiles (the items kernel, 1-D grid).  `tiles` is the
// most tiles one item of the pass can have.
int items_per_cta(int tiles) { return std::max(1, kTilesPerCta / std::max(1, tiles)); }

}  // namespace

cudaError_t launch_score_tc(ScoreTcParams& p, int D, int n_layer_span, cudaStream_t st) {
  if (!make_map(&p.map_q, p.q_win, D, (int64_t)p.B * p.Hq * p.win_rows, n_layer_span, p.qw_ls))
    return cudaErrorInvalidValue;
  if (!make_map(&p.map_k, p.k, D, (int64_t)p.B * p.Hkv * p.t_max, p.k_by_ref ? p.n_refs : n_layer_span, p.k_ls))
    return cudaErrorInvalidValue;
  const int row_blks = (p.win_rows + 127) / 128, key_blks = (p.t_max + 127) / 128;
  ScoreTcParams p0 = p, p1 = p;
  p0.items_per_cta = items_per_cta(key_blks);        // pass 0 item: key tiles up to t_max
  p1.items_per_cta = items_per_cta(p.G * row_blks);  // pass 1 item: row tiles of the group's heads
  auto grid_of = [](const ScoreTcParams& q, int blks, int heads) {
    const long long units = (long long)q.n_refs * q.B * heads;
    if (q.items_per_cta == 1) return dim3(blks, (unsigned)units);
    return dim3((unsigned)((units * blks + q.items_per_cta - 1) / q.items_per_cta));
  };
  const dim3 g0 = grid_of(p0, row_blks, p.Hq), g1 = grid_of(p1, key_blks, p.Hkv);
  cudaError_t e;
  if (D == 64) {
    if ((e = launch_pass<0, 64>(p0, g0, st)) != cudaSuccess) return e;
    return launch_pass<1, 64>(p1, g1, st);
  }
  if ((e = launch_pass<0, 128>(p0, g0, st)) != cudaSuccess) return e;
  return launch_pass<1, 128>(p1, g1, st);
}

int take_status_score_tc() { return take_status(); }

}  // namespace mpc
