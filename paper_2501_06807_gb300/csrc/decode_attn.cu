// Sparse decode attention over the selected clusters and the tail, with the
// decode-step append and the tail seal (Alg. 1; Alg. 2 Step 2; App. A).
// One unit = (ref, sequence b, kv head h); the rows a unit attends are the s
// rows of every selected cluster, then the tail rows already in the cache,
// then the row appended now, cut into 16-row tiles.
//
// bf16 caches: attn_bf16_persist_kernel, one persistent CTA per SM whose
// warps stream equal contiguous ranges of the list of all units' tiles
// (below, "bf16 path").
//
// fp32 caches: attn_f32_kernel, one CTA per (chunk of `tiles_per_split`
// tiles, unit).  Each of the CTA's four warps streams its tiles (key rows and
// value rows) from HBM into its own shared-memory ring with 1-D bulk copies
// (TMA engine, completion on an mbarrier), then computes the tile's scores
// for all query heads of the GQA group at once and updates an online
// softmax.  The four warps' partial results are merged in shared memory;
// with several chunks per unit the CTA writes (max, sum, o) to the workspace
// and the last CTA of the unit (atomic ticket, no waiting) merges them by
// log-sum-exp and writes o.
#include <mutex>

#include "kernels.cuh"
#include "seal.cuh"

namespace mpc {


constexpr int kWarps = 4;
constexpr int kStages = 2;


// Unit geometry shared by both dtype paths.
struct Unit {
  int layer, group, b, h, leader;
  int n, C1, tail, k1, n_sel_rows, n_att, n_tiles, t_begin, t_end;
  const int* sel;
};

__device__ __forceinline__ Unit make_unit_at(const AttnParams& p, int ri, int b, int h) {
  Unit u;
  u.h = h;
  u.b = b;
  u.layer = p.refs.layer[ri];
  u.group = p.refs.group[ri];
  u.leader = p.refs.leader[ri];
  const int s = p.pyr.s;
  u.n = p.n_tok[b];
  u.C1 = u.n / s;
  u.tail = u.n - u.C1 * s;
  u.k1 = p.sel_cap > 0 ? min(p.n_sel[b], min(u.C1, p.sel_cap)) : 0;
  u.n_sel_rows = u.k1 * s;
  u.n_att = u.n_sel_rows + u.tail + 1;
  u.n_tiles = (u.n_att + 15) / 16;
  u.t_begin = 0;
  u.t_end = u.n_tiles;
  u.sel = p.sel + ((int64_t)(u.group * p.B + b) * p.Hkv + h) * p.sel_cap;
  return u;
}

// Unit of a split-grid CTA: blockIdx.y = unit, blockIdx.x = chunk of tiles.
__device__ __forceinline__ Unit make_unit(const AttnParams& p) {
  const int unit = blockIdx.y;
  Unit u = make_unit_at(p, unit / (p.Hkv * p.B), (unit / p.Hkv) % p.B, unit % p.Hkv);
  u.t_begin = blockIdx.x * p.tiles_per_split;
  u.t_end = min(u.n_tiles, u.t_begin + p.tiles_per_split);
  return u;
}

// Cache row of attended index a (a < n_att - 1).  A selected id outside
// [0, C_1) (corrupt input) is reported and read as cluster 0.
__device__ __forceinline__ int src_row(const Unit& u, int s, int a) {
  if (a < u.n_sel_rows) {
    const int c = a / s;
    int id = u.sel[c];
    if (id < 0 || id >= u.C1) {
      atomicOr(&g_mpc_status, 4);
      id = 0;
    }
    return id * s + (a - c * s);
  }
  return u.C1 * s + (a - u.n_sel_rows);
}

// Issues the bulk copies of tile t into stage buffers (sK, sV); runs of
// consecutive cache rows are copied with one instruction each.  Records the
// swizzle key (cache row & 7) of every tile row.
template <int ROWB>
__device__ __forceinline__ void issue_tile(const Unit& u, int s, int t, const uint8_t* kbase,
                                           const uint8_t* vbase, uint8_t* sK, uint8_t* sV,
                                           int8_t* keys, uint64_t* bar, int lane,
                                           const void* q_src = nullptr, void* q_dst = nullptr,
                                           uint32_t q_bytes = 0) {
  const int r = lane & 15;
  const int a = t * 16 + r;
  const bool valid = a < u.n_att;
  const bool cur = a == u.n_att - 1;
  const bool from_cache = valid && !cur;
  const int src = from_cache ? src_row(u, s, a) : (cur ? u.n : 0);
  const int prev_src = __shfl_up_sync(0xffffffffu, src, 1);
  const int prev_fc = __shfl_up_sync(0xffffffffu, (int)from_cache, 1);
  const bool start = from_cache && (r == 0 || !prev_fc || src != prev_src + 1);
  if (lane < 16) keys[r] = (int8_t)(valid ? (src & 7) : (r & 7));
  const uint32_t mstart = __ballot_sync(0xffffffffu, start) & 0xffffu;
  const uint32_t mcache = __ballot_sync(0xffffffffu, from_cache) & 0xffffu;
  const int ncache = __popc(mcache);  // cache rows form a prefix of the tile
  if (lane == 0) mbar_arrive_expect_tx(bar, (uint32_t)(ncache * ROWB * 2) + (q_src ? q_bytes : 0u));
  __syncwarp();
  if (q_src != nullptr && lane == 16) bulk_g2s(q_dst, q_src, q_bytes, bar);
  if (lane < 16 && start) {
    const uint32_t later = mstart & ~((2u << r) - 1u);
    int end = later ? (__ffs(later) - 1) : ncache;
    end = min(end, ncache);
    const uint32_t bytes = (uint32_t)((end - r) * ROWB);
    bulk_g2s(sK + r * ROWB, kbase + (int64_t)src * ROWB, bytes, bar);
    bulk_g2s(sV + r * ROWB, vbase + (int64_t)src * ROWB, bytes, bar);
  }
}

// Shared-memory carve-up common to both kernels.
template <int D, int ESZ>
struct Smem {
  static constexpr int ROWB = D * ESZ;
  static constexpr int TILEB = 16 * ROWB;
  static constexpr int STAGE_BYTES = 2 * TILEB;
  static constexpr int RING = kWarps * kStages * STAGE_BYTES;
  static constexpr int BAR_OFF = RING;
  static constexpr int KEY_OFF = BAR_OFF + kWarps * kStages * 8;
  static constexpr int MERGE_OFF = KEY_OFF + kWarps * kStages * 16;
  static __host__ __device__ constexpr int merge_bytes(int G) { return kWarps * G * (D + 4) * 4; }
  static __host__ __device__ constexpr int total(int G) { return MERGE_OFF + merge_bytes(G) + G * D * 4; }
};

// Merges the warps' partials, then the splits', and writes o.  `mw` holds per
// warp and head: [0] = max (log2 units), [1] = sum, [4 ..] = o (unnormalised).
template <int D>
__device__ void merge_and_store(const AttnParams& p, const Unit& u, float* mw, int nwarps_used) {
  const int G = p.G;
  const int tid = threadIdx.x;
  __syncthreads();
  const int unit = blockIdx.y;
  float* outp = p.out + u.layer * p.out_ls + ((int64_t)u.b * p.Hq + u.h * G) * D;
  __shared__ float s_scale[kWarps][16];
  __shared__ float s_ml[16][2];
  if (tid < G) {
    float M = kNegInf;
    for (int w = 0; w < nwarps_used; ++w) M = fmaxf(M, mw[(w * G + tid) * (D + 4)]);
    float L = 0.f;
    for (int w = 0; w < nwarps_used; ++w) {
      const float mwv = mw[(w * G + tid) * (D + 4)];
      const float f = (mwv == kNegInf) ? 0.f : fast_exp2(mwv - M);
      s_scale[w][tid] = f;
      L += f * mw[(w * G + tid) * (D + 4) + 1];
    }
    s_ml[tid][0] = M;
    s_ml[tid][1] = L;
  }
  __syncthreads();
  if (p.n_split == 1) {
    for (int i = tid; i < G * D; i += blockDim.x) {
      const int g = i / D, c = i % D;
      float o = 0.f;
      for (int w = 0; w < nwarps_used; ++w) o += s_scale[w][g] * mw[(w * G + g) * (D + 4) + 4 + c];
      outp[g * D + c] = o / s_ml[g][1];
    }
    return;
  }
  float* mine = p.part + ((int64_t)unit * p.n_split + blockIdx.x) * G * (D + 4);
  for (int i = tid; i < G * (D + 4); i += blockDim.x) {
    const int g = i / (D + 4), c = i % (D + 4);
    float v;
    if (c == 0) v = s_ml[g][0];
    else if (c == 1) v = s_ml[g][1];
    else if (c < 4) v = 0.f;
    else {
      v = 0.f;
      for (int w = 0; w < nwarps_used; ++w) v += s_scale[w][g] * mw[(w * G + g) * (D + 4) + c];
    }
    mine[i] = v;
  }
  __threadfence();
  __syncthreads();
  __shared__ int s_last;
  if (tid == 0) {
    const int ticket = atomicAdd(&p.unit_counter[unit], 1);
    s_last = (ticket == p.n_split - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const float* all = p.part + (int64_t)unit * p.n_split * G * (D + 4);
  __shared__ float s_f[64][16];
  if (tid < G) {
    float M = kNegInf;
    for (int sp = 0; sp < p.n_split; ++sp) M = fmaxf(M, __ldcg(all + (sp * G + tid) * (D + 4)));
    float L = 0.f;
    for (int sp = 0; sp < p.n_split; ++sp) {
      const float m = __ldcg(all + (sp * G + tid) * (D + 4));
      const float f = (m == kNegInf) ? 0.f : fast_exp2(m - M);
      if (sp < 64) s_f[sp][tid] = f;
      L += f * __ldcg(all + (sp * G + tid) * (D + 4) + 1);
    }
    s_ml[tid][1] = L;
  }
  __syncthreads();
  for (int i = tid; i < G * D; i += blockDim.x) {
    const int g = i / D, c = i % D;
    float o = 0.f;
    for (int sp = 0; sp < p.n_split; ++sp) o += s_f[sp][g] * __ldcg(all + (sp * G + g) * (D + 4) + 4 + c);
    outp[g * D + c] = o / s_ml[g][1];
  }
  if (tid == 0) p.unit_counter[unit] = 0;
}

// Seals a full tail as a new finest-level cluster of a leader's pyramid
// (the pyramid update itself is seal_cluster in seal.cuh).
template <typename T, int D>
__device__ void seal_tail(const AttnParams& p, const Unit& u, const T* kcache) {
  if (!(u.leader && u.tail + 1 == p.pyr.s && p.rmax != nullptr)) return;
  seal_cluster<T, D>(p, u.group, u.b, u.h, u.C1, kcache);
}

__device__ __forceinline__ void finish_grid(const AttnParams& p) {
  if (!p.advance) return;
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const int total = gridDim.x * gridDim.y;
    const int ticket = atomicAdd(p.grid_counter, 1);
    if (ticket == total - 1) {
      __threadfence();
      // a sequence whose append was refused (no room left) keeps its count
      for (int b = 0; b < p.B; ++b) {
        const int n = p.n_tok[b];
        if (n >= 0 && n + 1 <= p.cap_tokens) p.n_tok[b] = n + 1;
      }
      *p.grid_counter = 0;
    }
  }
}

// ------------------------------------------------ bf16 path (persistent) ----
//
// One CTA per SM, four to eight warps.  The tiles of all units (every selected
// cluster row tile, tail and appended row of every (layer, sequence, kv
// head)) form one list, cut into contiguous, equal ranges, one per warp slot
// (slots interleaved over the CTAs, at most one slot per tile).  Every warp
// streams its range through its own ring of shared-memory stages (K and V
// tile rows), so every SM moves the same amount of KV.
//
// Tiles are staged with cp.async (16 bytes per lane, committed as one group
// per tile, so a warp keeps NST tiles in flight at the cost of a few
// instructions each).  With s a multiple of 16 every tile is one run of
// consecutive cache rows; other cluster sizes gather the rows one by one.
//
// Per tile the group's heads are the N dimension of the tensor-core products
// (S^T = K Q^T, O^T = V^T P^T with m16n8k16 bf16 mma, P split into bf16 hi +
// lo), so one 8-head n-tile covers a GQA group of up to 8 query heads.  P
// moves from the accumulator layout of S^T to the operand layout of P^T with
// movmatrix (an in-register 8x8 transpose).
//
// A unit finished inside one warp is written directly.  A unit split across
// warps is merged by its owner, the warp holding its first piece: that piece
// ends its warp's range, so it finishes last in time.  Every later piece is
// the first piece of its warp, finished early; it writes a partial (max,
// sum, o) record (one slot per warp) and signals the owner with a release
// reduction on the unit's counter, without waiting.  The owner waits (bounded)
// for the count, then folds the records into its registers by log-sum-exp.
// The grid is launched cooperatively (launch_persist), so every CTA whose
// piece an owner waits for is resident.

constexpr int kMaxPersistCtas = 152;

constexpr int kMaxBatchPersist = 512;
constexpr int kSelSmem = 256;  // selected ids staged per warp (longer lists are read from global)

template <int D>
struct PSmem {
  static constexpr int ROWB = D * 2;
  static constexpr int TILEB = 16 * ROWB;
  static __host__ __device__ constexpr int qbytes(int G) { return ((G * D * 2 + 127) / 128) * 128; }
  static __host__ __device__ constexpr int stage(int G) { return 2 * TILEB + qbytes(G); }
  // wpc warps per CTA, each with an nst-stage ring
  static __host__ __device__ constexpr int key_off(int G, int nst, int wpc) { return wpc * nst * stage(G); }
  static __host__ __device__ constexpr int sel_off(int G, int nst, int wpc) { return key_off(G, nst, wpc) + wpc * nst * 16; }
  static __host__ __device__ constexpr int tab_off(int G, int nst, int wpc) { return sel_off(G, nst, wpc) + wpc * kSelSmem * 4; }
  static __host__ __device__ constexpr int total(int G, int nst, int wpc, int B) { return tab_off(G, nst, wpc) + (4 * B + 2) * 4; }
};

// Warps per CTA and ring depth per warp (compile-time for
// cp.async.wait_group).  More warps hide the per-tile compute better than
// deeper rings at the same bytes in flight (measured: 2 x 12 and 4 x 6 are
// slower than 6 x 4; 8 x 3 is best with one query head per group, whose
// tiles carry the same mma work for a quarter of the heads).  d 64: 4 x 8.
// d 128, up to 8 heads per group: 8 x 3 (one head) or 6 x 4 when that fits
// shared memory with the batch's tables, else 4 x 5; up to 16 heads: 4 x 4.
struct PersistCfg {
  int wpc, nst;
};
inline PersistCfg persist_cfg(int D, int G, int B) {
  if (D == 64) return {4, 8};
  if (G == 1 && PSmem<128>::total(G, 3, 8, B) <= kSmemOptin) return {8, 3};
  if (G <= 8 && PSmem<128>::total(G, 4, 6, B) <= kSmemOptin) return {6, 4};
  return {4, G <= 8 ? 5 : 4};
}

struct Cursor {
  int ri, b, h, lt;
};

// In-register transpose of an 8x8 b16 matrix held in mma fragment layout.
__device__ __forceinline__ uint32_t movmatrix_t(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}

template <int D, int HN, int NST, int WPC>
__global__ void __launch_bounds__(WPC * 32, 1) attn_bf16_persist_kernel(const __grid_constant__ AttnParams p) {
  using S = PSmem<D>;
  constexpr int ROWB = S::ROWB;
  constexpr int TILEB = S::TILEB;
  constexpr int KS = D / 16;  // k-steps of S^T and m-tiles of O^T
  extern __shared__ __align__(128) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = p.G, B = p.B, Hkv = p.Hkv, s = p.pyr.s;
  const int STAGE = S::stage(G);
  constexpr int CH = ROWB / 16;  // 16-byte chunks per row
  uint8_t* ring = smem + warp * NST * STAGE;
  int8_t* keys = reinterpret_cast<int8_t*>(smem + S::key_off(G, NST, WPC)) + warp * NST * 16;
  int* sel_s = reinterpret_cast<int*>(smem + S::sel_off(G, NST, WPC)) + warp * kSelSmem;
  int* s_nt = reinterpret_cast<int*>(smem + S::tab_off(G, NST, WPC));  // tiles per unit of sequence b
  int* s_pre = s_nt + B;                                           // exclusive prefix of s_nt (B + 1)
  int* s_n = s_pre + B + 1;                                        // cache rows before the append
  int* s_k1 = s_n + B;                                             // selected clusters
  grid_dep_launch();
  grid_dep_wait();

  // ---- per-sequence table
  if (warp == 0) {
    int carry = 0;
    for (int b0 = 0; b0 < B; b0 += 32) {
      const int b = b0 + lane;
      int nt = 0, n = 0, k1 = 0;
      if (b < B) {
        // both counts are requested at once (one round trip, not two)
        n = p.n_tok[b];
        const int ns = p.sel_cap > 0 ? p.n_sel[b] : 0;
        if (n < 0 || n + 1 > p.cap_tokens) {
          atomicOr(&g_mpc_status, 2);  // no room for the append: skip the sequence
        } else {
          const int C1 = n / s;
          k1 = min(ns, min(C1, p.sel_cap));
          nt = (k1 * s + (n - C1 * s) + 1 + 15) / 16;
        }
      }
      int incl = nt;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      if (b < B) {
        s_nt[b] = nt;
        s_pre[b] = carry + incl - nt;
        s_n[b] = n;
        s_k1[b] = k1;
      }
      carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) s_pre[B] = carry;
  }
  __syncthreads();
  const bool fast = (s & 15) == 0;  // every tile is one run of consecutive rows
  const int s16 = s >> 4;

  const int64_t TPR = (int64_t)Hkv * s_pre[B];
  const int64_t NT = TPR * p.n_refs;
  const int64_t NW_all = (int64_t)gridDim.x * WPC;
  const int NW = (int)(NW_all < NT ? NW_all : NT);
  const int gw = warp * gridDim.x + blockIdx.x;
  const int64_t x0 = gw < NW ? NT * gw / NW : 0, x1 = gw < NW ? NT * (gw + 1) / NW : 0;
  auto warp_of = [&](int64_t x) { return (int)((x * NW + NW - 1) / NT); };
  auto locate = [&](int64_t x) {
    Cursor c;
    c.ri = (int)(x / TPR);
    const int64_t rem = x - c.ri * TPR;
    int lo = 0, hi = B - 1;  // largest b with Hkv * pre[b] <= rem
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if ((int64_t)Hkv * s_pre[mid] <= rem) lo = mid;
      else hi = mid - 1;
    }
    c.b = lo;
    const int64_t rem2 = rem - (int64_t)Hkv * s_pre[lo];
    c.h = (int)(rem2 / s_nt[lo]);
    c.lt = (int)(rem2 % s_nt[lo]);
    return c;
  };
  auto advance = [&](Cursor& c) {
    if (++c.lt < s_nt[c.b]) return;
    c.lt = 0;
    if (++c.h < Hkv) return;
    c.h = 0;
    do {
      if (++c.b == B) {
        c.b = 0;
        ++c.ri;
      }
    } while (s_nt[c.b] == 0);
  };
  auto unit_at = [&](const Cursor& c) {
    Unit u;
    u.h = c.h;
    u.b = c.b;
    u.layer = p.refs.layer[c.ri];
    u.group = p.refs.group[c.ri];
    u.leader = p.refs.leader[c.ri];
    u.n = s_n[c.b];
    u.C1 = u.n / s;
    u.tail = u.n - u.C1 * s;
    u.k1 = s_k1[c.b];
    u.n_sel_rows = u.k1 * s;
    u.n_att = u.n_sel_rows + u.tail + 1;
    u.n_tiles = s_nt[c.b];
    u.t_begin = 0;
    u.t_end = u.n_tiles;
    u.sel = p.sel + ((int64_t)(u.group * B + c.b) * Hkv + c.h) * p.sel_cap;
    return u;
  };
  auto kv_base = [&](const Unit& u, int which) {
    const bf16* base = (const bf16*)(which ? p.vc : p.kc) + u.layer * p.cache_ls +
                       (int64_t)(u.b * Hkv + u.h) * p.cap_tokens * D;
    return reinterpret_cast<const uint8_t*>(base);
  };
  const int nj = (int)(x1 - x0);

  // ---- issue side: runs NST tiles ahead of the compute side
  Unit iu;
  const uint8_t* ikb = nullptr;
  const uint8_t* ivb = nullptr;
  auto issue = [&](const Cursor& c, int j) {
    const bool first = (j == 0) || (c.lt == 0);
    if (first) {
      iu = unit_at(c);
      ikb = kv_base(iu, 0);
      ivb = kv_base(iu, 1);
      if (iu.k1 <= kSelSmem) {  // stage the unit's selected ids once
        __syncwarp();
        for (int i = lane; i < iu.k1; i += 32) sel_s[i] = iu.sel[i];
        __syncwarp();
        iu.sel = sel_s;
      }
    }
    uint8_t* sK = ring + (j % NST) * STAGE;
    uint8_t* sV = sK + TILEB;
    const int t = c.lt;
    const int a0 = t * 16;
    const int ncache = max(0, min(16, iu.n_att - 1 - a0));  // cache rows of the tile
    if (fast) {
      int src0;
      if (a0 < iu.n_sel_rows) {
        const int ci = t / s16;
        int id = iu.sel[ci];
        if (id < 0 || id >= iu.C1) {
          if (lane == 0) atomicOr(&g_mpc_status, 4);
          id = 0;
        }
        src0 = id * s + (a0 - ci * s);
      } else {
        src0 = iu.C1 * s + (a0 - iu.n_sel_rows);
      }
      const uint8_t* gk = ikb + (int64_t)src0 * ROWB;
      const uint8_t* gv = ivb + (int64_t)src0 * ROWB;
      for (int i = lane; i < ncache * CH; i += 32) {
        cp_async16(sK + i * 16, gk + i * 16);
        cp_async16(sV + i * 16, gv + i * 16);
      }
    } else {
      const int r = lane & 15;
      const int arow = a0 + r;
      int src = 0;
      if (r < ncache) src = src_row(iu, s, arow);
      else if (arow == iu.n_att - 1) src = iu.n;
      if (lane < 16) keys[(j % NST) * 16 + r] = (int8_t)((arow < iu.n_att) ? (src & 7) : (r & 7));
#pragma unroll 4
      for (int i = lane; i < 16 * CH; i += 32) {
        const int row = i / CH, ch = i % CH;
        const int srow = __shfl_sync(0xffffffffu, src, row);
        if (row < ncache) {
          cp_async16(sK + i * 16, ikb + (int64_t)srow * ROWB + ch * 16);
          cp_async16(sV + i * 16, ivb + (int64_t)srow * ROWB + ch * 16);
        }
      }
    }
    if (first) {
      const uint8_t* q = reinterpret_cast<const uint8_t*>((const bf16*)p.q + iu.layer * p.q_ls +
                                                          ((int64_t)iu.b * p.Hq + iu.h * G) * D);
      for (int i = lane; i < G * D * 2 / 16; i += 32) cp_async16(sK + 2 * TILEB + i * 16, q + i * 16);
    }
  };

  Cursor cc, ic;
  if (nj > 0) {
    cc = locate(x0);
    ic = cc;
    for (int j = 0; j < NST; ++j) {
      if (j < nj) {
        issue(ic, j);
        advance(ic);
      }
      cp_async_commit();
    }
  }

  // ---- compute side
  uint32_t qb[HN][KS][2];  // Q^T operand: k = channels, n = heads
  float o[KS][HN][4];      // O^T accumulators: m = channels, n = heads
  float m_run[HN][2], l_run[HN][2];
  Unit u;
  int u_ri = 0;
  bool have = false;
  const int r_tok = lane >> 2;      // token row of S^T (and +8)
  const int h_off = 2 * (lane & 3);  // first of this thread's two heads in an n-tile

  auto flush = [&]() {
    float lq[HN][2];
#pragma unroll
    for (int hn = 0; hn < HN; ++hn)
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        float v = l_run[hn][e];
        v += __shfl_xor_sync(0xffffffffu, v, 4);
        v += __shfl_xor_sync(0xffffffffu, v, 8);
        v += __shfl_xor_sync(0xffffffffu, v, 16);
        lq[hn][e] = v;
      }
    const int64_t ustart = (int64_t)u_ri * TPR + (int64_t)Hkv * s_pre[u.b] + (int64_t)u.h * s_nt[u.b];
    const int64_t uend = ustart + s_nt[u.b];
    const bool before = ustart < x0, after = uend > x1;
    float* outp = p.out + u.layer * p.out_ls + ((int64_t)u.b * p.Hq + u.h * G) * D;
    const int64_t unit_id = ((int64_t)u_ri * B + u.b) * Hkv + u.h;
    if (before) {
      // a later piece of a unit that began in an earlier warp: publish the
      // (max, sum, o) record and signal the unit's owner, without waiting
      float* dst = p.part + (int64_t)gw * G * (D + 4);
#pragma unroll
      for (int hn = 0; hn < HN; ++hn)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int g = hn * 8 + h_off + e;
          if (g < G) {
            if (r_tok == 0) {
              dst[g * (D + 4)] = m_run[hn][e];
              dst[g * (D + 4) + 1] = lq[hn][e];
            }
#pragma unroll
            for (int mt = 0; mt < KS; ++mt) {
              dst[g * (D + 4) + 4 + mt * 16 + r_tok] = o[mt][hn][e];
              dst[g * (D + 4) + 4 + mt * 16 + r_tok + 8] = o[mt][hn][2 + e];
            }
          }
        }
      __syncwarp();
      if (lane == 0) red_release_add(&p.unit_counter[unit_id], 1);
    } else {
      if (after) {
        // this warp holds the unit's first piece, which ends last in time:
        // wait for the later pieces' records and merge them into registers
        const int nother = warp_of(uend - 1) - gw;
        int arrived = 1;
        if (lane == 0) {
          if (ld_acquire(&p.unit_counter[unit_id]) < nother) {
            const uint64_t t0 = global_timer_ns();
            while (ld_acquire(&p.unit_counter[unit_id]) < nother) {
              if (global_timer_ns() - t0 > 1000000000ull) {
                atomicOr(&g_mpc_status, kStatusWaitTimeout);
                arrived = 0;
                break;
              }
              __nanosleep(64);
            }
          }
          // a wait that gave up leaves the counter to the late pieces (the
          // caller zero-fills the workspace again after flag 1)
          if (arrived) p.unit_counter[unit_id] = 0;
        }
        arrived = __shfl_sync(0xffffffffu, arrived, 0);
        // no partial output: a unit whose records did not all arrive keeps
        // its previous o and is reported by flag 1 only
        if (!arrived) goto unit_done;
        __syncwarp();
        // the records of warps gw + 1 .. gw + nother are contiguous: copy
        // them into this warp's ring (idle: the owner piece ends the warp's
        // range, after its last tile) with one batch of copies in flight,
        // instead of one dependent round trip per record
        const int rec = G * (D + 4);
        const float* recs = p.part + (int64_t)(gw + 1) * rec;
        const bool staged = nother * rec * 4 <= NST * STAGE;
        auto ld_rec = [&](const float* a) { return staged ? *a : __ldcg(a); };
        if (staged) {
          const uint8_t* src = reinterpret_cast<const uint8_t*>(recs);
          for (int i = lane; i < nother * rec / 4; i += 32) cp_async16(ring + i * 16, src + i * 16);
          cp_async_commit();
          cp_async_wait<0>();
          __syncwarp();
          recs = reinterpret_cast<const float*>(ring);
        }
        for (int k = 1; k <= nother; ++k) {
          const float* rec_k = recs + (int64_t)(k - 1) * rec;
#pragma unroll
          for (int hn = 0; hn < HN; ++hn)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int g = hn * 8 + h_off + e;
              if (g < G) {
                const float* rg = rec_k + g * (D + 4);
                const float mk = ld_rec(rg), lk = ld_rec(rg + 1);
                const float M = fmaxf(m_run[hn][e], mk);
                const float wa = (m_run[hn][e] == kNegInf) ? 0.f : fast_exp2(m_run[hn][e] - M);
                const float wb = (mk == kNegInf) ? 0.f : fast_exp2(mk - M);
                m_run[hn][e] = M;
                lq[hn][e] = lq[hn][e] * wa + lk * wb;
#pragma unroll
                for (int mt = 0; mt < KS; ++mt) {
                  o[mt][hn][e] = o[mt][hn][e] * wa + wb * ld_rec(rg + 4 + mt * 16 + r_tok);
                  o[mt][hn][2 + e] = o[mt][hn][2 + e] * wa + wb * ld_rec(rg + 4 + mt * 16 + r_tok + 8);
                }
              }
            }
        }
      }
#pragma unroll
      for (int hn = 0; hn < HN; ++hn)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int g = hn * 8 + h_off + e;
          if (g < G) {
            const float inv = 1.f / lq[hn][e];
#pragma unroll
            for (int mt = 0; mt < KS; ++mt) {
              outp[g * D + mt * 16 + r_tok] = o[mt][hn][e] * inv;
              outp[g * D + mt * 16 + r_tok + 8] = o[mt][hn][2 + e] * inv;
            }
          }
        }
    }
  unit_done:
    // the piece that holds the appended row seals a full tail
    if (uend <= x1) seal_tail<bf16, D>(p, u, reinterpret_cast<const bf16*>(kv_base(u, 0)));
  };

  for (int j = 0; j < nj; ++j) {
    const int st = j % NST;
    uint8_t* sK = ring + st * STAGE;
    uint8_t* sV = sK + TILEB;
    int8_t* kk = keys + st * 16;
    const bool new_unit = (j == 0) || (cc.lt == 0);
    if (new_unit) {
      if (have) flush();
      u = unit_at(cc);
      u_ri = cc.ri;
      have = true;
#pragma unroll
      for (int hn = 0; hn < HN; ++hn) {
        m_run[hn][0] = m_run[hn][1] = kNegInf;
        l_run[hn][0] = l_run[hn][1] = 0.f;
#pragma unroll
        for (int mt = 0; mt < KS; ++mt) o[mt][hn][0] = o[mt][hn][1] = o[mt][hn][2] = o[mt][hn][3] = 0.f;
      }
    }
    cp_async_wait<NST - 1>();  // this lane's copies of tile j have landed
    __syncwarp();
    if (new_unit) {
      // Q^T operand from the stage's q slot: b0 = q[head][2c, 2c+1], b1 = +8
      const bf16* qs = reinterpret_cast<const bf16*>(sK + 2 * TILEB);
#pragma unroll
      for (int hn = 0; hn < HN; ++hn) {
        const int hq = hn * 8 + r_tok;
#pragma unroll
        for (int ks = 0; ks < KS; ++ks) {
          const int c = ks * 16 + h_off;
          qb[hn][ks][0] = (hq < G) ? *reinterpret_cast<const uint32_t*>(qs + hq * D + c) : 0u;
          qb[hn][ks][1] = (hq < G) ? *reinterpret_cast<const uint32_t*>(qs + hq * D + c + 8) : 0u;
        }
      }
    }
    const int t = cc.lt;
    const int n_valid = min(16, u.n_att - t * 16);
    const int cur_r = (u.n_att - 1) - t * 16;
    if (cur_r < 16 || n_valid < 16) {
      constexpr int CH = ROWB / 16;
      if (cur_r >= 0 && cur_r < 16) {
        // the appended row goes from the inputs to the cache and to this tile
        const int64_t nb = u.layer * p.kvn_ls + (int64_t)(u.b * Hkv + u.h) * D;
        const uint4* kn = reinterpret_cast<const uint4*>((const bf16*)p.k_new + nb);
        const uint4* vn = reinterpret_cast<const uint4*>((const bf16*)p.v_new + nb);
        bf16* kcw = (bf16*)p.kc + u.layer * p.cache_ls + (int64_t)(u.b * Hkv + u.h) * p.cap_tokens * D;
        bf16* vcw = (bf16*)p.vc + u.layer * p.cache_ls + (int64_t)(u.b * Hkv + u.h) * p.cap_tokens * D;
        for (int i = lane; i < 2 * CH; i += 32) {
          const int ch = i % CH;
          const bool isv = i >= CH;
          const uint4 val = isv ? vn[ch] : kn[ch];
          const int pch = ch ^ (u.n & 7);
          *reinterpret_cast<uint4*>((isv ? sV : sK) + cur_r * ROWB + pch * 16) = val;
          reinterpret_cast<uint4*>((isv ? vcw : kcw) + (int64_t)u.n * D)[pch] = val;
        }
      }
      // rows past the end of the list are zeroed so that P V sees finite values
      for (int i = lane; i < (16 - n_valid) * CH; i += 32)
        reinterpret_cast<uint4*>(sV + n_valid * ROWB)[i] = make_uint4(0, 0, 0, 0);
      __syncwarp();
    }
    // S^T = K Q^T: 16 tokens x 8 heads per n-tile, two accumulators per
    // n-tile (even / odd k-steps) to halve the dependency chain
    float sc[HN][2][4];
#pragma unroll
    for (int hn = 0; hn < HN; ++hn)
#pragma unroll
      for (int a2 = 0; a2 < 2; ++a2) sc[hn][a2][0] = sc[hn][a2][1] = sc[hn][a2][2] = sc[hn][a2][3] = 0.f;
    {
      // A = K tile: matrices (tok 0-7, ch 2ks), (tok 8-15, 2ks), (tok 0-7, 2ks+1), (tok 8-15, 2ks+1)
      const int tok = ((lane >> 3) & 1) * 8 + (lane & 7);
      const int key = fast ? (tok & 7) : kk[tok];
      const uint32_t base = smem_u32(sK + tok * ROWB);
      const int chb = lane >> 4;
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        uint32_t a[4];
        ldsm_x4(base + ((((2 * ks + chb) ^ key)) << 4), a[0], a[1], a[2], a[3]);
#pragma unroll
        for (int hn = 0; hn < HN; ++hn) mma_bf16(sc[hn][ks & 1], a, qb[hn][ks][0], qb[hn][ks][1]);
      }
    }
    uint32_t pbh[HN][2], pbl[HN][2];
    float corr[HN][2];
#pragma unroll
    for (int hn = 0; hn < HN; ++hn) {
      float x[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int tk = r_tok + (e >> 1) * 8;
        x[e] = (t * 16 + tk < u.n_att) ? (sc[hn][0][e] + sc[hn][1][e]) * p.scale_log2 : kNegInf;
      }
      float pr[4];
#pragma unroll
      for (int e = 0; e < 2; ++e) {  // this thread's two heads
        float mx = fmaxf(x[e], x[e + 2]);
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
        const float mnew = fmaxf(m_run[hn][e], mx);
        corr[hn][e] = (m_run[hn][e] == kNegInf) ? 0.f : fast_exp2(m_run[hn][e] - mnew);
        m_run[hn][e] = mnew;
        pr[e] = fast_exp2(x[e] - mnew);
        pr[e + 2] = fast_exp2(x[e + 2] - mnew);
        l_run[hn][e] = l_run[hn][e] * corr[hn][e] + pr[e] + pr[e + 2];
      }
      // P^T operand (k = tokens, n = heads): transpose the 8x8 blocks of P
      const __nv_bfloat162 h01 = __floats2bfloat162_rn(pr[0], pr[1]);
      const __nv_bfloat162 h23 = __floats2bfloat162_rn(pr[2], pr[3]);
      const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
      pbh[hn][0] = movmatrix_t(*reinterpret_cast<const uint32_t*>(&h01));
      pbh[hn][1] = movmatrix_t(*reinterpret_cast<const uint32_t*>(&h23));
      pbl[hn][0] = movmatrix_t(pack_bf16(pr[0] - f01.x, pr[1] - f01.y));
      pbl[hn][1] = movmatrix_t(pack_bf16(pr[2] - f23.x, pr[3] - f23.y));
    }
#pragma unroll
    for (int mt = 0; mt < KS; ++mt)
#pragma unroll
      for (int hn = 0; hn < HN; ++hn) {
        o[mt][hn][0] *= corr[hn][0];
        o[mt][hn][1] *= corr[hn][1];
        o[mt][hn][2] *= corr[hn][0];
        o[mt][hn][3] *= corr[hn][1];
      }
    {
      // A = V^T tile: transposed matrices (tok 0-7, ch 2mt), (tok 0-7, 2mt+1), (tok 8-15, 2mt), (tok 8-15, 2mt+1)
      const int tok = (lane >> 4) * 8 + (lane & 7);
      const int key = fast ? (tok & 7) : kk[tok];
      const uint32_t base = smem_u32(sV + tok * ROWB);
      const int chb = (lane >> 3) & 1;
#pragma unroll
      for (int mt = 0; mt < KS; ++mt) {
        uint32_t a[4];
        ldsm_x4_t(base + ((((2 * mt + chb) ^ key)) << 4), a[0], a[1], a[2], a[3]);
#pragma unroll
        for (int hn = 0; hn < HN; ++hn) {
          mma_bf16(o[mt][hn], a, pbh[hn][0], pbh[hn][1]);
          mma_bf16(o[mt][hn], a, pbl[hn][0], pbl[hn][1]);
        }
      }
    }
    __syncwarp();
    if (j + NST < nj) {
      issue(ic, j + NST);
      advance(ic);
    }
    cp_async_commit();  // one group per tile, empty near the end
    advance(cc);
  }
  cp_async_wait<0>();
  if (have) flush();
  finish_grid(p);
}

// ------------------------------------------------------------- f32 path ----
template <int D, int GM>
__global__ void __launch_bounds__(128) attn_f32_kernel(const __grid_constant__ AttnParams p) {
  using S = Smem<D, 4>;
  constexpr int ROWB = S::ROWB;
  constexpr int PER = D / 32;  // output channels per lane
  extern __shared__ __align__(128) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  grid_dep_launch();
  grid_dep_wait();
  const Unit u = make_unit(p);
  const int s = p.pyr.s;
  const int G = p.G;
  float* kcache = (float*)p.kc + u.layer * p.cache_ls + (int64_t)(u.b * p.Hkv + u.h) * p.cap_tokens * D;
  float* vcache = (float*)p.vc + u.layer * p.cache_ls + (int64_t)(u.b * p.Hkv + u.h) * p.cap_tokens * D;
  float* mw = reinterpret_cast<float*>(smem + S::MERGE_OFF);
  float* qs = mw + kWarps * G * (D + 4);

  if (u.n < 0 || u.n + 1 > p.cap_tokens) {
    if (threadIdx.x == 0) atomicOr(&g_mpc_status, 2);
    finish_grid(p);
    return;
  }

  uint8_t* ring = smem + warp * kStages * S::STAGE_BYTES;
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + S::BAR_OFF) + warp * kStages;
  int8_t* keys = reinterpret_cast<int8_t*>(smem + S::KEY_OFF) + warp * kStages * 16;
  for (int i = lane; i < kStages * S::STAGE_BYTES / 16; i += 32)
    reinterpret_cast<uint4*>(ring)[i] = make_uint4(0, 0, 0, 0);
  {
    const float* qp = (const float*)p.q + u.layer * p.q_ls + ((int64_t)u.b * p.Hq + u.h * G) * D;
    for (int i = threadIdx.x; i < G * D; i += blockDim.x) qs[i] = qp[i];
  }
  if (lane == 0) {
    for (int st = 0; st < kStages; ++st) mbar_init(&bar[st], 1);
    fence_barrier_init();
  }
  fence_proxy_async_smem();
  __syncthreads();

  const int first = u.t_begin + warp;
  const int nj = (u.t_end > first) ? (u.t_end - first + kWarps - 1) / kWarps : 0;
  for (int j = 0; j < kStages && j < nj; ++j) {
    uint8_t* sK = ring + j * S::STAGE_BYTES;
    issue_tile<ROWB>(u, s, first + j * kWarps, (const uint8_t*)kcache, (const uint8_t*)vcache, sK,
                     sK + S::TILEB, keys + j * 16, &bar[j], lane);
  }

  float o[GM][PER];
  float m_run[GM], l_run[GM];
#pragma unroll
  for (int g = 0; g < GM; ++g) {
    m_run[g] = kNegInf;
    l_run[g] = 0.f;
#pragma unroll
    for (int i = 0; i < PER; ++i) o[g][i] = 0.f;
  }
  uint32_t phase = 0;
  bool ok = true;
  const int r = lane & 15, hf = lane >> 4;

  for (int j = 0; j < nj; ++j) {
    const int st = j % kStages;
    const int t = first + j * kWarps;
    uint8_t* sK = ring + st * S::STAGE_BYTES;
    uint8_t* sV = sK + S::TILEB;
    int8_t* kk = keys + st * 16;
    if (!mbar_wait_bounded(&bar[st], (phase >> st) & 1u)) {
      ok = false;
      break;
    }
    phase ^= (1u << st);
    const int cur_r = (u.n_att - 1) - t * 16;
    if (cur_r >= 0 && cur_r < 16) {
      const int64_t nb = u.layer * p.kvn_ls + (int64_t)(u.b * p.Hkv + u.h) * D;
      const uint4* kn = reinterpret_cast<const uint4*>((const float*)p.k_new + nb);
      const uint4* vn = reinterpret_cast<const uint4*>((const float*)p.v_new + nb);
      constexpr int CH = ROWB / 16;
      for (int i = lane; i < 2 * CH; i += 32) {
        const int ch = i % CH;
        const bool isv = i >= CH;
        const uint4 val = isv ? vn[ch] : kn[ch];
        const int pch = ch ^ (u.n & 7);
        *reinterpret_cast<uint4*>((isv ? sV : sK) + cur_r * ROWB + pch * 16) = val;
        reinterpret_cast<uint4*>((isv ? vcache : kcache) + (int64_t)u.n * D)[pch] = val;
      }
      __syncwarp();
    }
    // scores: lane (r, hf) takes row r, channels [hf D/2, (hf+1) D/2)
    const int key = kk[r];
    const float* krow = reinterpret_cast<const float*>(sK + r * ROWB);
    float sc[GM];
#pragma unroll
    for (int g = 0; g < GM; ++g) sc[g] = 0.f;
#pragma unroll
    for (int cc = 0; cc < D / 8; ++cc) {
      const int ch = hf * (D / 8) + cc;
      const float4 kv = *reinterpret_cast<const float4*>(krow + ((ch ^ key) << 2));
#pragma unroll
      for (int g = 0; g < GM; ++g) {
        if (g < G) {
          const float4 qv = *reinterpret_cast<const float4*>(qs + g * D + ch * 4);
          sc[g] = fmaf(qv.x, kv.x, sc[g]);
          sc[g] = fmaf(qv.y, kv.y, sc[g]);
          sc[g] = fmaf(qv.z, kv.z, sc[g]);
          sc[g] = fmaf(qv.w, kv.w, sc[g]);
        }
      }
    }
    const bool valid = t * 16 + r < u.n_att;
    float pg[GM];
#pragma unroll
    for (int g = 0; g < GM; ++g) {
      if (g >= G) continue;
      float v = sc[g] + __shfl_xor_sync(0xffffffffu, sc[g], 16);
      v = valid ? v * p.scale_log2 : kNegInf;
      float mx = v;
#pragma unroll
      for (int off = 1; off < 16; off <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
      const float mnew = fmaxf(m_run[g], mx);
      const float corr = (m_run[g] == kNegInf) ? 0.f : fast_exp2(m_run[g] - mnew);
      m_run[g] = mnew;
      pg[g] = fast_exp2(v - mnew);
      float sum = pg[g];
#pragma unroll
      for (int off = 1; off < 16; off <<= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
      l_run[g] = l_run[g] * corr + sum;
#pragma unroll
      for (int i = 0; i < PER; ++i) o[g][i] *= corr;
    }
    // O += P V: lane owns channels [lane PER, (lane+1) PER)
#pragma unroll 4
    for (int rr = 0; rr < 16; ++rr) {
      const int kr = kk[rr];
      const float* vrow = reinterpret_cast<const float*>(sV + rr * ROWB);
      const int c0 = lane * PER;
      const int ch = c0 >> 2;
      const float* vp = vrow + ((ch ^ kr) << 2) + (c0 & 3);
#pragma unroll
      for (int g = 0; g < GM; ++g) {
        if (g >= G) continue;
        const float pv = __shfl_sync(0xffffffffu, pg[g], rr);
#pragma unroll
        for (int i = 0; i < PER; ++i) o[g][i] = fmaf(pv, vp[i], o[g][i]);
      }
    }
    __syncwarp();
    if (j + kStages < nj) {
      fence_proxy_async_smem();
      __syncwarp();
      issue_tile<ROWB>(u, s, t + kStages * kWarps, (const uint8_t*)kcache, (const uint8_t*)vcache, sK,
                       sV, kk, &bar[st], lane);
    }
  }
  if (!ok)
    for (int st = 0; st < kStages; ++st) mbar_wait_bounded(&bar[st], (phase >> st) & 1u);

#pragma unroll
  for (int g = 0; g < GM; ++g) {
    if (g >= G) continue;
    float* dst = mw + (warp * G + g) * (D + 4);
    if (lane == 0) {
      dst[0] = (ok && nj > 0) ? m_run[g] : kNegInf;
      dst[1] = (ok && nj > 0) ? l_run[g] : 0.f;
    }
#pragma unroll
    for (int i = 0; i < PER; ++i) dst[4 + lane * PER + i] = ok ? o[g][i] : 0.f;
  }
  if (u.t_begin < u.n_tiles) {
    merge_and_store<D>(p, u, mw, kWarps);
    if ((u.n_att - 1) / 16 >= u.t_begin && (u.n_att - 1) / 16 < u.t_end) {
      __syncthreads();
      if (threadIdx.x < 32) seal_tail<float, D>(p, u, kcache);
    }
  } else if (p.n_split > 1) {
    for (int i = threadIdx.x; i < G * (D + 4); i += blockDim.x) mw[i] = (i % (D + 4) == 0) ? kNegInf : 0.f;
    merge_and_store<D>(p, u, mw, 1);
  }
  finish_grid(p);
}

// ------------------------------------------------------------- launch ----

int attn_smem_bytes(int dtype, int D, int G, int B) {
  if (dtype == MPC_BF16) {
    const PersistCfg c = persist_cfg(D, G, B);
    return D == 64 ? PSmem<64>::total(G, c.nst, c.wpc, B) : PSmem<128>::total(G, c.nst, c.wpc, B);
  }
  return D == 64 ? Smem<64, 4>::total(G) : Smem<128, 4>::total(G);
}

int attn_persist_ctas_max() { return kMaxPersistCtas; }
int attn_persist_batch_max() { return kMaxBatchPersist; }

template <typename K>
static cudaError_t launch_k(K kernel, dim3 grid, int smem, cudaStream_t st, const AttnParams& p, int threads = 128) {
  cudaError_t e = ensure_dyn_smem((const void*)kernel, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(kernel, grid, dim3(threads), smem, st, p);
}

// The persistent kernel's owners wait for pieces held by other CTAs, so its
// grid is launched cooperatively: all CTAs resident together.
template <typename K>
static cudaError_t launch_persist(K kernel, dim3 grid, int smem, cudaStream_t st, const AttnParams& p, int threads) {
  cudaError_t e = ensure_dyn_smem((const void*)kernel, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl_coop(kernel, grid, dim3(threads), smem, st, p);
}

// CTAs of the persistent grid: one per SM, at most kMaxPersistCtas.
static int persist_ctas() {
  static std::mutex mu;
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return kMaxPersistCtas;
  std::lock_guard<std::mutex> lk(mu);
  if (cached[dev] == 0) {
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
      sms = kMaxPersistCtas;
    cached[dev] = sms < kMaxPersistCtas ? sms : kMaxPersistCtas;
  }
  return cached[dev];
}

cudaError_t launch_attn(const AttnParams& p0, int dtype, int D, int n_units, cudaStream_t st) {
  AttnParams p = p0;
  if (dtype == MPC_BF16) {
    const PersistCfg c = persist_cfg(D, p.G, p.B);
    p.n_stages = c.nst;
    const int smem = attn_smem_bytes(dtype, D, p.G, p.B);
    const dim3 grid(persist_ctas());
    const int th = 32 * c.wpc;
#define MPC_PERSIST(DD, HH, NN, WW)                                                                 \
  if (D == DD && (p.G <= 8 ? 1 : 2) == HH && c.nst == NN && c.wpc == WW)                           \
    return launch_persist(attn_bf16_persist_kernel<DD, HH, NN, WW>, grid, smem, st, p, th);
    MPC_PERSIST(64, 1, 8, 4)
    MPC_PERSIST(128, 1, 3, 8)
    MPC_PERSIST(128, 1, 4, 6)
    MPC_PERSIST(128, 1, 5, 4)
    MPC_PERSIST(64, 2, 8, 4)
    MPC_PERSIST(128, 2, 4, 4)
#undef MPC_PERSIST
    return cudaErrorInvalidValue;
  }
  const dim3 grid(p.n_split, n_units);
  const int smem = attn_smem_bytes(dtype, D, p.G, p.B);
  const int G = p.G;
#define MPC_F32_CASE(DD, GG) \
  if (D == DD && G <= GG) return launch_k(attn_f32_kernel<DD, GG>, grid, smem, st, p);
  MPC_F32_CASE(64, 1) MPC_F32_CASE(64, 2) MPC_F32_CASE(64, 4) MPC_F32_CASE(64, 8)
  MPC_F32_CASE(128, 1) MPC_F32_CASE(128, 2) MPC_F32_CASE(128, 4) MPC_F32_CASE(128, 8)
#undef MPC_F32_CASE
  return cudaErrorInvalidValue;
}

int take_status_attn() { return take_status(); }

}  // namespace mpc
