// Sparse decode attention over the selected clusters and the tail, with the
// decode-step append and the tail seal (Alg. 1; Alg. 2 Step 2; App. A), for
// fp32 caches.  (bf16 caches take the decode step kernel, decode_step.cu,
// with the selections as inputs.)
//
// Work decomposition: one unit = (ref, sequence b, kv head h).  The rows a
// unit attends are listed in order: the s rows of every selected cluster,
// then the tail rows already in the cache, then the row appended now.  The
// list is cut into 16-row tiles and the tiles into `tiles_per_split` chunks,
// one CTA per (chunk, unit).  Each of the CTA's four warps streams its tiles
// (key rows and value rows) from HBM into its own shared-memory ring with 1-D
// bulk copies (TMA engine, completion on an mbarrier), then computes the
// tile's scores for all query heads of the GQA group at once and updates an
// online softmax.  The four warps' partial results are merged in shared
// memory; with several chunks per unit the CTA writes (max, sum, o) to the
// workspace and the last CTA of the unit (atomic ticket, no waiting) merges
// them by log-sum-exp and writes o.
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

template <typename K>
static cudaError_t launch_k(K kernel, dim3 grid, int smem, cudaStream_t st, const AttnParams& p, int threads = 128) {
  cudaError_t e = ensure_dyn_smem((const void*)kernel, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(kernel, grid, dim3(threads), smem, st, p);
}

cudaError_t launch_attn(const AttnParams& p0, int dtype, int D, int n_units, cudaStream_t st) {
  const AttnParams& p = p0;
  if (dtype != MPC_F32) return cudaErrorInvalidValue;
  const dim3 grid(p.n_split, n_units);
  const int smem = D == 64 ? Smem<64, 4>::total(p.G) : Smem<128, 4>::total(p.G);
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
