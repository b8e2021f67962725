// Hierarchical cluster selection of one decode step (Sec. 3.3-3.4, Eq. 3;
// Alg. 2 Step 2, Sim + topk) for the leader layer of each sharing group.
//
// One CTA per (ref, sequence b, kv head h).  The GQA group's queries are
// summed once (Eq. 3 is linear in q, so the sum scores the group), then the
// levels are walked from the coarsest down.  Each candidate is held as one
// 64-bit key (orderable score, inverted id: all keys distinct, larger score
// first, then smaller id), so the key alone carries the id and the score.
// The orderable score is the fp32 similarity's order-preserving bit pattern,
// or, for the fixed-point metric, the int32 score with its sign bit flipped.
//
// The walk is bounded by global-load latency, so the fp32 representatives
// a level needs are staged in shared memory by 1-D bulk copies (contiguous
// runs: the whole coarsest level, or the children of one kept cluster) on
// one mbarrier, and scoring is batched into as few dependent rounds as the
// pyramid allows.  The first round, requested as soon as the token count
// arrives (while q is still loading), copies the coarsest level and, while
// the units are few enough to be latency-bound and both fit the staging
// buffer, all clusters of the level below it, whose scores then need no
// round of their own (a three-level pyramid takes two rounds).  Per level, with a
// block barrier after each step:
//   1. rank: a candidate is kept iff fewer than k keys are larger, counted
//      by up to 32 threads per candidate over shared memory (a bitonic sort
//      of a copy gives the k-th key instead above 1024 candidates);
//   2. warp 0 compacts the kept positions in candidate order with ballots,
//      so the kept ids stay ascending;
//   3. the block writes the kept clusters' children as the next level's
//      keys, with their scores when the first round computed them.
#include "kernels.cuh"
#include "sel_score.cuh"

namespace mpc {

constexpr int kRankMax = 1024;  // candidates ranked by counting

constexpr int kSelChunk = 8192; // bytes per bulk copy

// Resident CTAs per SM asked of the 4-warp instantiation (many small units:
// latency-bound, so residency sets the throughput); the call caps the staged
// rows so that six CTAs' shared memory fits the SM.  Measured on the
// batch-32 paged workload: 5 CTAs (96 registers) 163 us per selection, 6
// (80 registers, no spills since the scoring keeps one float per chunk live)
// 151 us; 7 and 8 spill.
constexpr int kSelMinCtas128 = 6;

// Fixed-point Eq. 3 (ring Z_{2^64}, f fractional bits) of four channels:
// sum_j q_j rep_j with rep_j = tr(a enc(r_max_j)) + tr(b enc(r_min_j)), the
// products and sums wrapping modulo 2^64; tr is the arithmetic shift by f.
// x 2^f is exact in fp32, and the conversion rounds ties to even.
__device__ __forceinline__ unsigned long long fxp_dot4(const long long (&q)[4], float4 mx, float4 mn, float sc,
                                                       long long a, long long b, int f) {
  const float x[4] = {mx.x, mx.y, mx.z, mx.w}, y[4] = {mn.x, mn.y, mn.z, mn.w};
  unsigned long long acc = 0ull;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const long long ex = __float2ll_rn(x[j] * sc), ey = __float2ll_rn(y[j] * sc);
    const long long pa = (long long)((unsigned long long)a * (unsigned long long)ex) >> f;
    const long long pb = (long long)((unsigned long long)b * (unsigned long long)ey) >> f;
    const unsigned long long r = (unsigned long long)pa + (unsigned long long)pb;
    acc += (unsigned long long)q[j] * r;
  }
  return acc;
}

// Orderable key of a truncated ring dot product: tr(acc) saturated to int32.
__device__ __forceinline__ uint32_t fxp_oscore(unsigned long long acc, int f) {
  long long v = (long long)acc >> f;
  v = v > 2147483647ll ? 2147483647ll : (v < -2147483648ll ? -2147483648ll : v);
  return (uint32_t)(int32_t)v ^ 0x80000000u;
}

// Shared-memory layout of one select CTA (host and device): n_src staged
// row arrays (rep or mean, or r_max and r_min), then the summed query (fp32,
// or int64 encodings for the fixed-point metric), then the scalars.
struct SelLayout {
  size_t qsum, cs, keys, mark, kept, total;
  __host__ __device__ SelLayout(int D, int MC, int RB, int n_src) {
    qsum = (size_t)n_src * RB * D * 4;     // staged rows first (16-byte aligned)
    cs = qsum + (size_t)D * 8;              // orderable scores of the first round's children
    keys = (cs + (size_t)RB * 4 + 15) & ~(size_t)15;
    mark = keys + (size_t)MC * 16;          // two key arrays
    kept = mark + (size_t)MC * 4;
    total = kept + (size_t)MC * 4;
  }
};

// Warp-cooperative copy of nbytes (a multiple of 16) in chunks, lanes in
// parallel, completing on bar.
__device__ __forceinline__ void warp_copy(void* dst, const void* src, uint32_t nbytes, uint64_t* bar, int lane) {
  for (uint32_t off = (uint32_t)lane * kSelChunk; off < nbytes; off += 32u * kSelChunk) {
    const uint32_t nb = nbytes - off < (uint32_t)kSelChunk ? nbytes - off : (uint32_t)kSelChunk;
    bulk_g2s(static_cast<uint8_t*>(dst) + off, static_cast<const uint8_t*>(src) + off, nb, bar);
  }
}

// FXP: the fixed-point metric (its own instantiation, so the fp32 metrics
// keep their register budget).
template <typename T, int D, int NT, bool FXP>
__global__ void __launch_bounds__(NT, NT == 128 ? kSelMinCtas128 : 1) select_kernel(const __grid_constant__ SelectParams p) {
  constexpr int NW = NT / 32;
  constexpr int LPR = D / 4;     // lanes per representative row (one float4 each)
  constexpr int RPW = 32 / LPR;  // rows per warp-wide read
  constexpr int U = 8;           // rows per lane per pass
  constexpr uint32_t ROWB = D * 4;
  constexpr int kFastMax = 16 * NW;  // candidates ranked from registers (NW / 2 keys per lane)
  constexpr int kWarpMax = 32;       // candidates ranked by warp 0 alone (one per lane)
  extern __shared__ __align__(128) uint8_t smem[];
  const int MC = p.max_cand, RB = p.row_buf;
  const int NSRC = FXP ? 2 : select_n_src(p.metric);  // summary rows per candidate
  const SelLayout L(D, MC, RB, NSRC);
  float* rows = reinterpret_cast<float*>(smem);
  float* qsum = reinterpret_cast<float*>(smem + L.qsum);
  uint32_t* cs = reinterpret_cast<uint32_t*>(smem + L.cs);
  unsigned long long* keysA = reinterpret_cast<unsigned long long*>(smem + L.keys);
  unsigned long long* keysB = keysA + MC;
  int* mark = reinterpret_cast<int*>(smem + L.mark);
  int* kept = reinterpret_cast<int*>(smem + L.kept);
  __shared__ __align__(8) uint64_t s_bar;
  __shared__ int s_C[kMaxLevels], s_k[kMaxLevels];
  __shared__ int s_nk, s_next;
  __shared__ int s_walk[4];  // warp walk: level reached, candidates, kept, flags
  __shared__ uint32_t s_wmask[NW];

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int c4 = lane % LPR, sub = lane / LPR;
  const int unit = blockIdx.x;
  const int h = unit % p.Hkv, b = (unit / p.Hkv) % p.B, ri = unit / (p.Hkv * p.B);
  const int layer = p.refs.layer[ri], group = p.refs.group[ri];
  const int G = p.G;
  const int top = p.pyr.n_levels - 1;
  const int64_t unit_off = ((int64_t)(group * p.B + b) * p.Hkv + h) * p.pyr.rows * D;
  // staged source w of a candidate: rep (Eq. 3) or mean (average key), or
  // r_max then r_min (Eq. 2, fixed-point Eq. 3), each into its own RB-row
  // array of the buffer
  const float* one = p.metric == MPC_SIM_MEAN ? p.mean : p.rep;
  const float* src0[2] = {(NSRC == 2 ? p.rmax : one) + unit_off, (NSRC == 2 ? p.rmin : one) + unit_off};
  int* out = p.out_sel + ((int64_t)(group * p.B + b) * p.Hkv + h) * p.sel_cap;
  uint32_t phase = 0;
  bool timed_out = false;

  // similarity of staged row r for rows [0, nrows) of the buffer;
  // put(r, orderable score) runs on one lane of each row.
  //   Eq. 3: q_sum . rep;  mean: q_sum . mean;  Eq. 2: sum_i max(q_i r_max_i, q_i r_min_i);
  //   fixed point: integer, so the order of the ring sums does not matter
  auto score_rows = [&](int nrows, auto&& put) {
    const float* rows2 = rows + (size_t)RB * D;
    if constexpr (FXP) {
      const long long* qf = reinterpret_cast<const long long*>(qsum) + c4 * 4;
      const long long qx[4] = {qf[0], qf[1], qf[2], qf[3]};
      const int fb = p.frac_bits;
      const float sc = (float)(1 << fb);
      const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int r0 = warp * U * RPW; r0 < nrows; r0 += NW * U * RPW) {
        unsigned long long acc[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const int r = r0 + u * RPW + sub;
          const float4 v = r < nrows ? reinterpret_cast<const float4*>(rows + (size_t)r * D)[c4] : z;
          const float4 m = r < nrows ? reinterpret_cast<const float4*>(rows2 + (size_t)r * D)[c4] : z;
          acc[u] = fxp_dot4(qx, v, m, sc, p.fxp_a, p.fxp_b, fb);
        }
#pragma unroll
        for (int o = LPR / 2; o > 0; o >>= 1) {
#pragma unroll
          for (int u = 0; u < U; ++u) acc[u] += __shfl_xor_sync(0xffffffffu, acc[u], o);
        }
        if (c4 == 0) {
#pragma unroll
          for (int u = 0; u < U; ++u) {
            const int r = r0 + u * RPW + sub;
            if (r < nrows) put(r, fxp_oscore(acc[u], fb));
          }
        }
      }
    } else {
      // 4 lanes per row, each with a quarter of the channels and that
      // quarter of q in registers (row_partial: reads rotated by the row's
      // parity against bank conflicts, products summed in channel order)
      constexpr int V4 = D / 16;  // float4 chunks per lane
      const int ql = lane & 3, rs = lane >> 2, rot = rs & 1;
      float4 qv[V4];
      qv_load_order<D>(qv, qsum, ql, rot);
      for (int r0 = warp * 8; r0 < nrows; r0 += NW * 8) {
        const int r = r0 + rs;
        float a = 0.f;
        if (r < nrows) {
          a = NSRC == 1 ? row_partial<D, false>(rows + (size_t)r * D, nullptr, qv, ql, rot)
                        : row_partial<D, true>(rows + (size_t)r * D, rows2 + (size_t)r * D, qv, ql, rot);
        }
        a += __shfl_xor_sync(0xffffffffu, a, 1);
        a += __shfl_xor_sync(0xffffffffu, a, 2);
        if (ql == 0 && r < nrows) put(r, orderable(a));
      }
    }
  };
  auto wait_rows = [&]() {
    if (!mbar_wait_bounded(&s_bar, phase)) timed_out = true;
    phase ^= 1u;
  };

  if (tid == 0) {
    mbar_init(&s_bar, 1);
    fence_barrier_init();
  }
  grid_dep_launch();
  grid_dep_wait();

  // ---- first round, requested before the token count arrives: the
  // capacity rows [0, nT0) of the coarsest level at buffer row 0 and, when
  // spec0, the capacity of the level below it at buffer row capT (rows past
  // the live clusters are copied and never scored)
  const int capT = p.pyr.cap[top];
  const int capC = top > 0 ? p.pyr.cap[top - 1] : 0;
  const bool spec0 = p.spec_first && top > 0 && capT + capC <= RB;
  const int nT0 = capT < RB ? capT : RB;
  const int64_t offT = (int64_t)p.pyr.off[top] * D;
  const int64_t offC = (int64_t)(top > 0 ? p.pyr.off[top - 1] : 0) * D;
  if (warp == 0) {
    const int nCc = spec0 ? capC : 0;
    if (lane == 0) mbar_arrive_expect_tx(&s_bar, (uint32_t)(nT0 + nCc) * ROWB * NSRC);
    __syncwarp();
    for (int w = 0; w < NSRC; ++w) {
      warp_copy(rows + (size_t)w * RB * D, src0[w] + offT, (uint32_t)nT0 * ROWB, &s_bar, lane);
      if (nCc > 0) warp_copy(rows + ((size_t)w * RB + capT) * D, src0[w] + offC, (uint32_t)nCc * ROWB, &s_bar, lane);
    }
  }
  const int ntok = p.n_tok[b];
  int C[kMaxLevels];
  level_counts(p.pyr, ntok, C);

  // q_sum = sum over the group's query heads (fixed order); fixed point:
  // the ring sum of the heads' encodings
  const T* qp = (const T*)p.q + layer * p.q_ls + ((int64_t)b * p.Hq + h * G) * D;
  if constexpr (FXP) {
    const float sc = (float)(1 << p.frac_bits);
    for (int c = tid; c < D; c += NT) {
      unsigned long long acc = 0ull;
      for (int g = 0; g < G; ++g) acc += (unsigned long long)__float2ll_rn(to_float<T>(qp[g * D + c]) * sc);
      reinterpret_cast<long long*>(qsum)[c] = (long long)acc;
    }
  } else {
    for (int c = tid; c < D; c += NT) {
      float acc = 0.f;
      for (int g = 0; g < G; ++g) acc += to_float<T>(qp[g * D + c]);
      qsum[c] = acc;
    }
  }
  if (tid < kMaxLevels) {
    s_C[tid] = C[tid];
    s_k[tid] = tid < p.pyr.n_levels ? count_from_ppm(C[tid], p.keep_ppm[tid]) : 0;
  }
  bool overflow = C[0] > p.pyr.cap[0] || C[top] > MC;
  __syncthreads();
  wait_rows();

  int n = overflow ? 0 : C[top];
  {
    const int nC = top > 0 ? C[top - 1] : 0;
    const int own = n < nT0 ? n : nT0;
    score_rows(spec0 ? capT + nC : own, [&](int r, uint32_t sc) {
      if (r < own) keysA[r] = cand_key(sc, r);
      else if (r >= capT) cs[r - capT] = sc;
    });
    __syncthreads();
    // the rest of a coarsest level larger than the buffer
    for (int x0 = nT0; x0 < n; x0 += RB) {
      const int nb = min(RB, n - x0);
      if (warp == 0) {
        if (lane == 0) mbar_arrive_expect_tx(&s_bar, (uint32_t)nb * ROWB * NSRC);
        __syncwarp();
        for (int w = 0; w < NSRC; ++w)
          warp_copy(rows + (size_t)w * RB * D, src0[w] + offT + (int64_t)x0 * D, (uint32_t)nb * ROWB, &s_bar, lane);
      }
      wait_rows();
      score_rows(nb, [&](int r, uint32_t sc) { keysA[x0 + r] = cand_key(sc, x0 + r); });
      __syncthreads();
    }
  }
  bool have_child = spec0;  // cs holds the scores of all children of keysA[0, n)
  bool need_score = false;  // keysA holds ids only

  int nk = 0;
  for (int l = top; l >= 0 && !overflow; --l) {
    const int f = l > 0 ? p.pyr.fanout[l - 1] : 1;
    const int nC = l > 0 ? s_C[l - 1] : 0;
    if (need_score) {
      // a round over the candidates' own rows, in batches of RB rows,
      // copied by every thread in 16-byte pieces (the rows are scattered
      // runs of fl; spreading the copies over all warps issues them at once)
      constexpr int CPR = ROWB / 16;  // pieces per row
      const int64_t offL = (int64_t)p.pyr.off[l] * D;
      for (int x0 = 0; x0 < n; x0 += RB) {
        const int x1 = min(n, x0 + RB);
        for (int c = tid; c < (x1 - x0) * CPR; c += NT) {
          const int r = c / CPR, part = c - r * CPR;
          const int64_t srow = offL + (int64_t)cand_id(keysA[x0 + r]) * D + part * 4;
          for (int w = 0; w < NSRC; ++w) cp_async16(rows + ((size_t)w * RB + r) * D + part * 4, src0[w] + srow);
        }
        cp_async_commit();
        cp_async_wait<0>();
        __syncthreads();
        score_rows(x1 - x0, [&](int r, uint32_t sc) { keysA[x0 + r] = cand_key(sc, cand_id(keysA[x0 + r])); });
        __syncthreads();
      }
    }

    const int k = min(s_k[l], n);
    if (n <= kWarpMax) {
      // warp 0 ranks this level, expands the kept clusters, and goes on
      // down while the next level's scores are known and its candidates
      // fit, with no block barrier; it stops at level 0, or before a level
      // whose rows must be scored
      if (warp == 0) {
        const unsigned lt = (1u << lane) - 1u;
        unsigned long long* ka = keysA;
        unsigned long long* kb = keysB;
        int lw = l, nw = n, nkw = 0, flags = 0;  // flags: 1 need_score, 2 overflow, 4 swapped, 8 done
        bool hc = have_child;
        while (true) {
          const int kl = min(s_k[lw], nw);
          const int fw = lw > 0 ? p.pyr.fanout[lw - 1] : 1;
          const int nCw = lw > 0 ? s_C[lw - 1] : 0;
          // rank from registers: lane i holds candidate i; the keys of the
          // other lanes arrive by shuffle (all 32 independent, no memory)
          const unsigned long long ki = lane < nw ? ka[lane] : 0ull;
          int cnt = 0;
          if (kl < nw) {
#pragma unroll
            for (int j = 0; j < 32; ++j) cnt += (int)(__shfl_sync(0xffffffffu, ki, j) > ki);
          }
          const bool keep = lane < nw && cnt < kl;
          const unsigned bal = __ballot_sync(0xffffffffu, keep);
          if (keep) {
            const int pos = __popc(bal & lt);
            const int id = cand_id(ki);
            if (lw == 0) {
              if (pos < p.sel_cap) out[pos] = id;
            } else {
              for (int j = 0; j < fw; ++j) {
                const int cid = id * fw + j;
                if (cid < nCw) kb[pos * fw + j] = hc ? cand_key(cs[lane * fw + j], cid) : cand_key(0u, cid);
              }
            }
          }
          const int base = __popc(bal);
          const int last = bal ? __shfl_sync(0xffffffffu, cand_id(ki), 31 - __clz(bal)) : -1;
          nkw = base;
          if (lw == 0) {
            flags |= 8;
            break;
          }
          const int nn = base > 0 ? (base - 1) * fw + min(fw, nCw - last * fw) : 0;
          if (nn > MC) {
            flags |= 2;
            break;
          }
          __syncwarp();
          unsigned long long* t = ka;
          ka = kb;
          kb = t;
          flags ^= 4;
          nw = nn;
          --lw;
          if (!hc) {
            flags |= 1;
            break;
          }
          hc = false;
          if (nw > kWarpMax) break;
        }
        if (lane == 0) {
          s_walk[0] = lw;
          s_walk[1] = nw;
          s_walk[2] = nkw;
          s_walk[3] = flags;
        }
      }
      __syncthreads();
      const int flags = s_walk[3];
      nk = s_walk[2];
      if (flags & 4) {
        unsigned long long* t = keysA;
        keysA = keysB;
        keysB = t;
      }
      if (flags & 2) overflow = true;
      if (flags & 10) break;
      l = s_walk[0] + 1;  // the loop steps down to the level reached
      n = s_walk[1];
      need_score = (flags & 1) != 0;
      have_child = false;
      continue;
    }
    if (n <= kFastMax) {
      // rank, compact and expand in two barriers: every lane holds its
      // share of the keys; warp w ranks candidates [w C, w C + C) with one
      // warp-wide reduction each and records the kept ones in a bit mask;
      // after a barrier each warp places its kept clusters (and their
      // children) at the offset given by the masks of the warps before it
      constexpr int MJ = kFastMax / 32;  // keys per lane
      const int C = (n + NW - 1) / NW;
      const int c0 = warp * C;
      unsigned long long kj[MJ];
#pragma unroll
      for (int m = 0; m < MJ; ++m) kj[m] = lane + 32 * m < n ? keysA[lane + 32 * m] : 0ull;  // 0 is below every key
      uint32_t wmask = 0;
      for (int c = 0; c < C && c0 + c < n; ++c) {
        const unsigned long long ki = keysA[c0 + c];
        int cnt = 0;
#pragma unroll
        for (int m = 0; m < MJ; ++m) cnt += (int)(kj[m] > ki);
        if (k >= n || __reduce_add_sync(0xffffffffu, cnt) < k) wmask |= 1u << c;
      }
      if (lane == 0) s_wmask[warp] = wmask;
      __syncthreads();
      // kept before this warp, kept in total, and the last kept candidate
      const int cw = lane < NW ? __popc(s_wmask[lane]) : 0;
      int incl = cw;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      const int before = __shfl_sync(0xffffffffu, incl - cw, warp);
      const int total = __shfl_sync(0xffffffffu, incl, 31);
      const unsigned has = __ballot_sync(0xffffffffu, cw > 0);
      int nn = 0;
      if (l > 0 && total > 0) {
        const int wl = 31 - __clz(has);
        const int last = cand_id(keysA[wl * C + 31 - __clz(s_wmask[wl])]);
        nn = (total - 1) * f + min(f, nC - last * f);
      }
      const bool fits = l == 0 || nn <= MC;
      for (uint32_t mk = wmask; mk != 0 && fits; mk &= mk - 1) {
        const int c = __ffs(mk) - 1;
        const int pos = before + __popc(wmask & ((1u << c) - 1u));
        const int i = c0 + c;
        const int id = cand_id(keysA[i]);
        if (l == 0) {
          if (lane == 0 && pos < p.sel_cap) out[pos] = id;
        } else {
          for (int j = lane; j < f; j += 32) {
            const int cid = id * f + j;
            if (cid < nC) keysB[pos * f + j] = have_child ? cand_key(cs[i * f + j], cid) : cand_key(0u, cid);
          }
        }
      }
      nk = total;
      if (l == 0) break;
      if (!fits) {
        overflow = true;
        break;
      }
      need_score = !have_child;
      have_child = false;
      n = nn;
      __syncthreads();
      unsigned long long* t = keysA;
      keysA = keysB;
      keysB = t;
      continue;
    }

    // 1. mark[i] = candidate i is among the k largest keys
    if (k >= n) {
      for (int i = tid; i < n; i += NT) mark[i] = 1;
    } else if (n <= kRankMax) {
      int ncp = 1, sh = 0;
      while (ncp < n) ncp <<= 1;
      int tpc = NT / ncp;  // threads per candidate, a power of two
      tpc = tpc < 1 ? 1 : (tpc > 32 ? 32 : tpc);
      while ((1 << sh) < tpc) ++sh;
      const int work = n * tpc;
      const int work32 = (work + 31) & ~31;  // whole warps, so the shuffles see every lane
      for (int x = tid; x < work32; x += NT) {
        const int i = x >> sh, t = x & (tpc - 1);
        int rank = 0;
        if (x < work) {
          const unsigned long long ki = keysA[i];
          int j = t;
          for (; j + 3 * tpc < n; j += 4 * tpc) {
            const unsigned long long a0 = keysA[j], a1 = keysA[j + tpc], a2 = keysA[j + 2 * tpc], a3 = keysA[j + 3 * tpc];
            rank += (int)(a0 > ki) + (int)(a1 > ki) + (int)(a2 > ki) + (int)(a3 > ki);
          }
          for (; j < n; j += tpc) rank += keysA[j] > ki;
        }
        for (int o = tpc >> 1; o > 0; o >>= 1) rank += __shfl_xor_sync(0xffffffffu, rank, o);
        if (x < work && t == 0) mark[i] = rank < k;
      }
    } else {
      // bitonic sort (descending) of a copy of the keys gives the k-th key
      int P = 1;
      while (P < n) P <<= 1;
      for (int i = tid; i < P; i += NT) keysB[i] = i < n ? keysA[i] : 0ull;
      __syncthreads();
      for (int kk = 2; kk <= P; kk <<= 1) {
        for (int j = kk >> 1; j > 0; j >>= 1) {
          for (int i = tid; i < P; i += NT) {
            const int ixj = i ^ j;
            if (ixj > i) {
              const unsigned long long a = keysB[i], bb = keysB[ixj];
              const bool desc = (i & kk) == 0;
              if (desc ? (a < bb) : (a > bb)) {
                keysB[i] = bb;
                keysB[ixj] = a;
              }
            }
          }
          __syncthreads();
        }
      }
      const unsigned long long thr = keysB[k - 1];
      for (int i = tid; i < n; i += NT) mark[i] = keysA[i] >= thr;
    }
    __syncthreads();

    // 2. order-preserving compaction of the kept positions (warp 0)
    if (warp == 0) {
      const unsigned lt = (1u << lane) - 1u;
      int nkw = 0;
      for (int i0 = 0; i0 < n; i0 += 128) {
        bool fl4[4];
        unsigned bal[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) fl4[c] = i0 + 32 * c + lane < n && mark[i0 + 32 * c + lane] != 0;
#pragma unroll
        for (int c = 0; c < 4; ++c) bal[c] = __ballot_sync(0xffffffffu, fl4[c]);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          if (fl4[c]) {
            const int pos = nkw + __popc(bal[c] & lt);
            kept[pos] = i0 + 32 * c + lane;
            if (l == 0 && pos < p.sel_cap) out[pos] = cand_id(keysA[i0 + 32 * c + lane]);
          }
          nkw += __popc(bal[c]);
        }
      }
      __syncwarp();
      if (lane == 0) {
        s_nk = nkw;
        // children of the kept clusters: all full except possibly the last
        // cluster of the level, which can only be the last kept one
        int nxt = 0;
        if (l > 0 && nkw > 0) {
          const int last = cand_id(keysA[kept[nkw - 1]]);
          nxt = (nkw - 1) * f + min(f, nC - last * f);
        }
        s_next = nxt;
      }
    }
    __syncthreads();
    nk = s_nk;
    if (l == 0) break;

    // 3. the next level's candidates: children of the kept clusters, in order
    const int nn = s_next;
    if (nn > MC) {
      overflow = true;
      break;
    }
    for (int x = tid; x < nn; x += NT) {
      const int kk = x / f, j = x - kk * f;
      const int i = kept[kk];
      const int id = cand_id(keysA[i]) * f + j;
      keysB[x] = have_child ? cand_key(cs[i * f + j], id) : cand_key(0u, id);
    }
    need_score = !have_child;
    have_child = false;
    n = nn;
    __syncthreads();
    unsigned long long* t = keysA;
    keysA = keysB;
    keysB = t;
  }
  if (overflow || timed_out || nk > p.sel_cap) {
    if (tid == 0) atomicOr(&g_mpc_status, 4);
    nk = 0;
  }
  for (int i = tid; i < p.sel_cap; i += NT)
    if (i >= nk) out[i] = -1;
  if (tid == 0 && h == 0 && ri == 0) p.out_n_sel[b] = nk;
}

// Threads per CTA: 16 warps while the units fit one wave of SMs, 8 while
// they fit two CTAs per SM, else 4 (six CTAs per SM).
static int select_threads(int units) { return units <= 152 ? 512 : (units <= 304 ? 256 : 128); }
int select_threads_of(int units) { return select_threads(units); }

int select_smem_bytes(int D, int max_cand, int row_buf, int n_src) {
  return (int)SelLayout(D, max_cand, row_buf, n_src).total;
}

// Scoring the whole level below the coarsest in the first round saves a
// dependent round but reads the children of unkept clusters too: worth it
// while the units fit two CTAs per SM (latency-bound), not beyond.
int select_spec_first(int units) { return units <= 2 * 152 ? 1 : 0; }

template <typename K>
static cudaError_t launch_sel(K kernel, int units, int nt, int smem, cudaStream_t st, const SelectParams& p) {
  cudaError_t e = ensure_dyn_smem((const void*)kernel, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(kernel, dim3(units), dim3(nt), smem, st, p);
}

cudaError_t launch_select(const SelectParams& p, int dtype, int D, int units, cudaStream_t st) {
  const int smem = select_smem_bytes(D, p.max_cand, p.row_buf, select_n_src(p.metric));
  // the fixed-point metric is a diagnostic path: one thread count
  const int nt = p.metric == MPC_SIM_FXP ? 256 : select_threads(units);
#define MPC_SEL(TT, DD)                                                                            \
  if (D == DD) {                                                                                   \
    if (p.metric == MPC_SIM_FXP) return launch_sel(select_kernel<TT, DD, 256, true>, units, nt, smem, st, p); \
    if (nt == 512) return launch_sel(select_kernel<TT, DD, 512, false>, units, nt, smem, st, p);  \
    if (nt == 256) return launch_sel(select_kernel<TT, DD, 256, false>, units, nt, smem, st, p);  \
    return launch_sel(select_kernel<TT, DD, 128, false>, units, nt, smem, st, p);                 \
  }
  if (dtype == MPC_BF16) {
    MPC_SEL(bf16, 64)
    MPC_SEL(bf16, 128)
  } else {
    MPC_SEL(float, 64)
    MPC_SEL(float, 128)
  }
#undef MPC_SEL
  return cudaErrorInvalidValue;
}

int take_status_select() { return take_status(); }

}  // namespace mpc
