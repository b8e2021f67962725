// One whole decode step in one persistent launch (Alg. 2 Step 2): the
// hierarchical cluster selection of the leader layers (Sec. 3.3-3.4, Eq. 3;
// Alg. 2 Sim + topk) and, for every layer, the decode append and the sparse
// attention over the selected clusters and the tail (Alg. 1; App. A).
//
// Work items, claimed from two global counters, in this order:
//   1. selection units (leader ref, sequence b, kv head h).  A team of warps
//      of one CTA walks the unit's summary pyramid from the coarsest level
//      down (the same scores and ranking as mpc_select), writes the selected
//      ids and publishes them with a release store of the unit's ready flag;
//   2. attention chunks.  The rows a unit (ref, b, h) attends are listed
//      tail first (the rows after the last sealed cluster, then the row
//      appended now), padded to a whole 16-row tile, then the s rows of every
//      selected cluster; a chunk is up to CT consecutive tiles of one unit.
//      A warp claims chunks one at a time and streams their tiles through its
//      own ring of shared-memory stages (cp.async, one commit group per
//      tile), NST tiles ahead of its compute.
// A chunk waits for its group's ready flag only before it issues selected
// rows (bounded, 1 s), so tail tiles stream while the selection runs.  Every
// selection unit is claimed before any chunk, by a CTA that is running and
// never waits on another, so every such wait ends without assuming that the
// CTAs are co-resident.
// A unit cut into several chunks is merged by the last of its chunks to
// finish (a ticket on the unit's counter; nobody waits): every chunk writes a
// (max, sum, o) record, and the chunk that draws the last ticket folds the
// unit's records by log-sum-exp and writes o.  The tile arithmetic is the
// persistent attention kernel's (mma.sync m16n8k16, the GQA group's heads as
// N, P split into bf16 hi + lo).
#include <mutex>

#include "kernels.cuh"
#include "seal.cuh"
#include "sel_score.cuh"

namespace mpc {
namespace {

constexpr int kSelIds = kStepSelIds;  // selected ids a warp stages for the chunk it issues
constexpr int kCQ = 8;            // chunks between a warp's issue side and its compute side
constexpr int kMaxStepCtas = kStepCtasMax;
// control words of the workspace
constexpr int kCtlSelClaim = 0, kCtlAttClaim = 1, kCtlGrid = 2, kCtlEpoch = 3, kCtlAbort = 4;

__device__ __forceinline__ void named_bar(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}
__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* a) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(a) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_u32(unsigned* a, unsigned v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(a), "r"(v) : "memory");
}
__device__ __forceinline__ int atom_add_acq_rel(int* a, int v) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(a), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}

}  // namespace

// Shared memory of one CTA: per warp a ring of NST stages (K tile, V tile,
// the chunk's queries), the swizzle keys and metadata of its stages, the
// selected ids of the chunk it issues and its chunk queue; per team its
// scalars; the per-sequence table.  A selection team borrows its warps' rings
// as scratch (TeamLayout) before they stream.
template <int D>
struct StepSmem {
  static constexpr int ROWB = D * 2;
  static constexpr int TILEB = 16 * ROWB;
  static __host__ __device__ constexpr int qbytes(int G) { return ((G * D * 2 + 127) / 128) * 128; }
  static __host__ __device__ constexpr int stage(int G) { return 2 * TILEB + qbytes(G); }
  static __host__ __device__ constexpr int keys_off(int G, int nst, int wpc) { return wpc * nst * stage(G); }
  static __host__ __device__ constexpr int meta_off(int G, int nst, int wpc) { return keys_off(G, nst, wpc) + wpc * nst * 16; }
  static __host__ __device__ constexpr int selb_off(int G, int nst, int wpc) { return meta_off(G, nst, wpc) + wpc * nst * 4; }
  static __host__ __device__ constexpr int cq_off(int G, int nst, int wpc) { return selb_off(G, nst, wpc) + wpc * kSelIds * 4; }
  static __host__ __device__ constexpr int team_off(int G, int nst, int wpc) { return cq_off(G, nst, wpc) + wpc * kCQ * 8; }
  static __host__ __device__ constexpr int tab_off(int G, int nst, int wpc) { return team_off(G, nst, wpc) + wpc * 16; }
  static __host__ __device__ constexpr int total(int G, int nst, int wpc, int B) { return tab_off(G, nst, wpc) + (4 * B + 4) * 4; }
};

// Scratch of one selection team inside its warps' rings: the summed query,
// two candidate-key arrays, the first round's child scores, kept marks and
// positions, then the staged summary rows (n_src arrays of RB rows).
struct TeamLayout {
  int keysA, keysB, cs, mark, kept, rows, total;
  __host__ __device__ TeamLayout(int D, int MC, int RB, int n_src) {
    keysA = D * 4;
    keysB = keysA + MC * 8;
    cs = keysB + MC * 8;
    mark = cs + ((RB * 4 + 15) & ~15);
    kept = mark + MC * 4;
    rows = (kept + MC * 4 + 15) & ~15;
    total = rows + n_src * RB * D * 4;
  }
};

template <int D, int HN, int NST, int WPC>
__global__ void __launch_bounds__(WPC * 32, 1) decode_step_kernel(const __grid_constant__ StepParams sp) {
  using S = StepSmem<D>;
  constexpr int ROWB = S::ROWB;
  constexpr int TILEB = S::TILEB;
  constexpr int KS = D / 16;     // k-steps of S^T and m-tiles of O^T
  constexpr int CH = ROWB / 16;  // 16-byte chunks per K / V row
  const AttnParams& p = sp.a;
  extern __shared__ __align__(128) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = p.G, B = p.B, Hkv = p.Hkv, s = p.pyr.s, CT = sp.chunk_tiles;
  const int STAGE = S::stage(G);
  uint8_t* ring = smem + warp * NST * STAGE;
  int8_t* keys = reinterpret_cast<int8_t*>(smem + S::keys_off(G, NST, WPC)) + warp * NST * 16;
  int* meta = reinterpret_cast<int*>(smem + S::meta_off(G, NST, WPC)) + warp * NST;
  int* selb = reinterpret_cast<int*>(smem + S::selb_off(G, NST, WPC)) + warp * kSelIds;
  int2* cq = reinterpret_cast<int2*>(smem + S::cq_off(G, NST, WPC)) + warp * kCQ;
  int* s_team = reinterpret_cast<int*>(smem + S::team_off(G, NST, WPC));
  int* s_n = reinterpret_cast<int*>(smem + S::tab_off(G, NST, WPC));  // cache rows before the append, -1 refused
  int* s_nch = s_n + B;    // chunks per unit of sequence b
  int* s_k1 = s_nch + B;   // selected clusters: upper bound (selection in this call) or the caller's count
  int* s_pre = s_k1 + B;   // exclusive prefix of s_nch (B + 1)
  int* s_misc = s_pre + B + 1;
  const bool sel_in_call = sp.n_sel_units > 0;
  grid_dep_launch();
  grid_dep_wait();

  // ---- per-sequence table
  if (warp == 0) {
    int carry = 0;
    for (int b0 = 0; b0 < B; b0 += 32) {
      const int b = b0 + lane;
      int n = -1, nch = 0, k1 = 0;
      if (b < B) {
        const int nt = p.n_tok[b];
        const int ns = (!sel_in_call && p.sel_cap > 0) ? p.n_sel[b] : 0;
        if (nt < 0 || nt + 1 > p.cap_tokens) {
          atomicOr(&g_mpc_status, 2);  // no room for the append: skip the sequence
        } else {
          n = nt;
          const int C1 = n / s, tail = n - C1 * s, tt = (tail + 16) >> 4;
          if (p.sel_cap > 0)
            k1 = sel_in_call ? min(count_from_ppm(C1, sp.keep_ppm[0]), min(C1, p.sel_cap))
                             : max(0, min(ns, min(C1, p.sel_cap)));
          const int ntm = tt + (k1 * s + 15) / 16;
          nch = (ntm + CT - 1) / CT;
        }
      }
      int incl = nch;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      if (b < B) {
        s_n[b] = n;
        s_nch[b] = nch;
        s_k1[b] = k1;
        s_pre[b] = carry + incl - nch;
      }
      carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) {
      s_pre[B] = carry;
      s_misc[0] = (int)((unsigned)__ldcg(&sp.ctl[kCtlEpoch]) + 1u);
    }
  }
  __syncthreads();
  const unsigned want = (unsigned)s_misc[0];  // value of a ready flag published in this call

  // ================================================= selection teams ====
  if (sel_in_call) {
    const int TW = sp.team_warps, NTT = TW * 32;
    const int team = warp / TW, twarp = warp - team * TW;
    const int tl = threadIdx.x - team * NTT;
    const int MC = sp.max_cand, RB = sp.row_buf, NSRC = sp.n_src;
    const TeamLayout TL(D, MC, RB, NSRC);
    uint8_t* treg = smem + (size_t)team * TW * NST * STAGE;
    float* qsum = reinterpret_cast<float*>(treg);
    unsigned long long* const kA0 = reinterpret_cast<unsigned long long*>(treg + TL.keysA);
    unsigned long long* const kB0 = reinterpret_cast<unsigned long long*>(treg + TL.keysB);
    uint32_t* cs = reinterpret_cast<uint32_t*>(treg + TL.cs);
    int* mark = reinterpret_cast<int*>(treg + TL.mark);
    int* kept = reinterpret_cast<int*>(treg + TL.kept);
    float* rows = reinterpret_cast<float*>(treg + TL.rows);
    float* rows2 = rows + (size_t)RB * D;
    int* tsc = s_team + team * 4;
    auto tsync = [&]() {
      if (TW == 1) __syncwarp();
      else named_bar(1 + team, NTT);
    };
    const int top = p.pyr.n_levels - 1;
    constexpr int CPR = D * 4 / 16;  // 16-byte pieces per summary row

    // similarity of staged rows [0, nrows); put(r, orderable score) runs on
    // one lane per row (row_partial: the arithmetic of mpc_select)
    auto score = [&](int nrows, auto&& put) {
      constexpr int V4 = D / 16;
      const int ql = lane & 3, rs = lane >> 2, rot = rs & 1;
      float4 qv[V4];
#pragma unroll
      for (int jj = 0; jj < V4; ++jj) qv[jj] = reinterpret_cast<const float4*>(qsum)[ql + 4 * jj];
      for (int r0 = twarp * 8; r0 < nrows; r0 += TW * 8) {
        const int r = r0 + rs;
        float a = 0.f;
        if (r < nrows)
          a = NSRC == 1 ? row_partial<D, false>(rows + (size_t)r * D, nullptr, qv, ql, rot)
                        : row_partial<D, true>(rows + (size_t)r * D, rows2 + (size_t)r * D, qv, ql, rot);
        a += __shfl_xor_sync(0xffffffffu, a, 1);
        a += __shfl_xor_sync(0xffffffffu, a, 2);
        if (ql == 0 && r < nrows) put(r, orderable(a));
      }
    };
    // mark[i] = candidate i is among the k largest keys (fewer than k larger)
    auto rank_mark = [&](const unsigned long long* ka, int nc, int k) {
      if (k >= nc) {
        for (int i = tl; i < nc; i += NTT) mark[i] = 1;
        return;
      }
      int tpc = 1, sh = 0;  // threads per candidate
      while (tpc < 32 && tpc * 2 * nc <= NTT) {
        tpc <<= 1;
        ++sh;
      }
      const int work = nc << sh, work32 = (work + 31) & ~31;
      for (int x = tl; x < work32; x += NTT) {
        const int i = x >> sh, t = x & (tpc - 1);
        int cnt = 0;
        if (x < work) {
          const unsigned long long ki = ka[i];
          int j = t;
          for (; j + 3 * tpc < nc; j += 4 * tpc)
            cnt += (int)(ka[j] > ki) + (int)(ka[j + tpc] > ki) + (int)(ka[j + 2 * tpc] > ki) + (int)(ka[j + 3 * tpc] > ki);
          for (; j < nc; j += tpc) cnt += (int)(ka[j] > ki);
        }
        for (int o = tpc >> 1; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
        if (x < work && t == 0) mark[i] = cnt < k;
      }
    };

    while (true) {
      if (tl == 0) tsc[0] = atomicAdd(&sp.ctl[kCtlSelClaim], 1);
      tsync();
      const int su = tsc[0];
      if (su >= sp.n_sel_units) break;
      const int ril = su / (B * Hkv), b = (su / Hkv) % B, h = su % Hkv;
      const int ri = sp.lead_ref[ril];
      const int layer = p.refs.layer[ri], group = p.refs.group[ri];
      const int n = s_n[b];
      int C[kMaxLevels];
      level_counts(p.pyr, n > 0 ? n : 0, C);
      const int64_t uoff = ((int64_t)(group * B + b) * Hkv + h) * p.pyr.rows * D;
      const float* srcA = sp.src0 + uoff;
      const float* srcB = (NSRC == 2 ? sp.src1 : sp.src0) + uoff;
      int* out = sp.sel_out + ((int64_t)(group * B + b) * Hkv + h) * p.sel_cap;
      bool bad = n >= 0 && (C[0] > p.pyr.cap[0] || C[top] > MC);
      int nk = 0;
      unsigned long long* kA = kA0;
      unsigned long long* kB = kB0;
      if (n >= 0 && !bad && C[0] > 0 && p.sel_cap > 0) {
        // first round: the live rows of the coarsest level and, when they
        // fit with it, all live rows of the level below (scored now, so that
        // level needs no round of its own)
        const int nT = C[top];
        const int nC1 = top > 0 ? C[top - 1] : 0;
        const bool spec = sp.spec && top > 0 && nT + nC1 <= RB;
        const int own = nT < RB ? nT : RB;
        const int64_t offT = (int64_t)p.pyr.off[top] * D;
        const int64_t offC = (int64_t)(top > 0 ? p.pyr.off[top - 1] : 0) * D;
        for (int c = tl; c < own * CPR; c += NTT) {
          cp_async16(rows + c * 4, srcA + offT + c * 4);
          if (NSRC == 2) cp_async16(rows2 + c * 4, srcB + offT + c * 4);
        }
        if (spec)
          for (int c = tl; c < nC1 * CPR; c += NTT) {
            cp_async16(rows + (size_t)nT * D + c * 4, srcA + offC + c * 4);
            if (NSRC == 2) cp_async16(rows2 + (size_t)nT * D + c * 4, srcB + offC + c * 4);
          }
        cp_async_commit();
        // q_sum = sum over the group's query heads (Eq. 3 is linear in q)
        const bf16* qp = (const bf16*)p.q + layer * p.q_ls + ((int64_t)b * p.Hq + h * G) * D;
        for (int c = tl; c < D; c += NTT) {
          float acc = 0.f;
          for (int g = 0; g < G; ++g) acc += __bfloat162float(qp[g * D + c]);
          qsum[c] = acc;
        }
        cp_async_wait<0>();
        tsync();
        score(spec ? nT + nC1 : own, [&](int r, uint32_t sc) {
          if (r < own) kA[r] = cand_key(sc, r);
          else cs[r - nT] = sc;
        });
        tsync();
        for (int x0 = own; x0 < nT; x0 += RB) {  // the rest of a coarsest level larger than the buffer
          const int nb = min(RB, nT - x0);
          for (int c = tl; c < nb * CPR; c += NTT) {
            cp_async16(rows + c * 4, srcA + offT + (int64_t)x0 * D + c * 4);
            if (NSRC == 2) cp_async16(rows2 + c * 4, srcB + offT + (int64_t)x0 * D + c * 4);
          }
          cp_async_commit();
          cp_async_wait<0>();
          tsync();
          score(nb, [&](int r, uint32_t sc) { kA[x0 + r] = cand_key(sc, x0 + r); });
          tsync();
        }
        bool have_child = spec, need_score = false;
        int nc = nT;
        for (int l = top; l >= 0; --l) {
          const int f = l > 0 ? p.pyr.fanout[l - 1] : 1;
          const int nCl = l > 0 ? C[l - 1] : 0;
          if (need_score) {
            // a round over the candidates' own rows (runs of children of the
            // kept clusters), in batches of RB rows
            const int64_t offL = (int64_t)p.pyr.off[l] * D;
            for (int x0 = 0; x0 < nc; x0 += RB) {
              const int x1 = min(nc, x0 + RB);
              for (int c = tl; c < (x1 - x0) * CPR; c += NTT) {
                const int r = c / CPR, part = c - r * CPR;
                const int64_t srow = offL + (int64_t)cand_id(kA[x0 + r]) * D + part * 4;
                cp_async16(rows + (size_t)r * D + part * 4, srcA + srow);
                if (NSRC == 2) cp_async16(rows2 + (size_t)r * D + part * 4, srcB + srow);
              }
              cp_async_commit();
              cp_async_wait<0>();
              tsync();
              score(x1 - x0, [&](int r, uint32_t sc) { kA[x0 + r] = cand_key(sc, cand_id(kA[x0 + r])); });
              tsync();
            }
          }
          rank_mark(kA, nc, min(count_from_ppm(C[l], sp.keep_ppm[l]), nc));
          tsync();
          // order-preserving compaction of the kept candidates (ids stay ascending)
          if (twarp == 0) {
            const unsigned lt = (1u << lane) - 1u;
            int nkw = 0;
            for (int i0 = 0; i0 < nc; i0 += 32) {
              const bool fl = i0 + lane < nc && mark[i0 + lane] != 0;
              const unsigned bal = __ballot_sync(0xffffffffu, fl);
              if (fl) kept[nkw + __popc(bal & lt)] = i0 + lane;
              nkw += __popc(bal);
            }
            __syncwarp();
            if (lane == 0) {
              // children of the kept clusters: all full except possibly those
              // of the level's last cluster, which is the last kept one
              int nn = 0;
              if (l > 0 && nkw > 0) {
                const int last = cand_id(kA[kept[nkw - 1]]);
                nn = (nkw - 1) * f + min(f, nCl - last * f);
              }
              tsc[1] = nkw;
              tsc[2] = nn;
            }
          }
          tsync();
          nk = tsc[1];
          if (l == 0) break;
          const int nn = tsc[2];
          if (nn > MC) {
            bad = true;
            break;
          }
          for (int x = tl; x < nn; x += NTT) {
            const int kk = x / f, j = x - kk * f;
            const int id = cand_id(kA[kept[kk]]) * f + j;
            kB[x] = have_child ? cand_key(cs[id], id) : cand_key(0u, id);
          }
          tsync();
          unsigned long long* t = kA;
          kA = kB;
          kB = t;
          nc = nn;
          need_score = !have_child;
          have_child = false;
        }
      }
      if (bad || nk > p.sel_cap) {
        if (tl == 0) atomicOr(&g_mpc_status, 4);
        nk = 0;
      }
      for (int pos = tl; pos < p.sel_cap; pos += NTT) out[pos] = pos < nk ? cand_id(kA[kept[pos]]) : -1;
      if (tl == 0) {
        sp.sel_cnt[su] = nk;
        if (ril == 0 && h == 0) sp.n_sel_out[b] = nk;
      }
      tsync();
      if (tl == 0) {
        __threadfence();
        st_release_u32(&sp.ready[su], want);
      }
    }
  }

  // ================================================ attention chunks ====
  const bool fast = (s & 15) == 0;  // every selected tile is one run of consecutive cache rows
  const int64_t TPR = (int64_t)Hkv * s_pre[B];
  const int64_t NCH = TPR * p.n_refs;

  struct Geo {
    int x, ri, b, h, c, n, C1, tail, tt, t0, t1, k1, nne, su;
  };
  // chunk x of the call: unit (ri, b, h), its rows and tiles; k1 = selected
  // clusters if known, else -1
  auto geo_of = [&](int x, int k1) {
    Geo g;
    g.x = x;
    g.ri = (int)(x / TPR);
    const int64_t rem = x - (int64_t)g.ri * TPR;
    int lo = 0, hi = B - 1;  // largest b with Hkv * pre[b] <= rem
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if ((int64_t)Hkv * s_pre[mid] <= rem) lo = mid;
      else hi = mid - 1;
    }
    g.b = lo;
    const int64_t rem2 = rem - (int64_t)Hkv * s_pre[lo];
    const int nch = s_nch[lo];
    g.h = (int)(rem2 / nch);
    g.c = (int)(rem2 - (int64_t)g.h * nch);
    g.n = s_n[lo];
    g.C1 = g.n / s;
    g.tail = g.n - g.C1 * s;
    g.tt = (g.tail + 16) >> 4;  // tail tiles: the tail rows and the appended row
    const int ntm = g.tt + (s_k1[lo] * s + 15) / 16;
    g.t0 = g.c * CT;
    g.t1 = min(g.t0 + CT, ntm);
    const int li = sel_in_call ? sp.lead_of[g.ri] : -1;
    g.su = li >= 0 ? (li * B + g.b) * Hkv + g.h : -1;
    if (g.su < 0) k1 = s_k1[lo];  // selections are the caller's
    g.k1 = k1;
    g.nne = -1;
    if (k1 >= 0) {
      const int nt = g.tt + (k1 * s + 15) / 16;
      g.t1 = min(g.t1, nt);
      g.nne = (nt + CT - 1) / CT;  // chunks of the unit that hold tiles
    }
    return g;
  };
  bool abort = false;
  // waits (bounded) for the ready flag of selection unit su
  auto wait_ready = [&](int su) -> bool {
    int ok = 1;
    if (lane == 0 && ld_acquire_u32(&sp.ready[su]) != want) {
      const uint64_t t0 = global_timer_ns();
      while (ld_acquire_u32(&sp.ready[su]) != want) {
        if (global_timer_ns() - t0 > 1000000000ull) {
          atomicOr(&g_mpc_status, kStatusWaitTimeout);
          atomicExch(&sp.ctl[kCtlAbort], 1);
          ok = 0;
          break;
        }
        __nanosleep(64);
      }
    }
    ok = __shfl_sync(0xffffffffu, ok, 0);
    __syncwarp();
    return ok != 0;
  };

  // ---- issue side
  int pend = 0;  // claim in flight (lane 0)
  if (lane == 0) pend = atomicAdd(&sp.ctl[kCtlAttClaim], 1);
  Geo gi;
  gi.t0 = gi.t1 = 0;
  int it = 0, ci0 = 0, seq_i = 0, cq_push = 0;
  bool idone = false;

  // moves the issue side to the next chunk that holds tiles; false once the
  // claims run out (or a wait gave up)
  auto next_chunk = [&]() -> bool {
    while (true) {
      const int x = __shfl_sync(0xffffffffu, pend, 0);
      if ((int64_t)x >= NCH) return false;
      if (lane == 0) pend = atomicAdd(&sp.ctl[kCtlAttClaim], 1);  // the next claim, ahead of need
      Geo g = geo_of(x, -1);
      if (g.su >= 0 && g.t1 > g.tt) {
        if (!wait_ready(g.su)) {
          abort = true;
          return false;
        }
        g = geo_of(x, __ldcg(&sp.sel_cnt[g.su]));
      }
      if (g.t0 >= g.t1) continue;  // past the unit's last selected tile
      if (g.t1 > g.tt) {
        // the selected ids this chunk's tiles read
        const int a_lo = 16 * (max(g.t0, g.tt) - g.tt);
        const int a_hi = min(16 * (g.t1 - g.tt), g.k1 * s);
        ci0 = a_lo / s;
        const int nci = (a_hi - 1) / s + 1 - ci0;
        const int* srow = p.sel + ((int64_t)(p.refs.group[g.ri] * B + g.b) * Hkv + g.h) * p.sel_cap;
        for (int i = lane; i < nci; i += 32) {
          int id = __ldcg(srow + ci0 + i);
          if (id < 0 || id >= g.C1) {  // corrupt input: reported, read as cluster 0
            atomicOr(&g_mpc_status, 4);
            id = 0;
          }
          selb[i] = id;
        }
        __syncwarp();
      }
      if (lane == 0) cq[cq_push % kCQ] = make_int2(x, g.k1);
      ++cq_push;
      gi = g;
      it = g.t0;
      return true;
    }
  };
  auto kv_off = [&](const Geo& g) {
    return (int64_t)p.refs.layer[g.ri] * p.cache_ls + (int64_t)(g.b * Hkv + g.h) * p.cap_tokens * D;
  };
  // issues the next tile into its stage; false when there is none
  auto issue_one = [&]() -> bool {
    if (it >= gi.t1 && !next_chunk()) return false;
    const int t = it++;
    const int slot = seq_i % NST;
    uint8_t* sK = ring + slot * STAGE;
    uint8_t* sV = sK + TILEB;
    const int64_t co = kv_off(gi);
    const uint8_t* kb = reinterpret_cast<const uint8_t*>((const bf16*)p.kc + co);
    const uint8_t* vb = reinterpret_cast<const uint8_t*>((const bf16*)p.vc + co);
    int nv, cur = -1;
    if (t < gi.tt) {
      // tail rows (consecutive in the cache) and the appended row's slot
      const int a0 = 16 * t;
      const int ncache = max(0, min(16, gi.tail - a0));
      nv = min(16, gi.tail + 1 - a0);
      if (gi.tail >= a0 && gi.tail < a0 + 16) cur = gi.tail - a0;
      const int row0 = gi.C1 * s + a0;
      if (!fast && lane < 16) keys[slot * 16 + lane] = (int8_t)((row0 + lane) & 7);
      const uint8_t* gk = kb + (int64_t)row0 * ROWB;
      const uint8_t* gv = vb + (int64_t)row0 * ROWB;
      for (int i = lane; i < ncache * CH; i += 32) {
        cp_async16(sK + i * 16, gk + i * 16);
        cp_async16(sV + i * 16, gv + i * 16);
      }
    } else {
      const int a0 = 16 * (t - gi.tt);
      nv = min(16, gi.k1 * s - a0);
      if (fast) {
        const int ci = a0 / s;
        const int src0 = selb[ci - ci0] * s + (a0 - ci * s);
        const uint8_t* gk = kb + (int64_t)src0 * ROWB;
        const uint8_t* gv = vb + (int64_t)src0 * ROWB;
        for (int i = lane; i < 16 * CH; i += 32) {
          cp_async16(sK + i * 16, gk + i * 16);
          cp_async16(sV + i * 16, gv + i * 16);
        }
      } else {
        const int r = lane & 15, a = a0 + r;
        int src = 0;
        if (r < nv) {
          const int ci = a / s;
          src = selb[ci - ci0] * s + (a - ci * s);
        }
        if (lane < 16) keys[slot * 16 + r] = (int8_t)((r < nv) ? (src & 7) : (r & 7));
#pragma unroll 4
        for (int i = lane; i < 16 * CH; i += 32) {
          const int row = i / CH, ch = i - row * CH;
          const int srow = __shfl_sync(0xffffffffu, src, row);
          if (row < nv) {
            cp_async16(sK + i * 16, kb + (int64_t)srow * ROWB + ch * 16);
            cp_async16(sV + i * 16, vb + (int64_t)srow * ROWB + ch * 16);
          }
        }
      }
    }
    const bool first = t == gi.t0, last = t == gi.t1 - 1;
    if (first) {  // the unit's queries ride with the chunk's first tile
      const uint8_t* q = reinterpret_cast<const uint8_t*>((const bf16*)p.q + p.refs.layer[gi.ri] * p.q_ls +
                                                          ((int64_t)gi.b * p.Hq + gi.h * G) * D);
      for (int i = lane; i < G * D * 2 / 16; i += 32) cp_async16(sK + 2 * TILEB + i * 16, q + i * 16);
    }
    if (lane == 0) meta[slot] = nv | ((cur + 1) << 5) | (first ? 1 << 10 : 0) | (last ? 1 << 11 : 0);
    ++seq_i;
    return true;
  };

  // ---- compute side
  uint32_t qb[HN][KS][2];  // Q^T operand: k = channels, n = heads
  float o[KS][HN][4];      // O^T accumulators: m = channels, n = heads
  float m_run[HN][2], l_run[HN][2];
  Geo gc;
  gc.x = 0;
  int seq_c = 0, cq_pop = 0;
  const int r_tok = lane >> 2;       // token row of S^T (and +8)
  const int h_off = 2 * (lane & 3);  // first of this thread's two heads in an n-tile

  // folds the unit's nr records (from R0 on) by log-sum-exp and writes o
  auto merge_records = [&](const float* R0, int nr, float* outp) {
    const int REC = G * (D + 4);
    constexpr int D4 = D / 4;
    for (int q4 = lane; q4 < G * D4; q4 += 32) {
      const int g = q4 / D4, c4 = q4 - g * D4;
      const float* base = R0 + g * (D + 4);
      float M = kNegInf;
#pragma unroll 4
      for (int k = 0; k < nr; ++k) M = fmaxf(M, __ldcg(base + (int64_t)k * REC));
      float L = 0.f;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
      for (int k = 0; k < nr; ++k) {
        const float* rk = base + (int64_t)k * REC;
        const float m = __ldcg(rk);
        const float w = (m == kNegInf) ? 0.f : fast_exp2(m - M);
        L = fmaf(w, __ldcg(rk + 1), L);
        const float4 v = __ldcg(reinterpret_cast<const float4*>(rk + 4) + c4);
        acc.x = fmaf(w, v.x, acc.x);
        acc.y = fmaf(w, v.y, acc.y);
        acc.z = fmaf(w, v.z, acc.z);
        acc.w = fmaf(w, v.w, acc.w);
      }
      const float inv = 1.f / L;
      float* op = outp + g * D + 4 * c4;
      op[0] = acc.x * inv;
      op[1] = acc.y * inv;
      op[2] = acc.z * inv;
      op[3] = acc.w * inv;
    }
  };

  // end of chunk gc: write o, or the chunk's record and a ticket (the last
  // ticket merges); the chunk that holds the appended row seals a full tail
  auto flush = [&]() {
    if (gc.k1 < 0) {  // tail tiles only: the selected count is needed now
      if (!wait_ready(gc.su)) {
        abort = true;
        return;
      }
      gc = geo_of(gc.x, __ldcg(&sp.sel_cnt[gc.su]));
    }
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
    float* outp = p.out + p.refs.layer[gc.ri] * p.out_ls + ((int64_t)gc.b * p.Hq + gc.h * G) * D;
    if (gc.nne <= 1) {
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
    } else {
      const int REC = G * (D + 4);
      float* dst = p.part + (int64_t)gc.x * REC;
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
      const int64_t uid = ((int64_t)gc.ri * B + gc.b) * Hkv + gc.h;
      int t = 0;
      if (lane == 0) t = atom_add_acq_rel(&p.unit_counter[uid], 1);
      t = __shfl_sync(0xffffffffu, t, 0);
      if (t == gc.nne - 1) {  // every other chunk of the unit has written its record
        if (lane == 0) p.unit_counter[uid] = 0;
        __syncwarp();
        merge_records(p.part + (int64_t)(gc.x - gc.c) * REC, gc.nne, outp);
      }
    }
    const int tcur = gc.tail >> 4;  // tile of the appended row
    if (p.refs.leader[gc.ri] && gc.tail + 1 == s && p.rmax != nullptr && tcur >= gc.t0 && tcur < gc.t1) {
      __syncwarp();
      seal_cluster<bf16, D>(p, p.refs.group[gc.ri], gc.b, gc.h, gc.C1, (const bf16*)p.kc + kv_off(gc));
    }
  };

  for (int j = 0; j < NST; ++j) {
    if (!idone) idone = !issue_one();
    cp_async_commit();
  }
  while (seq_c < seq_i) {
    const int slot = seq_c % NST;
    uint8_t* sK = ring + slot * STAGE;
    uint8_t* sV = sK + TILEB;
    const int8_t* kk = keys + slot * 16;
    cp_async_wait<NST - 1>();  // this lane's copies of the tile have landed
    __syncwarp();
    const int mtw = meta[slot];
    const int nv = mtw & 31, cur_r = ((mtw >> 5) & 31) - 1;
    const bool first = (mtw >> 10) & 1, last = (mtw >> 11) & 1;
    if (first) {
      const int2 e = cq[cq_pop % kCQ];
      ++cq_pop;
      gc = geo_of(e.x, e.y);
#pragma unroll
      for (int hn = 0; hn < HN; ++hn) {
        m_run[hn][0] = m_run[hn][1] = kNegInf;
        l_run[hn][0] = l_run[hn][1] = 0.f;
#pragma unroll
        for (int mt = 0; mt < KS; ++mt) o[mt][hn][0] = o[mt][hn][1] = o[mt][hn][2] = o[mt][hn][3] = 0.f;
      }
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
    if (cur_r >= 0 || nv < 16) {
      if (cur_r >= 0) {
        // the appended row goes from the inputs to the cache and to this tile
        const int layer = p.refs.layer[gc.ri];
        const int64_t nb = layer * p.kvn_ls + (int64_t)(gc.b * Hkv + gc.h) * D;
        const uint4* kn = reinterpret_cast<const uint4*>((const bf16*)p.k_new + nb);
        const uint4* vn = reinterpret_cast<const uint4*>((const bf16*)p.v_new + nb);
        bf16* kcw = (bf16*)p.kc + kv_off(gc);
        bf16* vcw = (bf16*)p.vc + kv_off(gc);
        for (int i = lane; i < 2 * CH; i += 32) {
          const int ch = i % CH;
          const bool isv = i >= CH;
          const uint4 val = isv ? vn[ch] : kn[ch];
          const int pch = ch ^ (gc.n & 7);
          *reinterpret_cast<uint4*>((isv ? sV : sK) + cur_r * ROWB + pch * 16) = val;
          reinterpret_cast<uint4*>((isv ? vcw : kcw) + (int64_t)gc.n * D)[pch] = val;
        }
      }
      // rows past the end of the list are zeroed so that P V sees finite values
      for (int i = lane; i < (16 - nv) * CH; i += 32)
        reinterpret_cast<uint4*>(sV + nv * ROWB)[i] = make_uint4(0, 0, 0, 0);
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
        x[e] = (tk < nv) ? (sc[hn][0][e] + sc[hn][1][e]) * p.scale_log2 : kNegInf;
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
      pbh[hn][0] = movmatrix_trans(*reinterpret_cast<const uint32_t*>(&h01));
      pbh[hn][1] = movmatrix_trans(*reinterpret_cast<const uint32_t*>(&h23));
      pbl[hn][0] = movmatrix_trans(pack_bf16(pr[0] - f01.x, pr[1] - f01.y));
      pbl[hn][1] = movmatrix_trans(pack_bf16(pr[2] - f23.x, pr[3] - f23.y));
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
    ++seq_c;
    // refill the stage just consumed before the chunk's flush, so the ring
    // keeps streaming while a last chunk merges its unit
    if (!idone && !abort) idone = !issue_one();
    cp_async_commit();
    if (last && !abort) flush();
  }
  cp_async_wait<0>();

  // ---- the last CTA to finish advances the token counts and resets the
  // control words for the next call
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const int t = atomicAdd(&sp.ctl[kCtlGrid], 1);
    s_misc[1] = (t == (int)gridDim.x - 1);
  }
  __syncthreads();
  if (s_misc[1]) {
    __threadfence();
    if (__ldcg(&sp.ctl[kCtlAbort]) != 0) {
      // a wait gave up: merges of this call may be incomplete, so every
      // unit counter starts the next call from zero
      const int64_t units = (int64_t)p.n_refs * B * Hkv;
      for (int64_t i = threadIdx.x; i < units; i += blockDim.x) p.unit_counter[i] = 0;
    }
    if (threadIdx.x == 0) {
      if (p.advance)
        for (int b = 0; b < B; ++b) {  // a sequence whose append was refused keeps its count
          const int n = p.n_tok[b];
          if (n >= 0 && n + 1 <= p.cap_tokens) p.n_tok[b] = n + 1;
        }
      sp.ctl[kCtlSelClaim] = 0;
      sp.ctl[kCtlAttClaim] = 0;
      sp.ctl[kCtlAbort] = 0;
      sp.ctl[kCtlEpoch] = (int)want;
      sp.ctl[kCtlGrid] = 0;
    }
  }
}

// ------------------------------------------------------------- launch ----

void step_shape(int D, int G, int B, int* wpc, int* nst) {
  if (D == 64) {
    *wpc = 4;
    *nst = 8;
    return;
  }
  if (G == 1 && StepSmem<128>::total(G, 3, 8, B) <= kSmemOptin) {
    *wpc = 8;
    *nst = 3;
  } else if (G <= 8 && StepSmem<128>::total(G, 4, 6, B) <= kSmemOptin) {
    *wpc = 6;
    *nst = 4;
  } else {
    *wpc = 4;
    *nst = G <= 8 ? 5 : 4;
  }
}

int step_smem_bytes(int D, int G, int B) {
  int wpc, nst;
  step_shape(D, G, B, &wpc, &nst);
  return D == 64 ? StepSmem<64>::total(G, nst, wpc, B) : StepSmem<128>::total(G, nst, wpc, B);
}

int step_row_buf(int D, int G, int B, int team_warps, int max_cand, int n_src) {
  int wpc, nst;
  step_shape(D, G, B, &wpc, &nst);
  const int st = D == 64 ? StepSmem<64>::stage(G) : StepSmem<128>::stage(G);
  const int region = team_warps * nst * st;
  int rb = (region - TeamLayout(D, max_cand, 0, n_src).total) / (D * 4 * n_src + 4);
  while (rb > 0 && TeamLayout(D, max_cand, rb, n_src).total > region) --rb;
  return rb > 0 ? rb : 0;
}

int step_ctas() {
  static std::mutex mu;
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return kMaxStepCtas;
  std::lock_guard<std::mutex> lk(mu);
  if (cached[dev] == 0) {
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
      sms = kMaxStepCtas;
    cached[dev] = sms < kMaxStepCtas ? sms : kMaxStepCtas;
  }
  return cached[dev];
}

cudaError_t launch_step(const StepParams& p, int D, cudaStream_t st) {
  int wpc, nst;
  step_shape(D, p.a.G, p.a.B, &wpc, &nst);
  const int smem = step_smem_bytes(D, p.a.G, p.a.B);
  const int hn = p.a.G <= 8 ? 1 : 2;
  auto go = [&](auto kernel) -> cudaError_t {
    cudaError_t e = ensure_dyn_smem((const void*)kernel, smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(kernel, dim3(step_ctas()), dim3(32 * wpc), smem, st, p);
  };
#define MPC_STEP(DD, HH, NN, WW) \
  if (D == DD && hn == HH && nst == NN && wpc == WW) return go(decode_step_kernel<DD, HH, NN, WW>);
  MPC_STEP(64, 1, 8, 4)
  MPC_STEP(128, 1, 3, 8)
  MPC_STEP(128, 1, 4, 6)
  MPC_STEP(128, 1, 5, 4)
  MPC_STEP(64, 2, 8, 4)
  MPC_STEP(128, 2, 4, 4)
#undef MPC_STEP
  return cudaErrorInvalidValue;
}

int take_status_step() { return take_status(); }

}  // namespace mpc
