// One whole decode step in one persistent launch (Alg. 2 Step 2): the
// hierarchical cluster selection of the leader layers (Sec. 3.3-3.4, Eq. 3;
// Alg. 2 Sim + topk) and, for every layer, the decode append and the sparse
// attention over the selected clusters and the tail (Alg. 1; App. A).
//
// Phase 1, selection.  Selection units (leader ref, sequence b, kv head h)
// are claimed from a global counter by teams of warps (the CTA's warps, or
// groups of them when the units outnumber the CTAs).  A team walks the
// unit's summary pyramid from the coarsest level down with the scores and
// the ranking of mpc_select: each round stages the candidates' fp32 summary
// rows with cp.async and scores them (4 lanes per row, row_partial), a
// counting rank marks the k largest, an ordered compaction keeps the ids
// ascending, and the kept clusters' children become the next level's
// candidates.  The selected ids and their count are published as tagged
// 32-bit words (a 16-bit call tag above a 16-bit value) in the workspace, so
// a reader validates each word it reads and needs no flag, fence or second
// round trip.  Every selection unit is claimed by a running CTA that waits on
// no other, so every wait for a tag ends without assuming co-residency.
//
// Phase 2, attention (the persistent attention kernel's schedule).  The rows
// a unit (ref, b, h) attends are listed tail first (the rows after the last
// sealed cluster, then the row appended now, padded to a whole 16-row tile),
// then the s rows of every selected cluster, and cut into 16-row tiles.  The
// tiles of all units form one list, cut into equal contiguous ranges, one per
// warp slot (slots interleaved over the CTAs).  A warp streams its range
// through its own ring of shared-memory stages (cp.async, one commit group
// per tile, NST tiles ahead of its compute) and computes each tile on the
// tensor cores (mma.sync m16n8k16, the GQA group's heads as N, P split into
// bf16 hi + lo).  A unit cut over several warps is merged by the last of its
// pieces to finish (a ticket on the unit's counter; nobody waits): its owner
// (the warp holding the unit's first piece, which ends that warp's range and
// so usually finishes last) folds the other pieces' records, staged in its
// idle ring, into its registers; any other last piece folds them from L2.
#include <mutex>

#include "kernels.cuh"
#include "seal.cuh"
#include "sel_score.cuh"

namespace mpc {
namespace {

constexpr int kSelIds = kStepSelIds;  // selected ids a warp stages at once
constexpr int kMaxStepCtas = kStepCtasMax;
// control words of the workspace
constexpr int kCtlSelClaim = 0, kCtlTeamsDone = 1, kCtlStarted = 2, kCtlEpoch = 3, kCtlSliceClaim = 4,
              kCtlWarpsDone = 5;
constexpr uint64_t kWaitNs = 1000000000ull;  // bound of every wait (1 s)

__device__ __forceinline__ void named_bar(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}
__device__ __forceinline__ int atom_add_acq_rel(int* a, int v) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(a), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ unsigned ld_relaxed_u32(const unsigned* a) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(a) : "memory");
  return v;
}
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}
// tag of the words published by a call: 1 .. 65535, never the tag of the
// previous call and never 0 (a zero-filled workspace holds no valid word)
__device__ __forceinline__ unsigned call_tag(unsigned want) { return (want % 65535u) + 1u; }

}  // namespace

// Shared memory of one CTA: per warp a ring of NST stages (K tile, V tile,
// the unit's queries), the swizzle keys and metadata of its stages and its
// staged selected ids; per team its scalars; the per-sequence table.  A
// selection team borrows its warps' rings as scratch (TeamLayout).
template <int D>
struct StepSmem {
  static constexpr int ROWB = D * 2;
  static constexpr int TILEB = 16 * ROWB;
  static __host__ __device__ constexpr int qbytes(int G) { return ((G * D * 2 + 127) / 128) * 128; }
  static __host__ __device__ constexpr int stage(int G) { return 2 * TILEB + qbytes(G); }
  static __host__ __device__ constexpr int keys_off(int G, int nst, int wpc) { return wpc * nst * stage(G); }
  static __host__ __device__ constexpr int meta_off(int G, int nst, int wpc) { return keys_off(G, nst, wpc) + wpc * nst * 16; }
  static __host__ __device__ constexpr int selb_off(int G, int nst, int wpc) { return meta_off(G, nst, wpc) + wpc * nst * 4; }
  static __host__ __device__ constexpr int team_off(int G, int nst, int wpc) { return selb_off(G, nst, wpc) + wpc * kSelIds * 4; }
  static __host__ __device__ constexpr int tab_off(int G, int nst, int wpc) { return team_off(G, nst, wpc) + wpc * 32; }
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
  const int G = p.G, B = p.B, Hkv = p.Hkv, s = p.pyr.s;
  const int STAGE = S::stage(G);
  uint8_t* ring = smem + warp * NST * STAGE;
  int8_t* keys = reinterpret_cast<int8_t*>(smem + S::keys_off(G, NST, WPC)) + warp * NST * 16;
  int* meta = reinterpret_cast<int*>(smem + S::meta_off(G, NST, WPC)) + warp * NST;
  int* selb = reinterpret_cast<int*>(smem + S::selb_off(G, NST, WPC)) + warp * kSelIds;
  int* s_team = reinterpret_cast<int*>(smem + S::team_off(G, NST, WPC));
  int* s_n = reinterpret_cast<int*>(smem + S::tab_off(G, NST, WPC));  // cache rows before the append, -1 refused
  int* s_nt = s_n + B;     // tiles per unit of sequence b (with the most clusters it can select)
  int* s_k1 = s_nt + B;    // selected clusters: that bound (selection in this call) or the caller's count
  int* s_pre = s_k1 + B;   // exclusive prefix of s_nt (B + 1)
  int* s_misc = s_pre + B + 1;
  const bool sel_in_call = sp.n_sel_units > 0;
  const int recw = 1 + p.sel_cap;  // words of a published selection: count, then ids
  grid_dep_launch();
  grid_dep_wait();
  // the first selection claim of each team goes out with the table's loads
  int first_claim = 0;
  if (sel_in_call && threadIdx.x % (32 * sp.team_warps) == 0) first_claim = atomicAdd(&sp.ctl[kCtlSelClaim], 1);

  // ---- per-sequence table (every load of the warp in flight at once)
  if (warp == 0) {
    const int epoch = lane == 0 ? __ldcg(&sp.ctl[kCtlEpoch]) : 0;
    int carry = 0;
    for (int b0 = 0; b0 < B; b0 += 32) {
      const int b = b0 + lane;
      int n = -1, nt = 0, k1 = 0;
      if (b < B) {
        const int ntok = p.n_tok[b];
        const int ns = (!sel_in_call && p.sel_cap > 0) ? p.n_sel[b] : 0;
        if (ntok < 0 || ntok + 1 > p.cap_tokens) {
          atomicOr(&g_mpc_status, 2);  // no room for the append: skip the sequence
        } else {
          n = ntok;
          const int C1 = n / s, tail = n - C1 * s, tt = (tail + 16) >> 4;
          if (p.sel_cap > 0)
            k1 = sel_in_call ? min(count_from_ppm(C1, sp.keep_ppm[0]), min(C1, p.sel_cap))
                             : max(0, min(ns, min(C1, p.sel_cap)));
          nt = tt + (k1 * s + 15) / 16;
        }
      }
      int incl = nt;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      if (b < B) {
        s_n[b] = n;
        s_nt[b] = nt;
        s_k1[b] = k1;
        s_pre[b] = carry + incl - nt;
      }
      carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) {
      s_pre[B] = carry;
      s_misc[0] = (int)call_tag((unsigned)epoch + 1u);
    }
    // the last CTA to get here (every CTA has read the token counts and the
    // call counter) advances both for the next call; a sequence whose append
    // was refused keeps its count
    // (acquire-release: this CTA's reads above happen before the add, and
    // the last CTA's writes below after every other CTA's add)
    int last = 0;
    if (lane == 0) last = atom_add_acq_rel(&sp.ctl[kCtlStarted], 1) == (int)gridDim.x - 1;
    if (__shfl_sync(0xffffffffu, last, 0)) {
      if (p.advance)
        for (int b = lane; b < B; b += 32) {
          const int n = p.n_tok[b];
          if (n >= 0 && n + 1 <= p.cap_tokens) p.n_tok[b] = n + 1;
        }
      if (lane == 0) {
        sp.ctl[kCtlEpoch] = epoch + 1;
        sp.ctl[kCtlStarted] = 0;
      }
    }
  }
  __syncthreads();
  const unsigned tag = (unsigned)s_misc[0];  // tag of the words this call publishes

  // ================================================= selection teams ====
  if (sel_in_call) {
    const int TW = sp.team_warps, NTT = TW * 32;
    const int team = warp / TW, twarp = warp - team * TW;
    const int tl = threadIdx.x - team * NTT;
    const int MC = sp.max_cand, RB = sp.row_buf, NSRC = sp.n_src;
    const TeamLayout TL(D, MC, RB, NSRC);
    uint8_t* treg = smem + (size_t)team * TW * NST * STAGE;
    float* qsum = reinterpret_cast<float*>(treg);
    unsigned long long* kA = reinterpret_cast<unsigned long long*>(treg + TL.keysA);
    unsigned long long* kB = reinterpret_cast<unsigned long long*>(treg + TL.keysB);
    uint32_t* cs = reinterpret_cast<uint32_t*>(treg + TL.cs);
    int* mark = reinterpret_cast<int*>(treg + TL.mark);
    int* kept = reinterpret_cast<int*>(treg + TL.kept);
    float* rows = reinterpret_cast<float*>(treg + TL.rows);
    float* rows2 = rows + (size_t)RB * D;
    int* tsc = s_team + team * 8;  // claimed unit, walk status, level, count; then the team's mbarrier
    uint64_t* tbar = reinterpret_cast<uint64_t*>(tsc + 6);
    constexpr uint32_t ROWF = D * 4;  // bytes of a summary row
    const float* srcA_of_unit = sp.src0;  // the claimed unit's staged arrays
    const float* srcB_of_unit = sp.src0;
    auto tsync = [&]() {
      if (TW == 1) __syncwarp();
      else named_bar(1 + team, NTT);
    };
    const int top = p.pyr.n_levels - 1;
    constexpr int CPR = D * 4 / 16;  // 16-byte pieces per summary row
    constexpr int V4 = D / 16;
    const int ql = lane & 3, rs = lane >> 2, rot = rs & 1;

    if (tl == 0) {
      mbar_init(tbar, 1);
      fence_barrier_init();
    }
    uint32_t phase = 0;
    // 16-byte aligned runs of summary rows into the staging buffer with 1-D
    // bulk copies, split over the lanes of the calling warp, completing on
    // the team's mbarrier (the caller registered the bytes)
    auto bulk_rows = [&](int dst_row, int64_t src_elem, int nrows) {
      for (int w = 0; w < NSRC; ++w) {
        float* dst = (w ? rows2 : rows) + (size_t)dst_row * D;
        const float* src = (w ? srcB_of_unit : srcA_of_unit) + src_elem;
        const uint32_t nbytes = (uint32_t)nrows * ROWF;
        for (uint32_t off = (uint32_t)lane * 8192u; off < nbytes; off += 32u * 8192u)
          bulk_g2s(reinterpret_cast<uint8_t*>(dst) + off, reinterpret_cast<const uint8_t*>(src) + off,
                   nbytes - off < 8192u ? nbytes - off : 8192u, tbar);
      }
    };
    int claim = first_claim;  // the team leader's claim, issued before the table was read
    while (true) {
      if (tl == 0) tsc[0] = claim;
      tsync();
      const int su = tsc[0];
      if (su >= sp.n_sel_units) {
        // every unit is claimed; the last team to leave resets the counter
        if (tl == 0 && atomicAdd(&sp.ctl[kCtlTeamsDone], 1) == (int)gridDim.x * (WPC / TW) - 1) {
          sp.ctl[kCtlSelClaim] = 0;
          sp.ctl[kCtlTeamsDone] = 0;
        }
        break;
      }
      if (tl == 0) claim = atomicAdd(&sp.ctl[kCtlSelClaim], 1);  // the next unit, ahead of need
      const int ril = su / (B * Hkv), b = (su / Hkv) % B, h = su % Hkv;
      const int ri = sp.lead_ref[ril];
      const int layer = p.refs.layer[ri], group = p.refs.group[ri];
      const int n = s_n[b];
      int C[kMaxLevels];
      level_counts(p.pyr, n > 0 ? n : 0, C);
      const int64_t uoff = ((int64_t)(group * B + b) * Hkv + h) * p.pyr.rows * D;
      srcA_of_unit = sp.src0 + uoff;
      srcB_of_unit = (NSRC == 2 ? sp.src1 : sp.src0) + uoff;
      int* out = sp.sel_out + ((int64_t)(group * B + b) * Hkv + h) * p.sel_cap;
      unsigned* pub = sp.sel_pub + (int64_t)su * recw;
      bool bad = n >= 0 && (C[0] > p.pyr.cap[0] || C[top] > MC);
      int nk = 0;
      bool written = false;  // the ids are in out / pub already (the warp walk writes them)
      if (n >= 0 && !bad && C[0] > 0) {
        // the coarsest level's clusters are the first candidates; when they
        // fit together, every cluster of the level below is staged and
        // scored in the same round ("extra" rows, scores kept in cs), so
        // that level needs no round of its own.  Warp 0 requests the round
        // with bulk copies before anything else, so that the query loads
        // below overlap it.
        int nc = C[top];
        int extra = (sp.spec && top > 0 && nc + C[top - 1] <= RB) ? C[top - 1] : 0;
        bool requested = nc + extra <= RB;
        if (requested && twarp == 0) {
          if (lane == 0) mbar_arrive_expect_tx(tbar, (uint32_t)(nc + extra) * ROWF * NSRC);
          __syncwarp();
          bulk_rows(0, (int64_t)p.pyr.off[top] * D, nc);
          if (extra) bulk_rows(nc, (int64_t)p.pyr.off[top - 1] * D, extra);
        }
        // q_sum = sum over the group's query heads (Eq. 3 is linear in q)
        const bf16* qp = (const bf16*)p.q + layer * p.q_ls + ((int64_t)b * p.Hq + h * G) * D;
        for (int c = tl; c < D; c += NTT) {
          float acc = 0.f;
          for (int g = 0; g < G; ++g) acc += __bfloat162float(qp[g * D + c]);
          qsum[c] = acc;
        }
        for (int i = tl; i < nc; i += NTT) kA[i] = cand_key(0u, i);
        bool have_child = extra > 0, need = true;
        tsync();
        int l = top;
        while (true) {
          if (need) {
            // stage and score the candidates' rows (then the extra rows), RB at
            // a time: a round requested with bulk copies is waited for on the
            // mbarrier; otherwise every thread copies 16-byte pieces
            const int64_t offL = (int64_t)p.pyr.off[l] * D;
            const int64_t offX = (int64_t)(l > 0 ? p.pyr.off[l - 1] : 0) * D;
            const int total = nc + extra;
            for (int x0 = 0; x0 < total; x0 += RB) {
              const int nb = min(RB, total - x0);
              if (requested) {
                if (!mbar_wait_bounded(tbar, phase)) bad = true;
                phase ^= 1u;
              } else {
                for (int c = tl; c < nb * CPR; c += NTT) {
                  const int r = c / CPR, part = c - r * CPR, x = x0 + r;
                  const int64_t srow = (x < nc ? offL + (int64_t)cand_id(kA[x]) * D : offX + (int64_t)(x - nc) * D) + part * 4;
                  cp_async16(rows + (size_t)r * D + part * 4, srcA_of_unit + srow);
                  if (NSRC == 2) cp_async16(rows2 + (size_t)r * D + part * 4, srcB_of_unit + srow);
                }
                cp_async_commit();
                cp_async_wait<0>();
              }
              tsync();
              float4 qv[V4];
              qv_load_order<D>(qv, qsum, ql, rot);
              for (int r0 = twarp * 8; r0 < nb; r0 += TW * 8) {
                const int r = r0 + rs;
                float a = 0.f;
                if (r < nb)
                  a = NSRC == 1 ? row_partial<D, false>(rows + (size_t)r * D, nullptr, qv, ql, rot)
                                : row_partial<D, true>(rows + (size_t)r * D, rows2 + (size_t)r * D, qv, ql, rot);
                a += __shfl_xor_sync(0xffffffffu, a, 1);
                a += __shfl_xor_sync(0xffffffffu, a, 2);
                if (ql == 0 && r < nb) {
                  const int x = x0 + r;
                  if (x < nc) kA[x] = cand_key(orderable(a), cand_id(kA[x]));
                  else cs[x - nc] = orderable(a);
                }
              }
              fence_proxy_async_smem();  // the staged rows may next be refilled by bulk copies
              tsync();
            }
            extra = 0;
            requested = false;
          }
          int nn = 0;  // candidates of the next level
          if (nc <= 32) {
            // warp 0 walks the levels whose candidates fit a warp, in
            // registers (lane i holds candidate i): a candidate is kept iff
            // fewer than k keys are larger; the kept clusters' children
            // (scores known from the first round) continue the walk without
            // a barrier; at the finest level it writes the selection
            if (twarp == 0) {
              const unsigned lt = (1u << lane) - 1u;
              unsigned long long key = lane < nc ? kA[lane] : 0ull;
              int lw = l, ncw = nc, st = 0;  // st: 0 finished, 1 next level handed over
              bool hc = have_child;
              while (true) {
                const int kw = min(count_from_ppm(C[lw], sp.keep_ppm[lw]), ncw);
                int cnt = 0;
                if (kw < ncw) {
#pragma unroll
                  for (int j = 0; j < 32; ++j) cnt += (int)(__shfl_sync(0xffffffffu, key, j) > key);
                }
                const bool keep = lane < ncw && cnt < kw;
                const unsigned bal = __ballot_sync(0xffffffffu, keep);
                const int nkw = __popc(bal), pos = __popc(bal & lt);
                const int id = cand_id(key);
                // the kept ids in order
                if (keep) kept[pos] = id;
                __syncwarp();
                if (lw == 0) {
                  const bool ok = nkw <= p.sel_cap;
                  for (int q = lane; q < p.sel_cap; q += 32) {
                    const int v = (ok && q < nkw) ? kept[q] : -1;
                    out[q] = v;
                    pub[1 + q] = (tag << 16) | ((unsigned)v & 0xffffu);
                  }
                  nk = ok ? nkw : 0;
                  if (!ok && lane == 0) atomicOr(&g_mpc_status, 4);
                  break;
                }
                // and their children
                const int fw = p.pyr.fanout[lw - 1], nC = C[lw - 1];
                const int last = nkw > 0 ? kept[nkw - 1] : 0;
                const int nnw = nkw > 0 ? (nkw - 1) * fw + min(fw, nC - last * fw) : 0;
                if (hc && nnw <= 32) {
                  const int child = lane < nnw ? kept[lane / fw] * fw + lane % fw : 0;
                  __syncwarp();
                  key = lane < nnw ? cand_key(cs[child], child) : 0ull;
                  --lw;
                  ncw = nnw;
                  hc = false;
                  continue;
                }
                if (nnw > MC) {
                  st = 2;
                } else {
                  for (int x = lane; x < nnw; x += 32) {
                    const int child = kept[x / fw] * fw + x % fw;
                    kB[x] = cand_key(hc ? cs[child] : 0u, child);
                  }
                  st = hc ? 3 : 1;  // 3: the children's scores are known (more than 32 of them)
                  if (!hc && nnw <= RB) {
                    // request the children's rows now: one bulk copy per kept
                    // cluster (its children are consecutive rows of the level)
                    if (lane == 0) mbar_arrive_expect_tx(tbar, (uint32_t)nnw * ROWF * NSRC);
                    __syncwarp();
                    const int64_t offC = (int64_t)p.pyr.off[lw - 1] * D;
                    for (int pp = lane; pp < nkw; pp += 32) {
                      const int c0 = kept[pp] * fw, cnt = min(fw, nC - c0);
                      for (int w = 0; w < NSRC; ++w)
                        bulk_g2s((w ? rows2 : rows) + (size_t)pp * fw * D, (w ? srcB_of_unit : srcA_of_unit) + offC + (int64_t)c0 * D,
                                 (uint32_t)cnt * ROWF, tbar);
                    }
                    st = 4;  // 4: to be scored, rows requested
                  }
                }
                ncw = nnw;
                --lw;
                break;
              }
              if (lane == 0) {
                tsc[1] = st;
                tsc[2] = lw;
                tsc[3] = st == 0 ? nk : ncw;
              }
            }
            tsync();
            const int st = tsc[1];
            if (st == 0) {
              nk = tsc[3];
              written = true;
              break;
            }
            if (st == 2) {
              bad = true;
              break;
            }
            l = tsc[2];
            nn = tsc[3];
            need = st == 1 || st == 4;
            requested = st == 4;
          } else {
            // the team ranks more candidates than a warp holds: a candidate
            // is kept iff fewer than k keys are larger, counted by tpc threads
            // per candidate over shared memory (four independent sums each)
            const int k = min(count_from_ppm(C[l], sp.keep_ppm[l]), nc);
            {
              int tpc = 1, sh = 0;  // threads per candidate
              while (tpc < 32 && tpc * 2 * nc <= NTT) {
                tpc <<= 1;
                ++sh;
              }
              const int work = nc << sh, work32 = (work + 31) & ~31;
              for (int x = tl; x < work32; x += NTT) {
                const int i = x >> sh, t = x & (tpc - 1);
                int c0 = 0, c1 = 0, c2 = 0, c3 = 0;
                if (x < work && k < nc) {
                  const unsigned long long ki = kA[i];
                  int j = t;
                  for (; j + 3 * tpc < nc; j += 4 * tpc) {
                    c0 += (int)(kA[j] > ki);
                    c1 += (int)(kA[j + tpc] > ki);
                    c2 += (int)(kA[j + 2 * tpc] > ki);
                    c3 += (int)(kA[j + 3 * tpc] > ki);
                  }
                  for (; j < nc; j += tpc) c0 += (int)(kA[j] > ki);
                }
                int cnt = (c0 + c1) + (c2 + c3);
                for (int o = tpc >> 1; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
                if (x < work && t == 0) mark[i] = cnt < k;
              }
            }
            tsync();
            // order-preserving compaction of the kept candidates (ids stay ascending)
            if (twarp == 0) {
              const unsigned lt = (1u << lane) - 1u;
              int nkw = 0;
              for (int i0 = 0; i0 < nc; i0 += 32) {
                const bool fl = i0 + lane < nc && mark[i0 + lane] != 0;
                const unsigned bal = __ballot_sync(0xffffffffu, fl);
                if (fl) kept[nkw + __popc(bal & lt)] = cand_id(kA[i0 + lane]);
                nkw += __popc(bal);
              }
              __syncwarp();
              if (lane == 0) {
                // children of the kept clusters: all full except possibly those
                // of the level's last cluster, which is the last kept one
                int nnw = 0;
                if (l > 0 && nkw > 0) {
                  const int f = p.pyr.fanout[l - 1];
                  nnw = (nkw - 1) * f + min(f, C[l - 1] - kept[nkw - 1] * f);
                }
                tsc[1] = nkw;
                tsc[2] = nnw;
              }
            }
            tsync();
            nk = tsc[1];
            if (l == 0) {
              if (nk > p.sel_cap) {
                bad = true;
                break;
              }
              for (int q = tl; q < p.sel_cap; q += NTT) {
                const int v = q < nk ? kept[q] : -1;
                out[q] = v;
                pub[1 + q] = (tag << 16) | ((unsigned)v & 0xffffu);
              }
              written = true;
              break;
            }
            nn = tsc[2];
            if (nn > MC) {
              bad = true;
              break;
            }
            const int f = p.pyr.fanout[l - 1];
            for (int x = tl; x < nn; x += NTT) {
              const int child = kept[x / f] * f + x % f;
              kB[x] = cand_key(have_child ? cs[child] : 0u, child);
            }
            need = !have_child;
            --l;
          }
          tsync();
          unsigned long long* t = kA;
          kA = kB;
          kB = t;
          nc = nn;
          have_child = false;
        }
      }
      if (bad) {
        if (tl == 0) atomicOr(&g_mpc_status, 4);
        nk = 0;
        written = false;
      }
      if (!written)  // no cluster, a refused sequence, or a flagged overflow
        for (int q = tl; q < p.sel_cap; q += NTT) {
          out[q] = -1;
          pub[1 + q] = (tag << 16) | 0xffffu;
        }
      if (tl == 0) {
        pub[0] = (tag << 16) | (unsigned)nk;
        if (ril == 0 && h == 0) sp.n_sel_out[b] = nk;
      }
      tsync();  // the team's scratch is free for the next unit
    }
  }

  // ================================================ attention ranges ====
  const bool fast = (s & 15) == 0;  // every selected tile is one run of consecutive cache rows
  const int64_t TPR = (int64_t)Hkv * s_pre[B];
  const int64_t NT = TPR * p.n_refs;
  const int64_t NW_all = (int64_t)gridDim.x * WPC;
  // the list's first xA tiles are cut into equal contiguous ranges, one per
  // warp slot (slots [0, NW), interleaved over the CTAs); the other tiles
  // into NB equal slices (slots NW + k) that warps claim once their range is
  // done, so that warps on slower SMs take fewer of them
  const int64_t xA = sp.slice_tiles > 0 ? NT * (int64_t)sp.static_ppm / 1000000 : NT;
  const int NW = (int)(NW_all < xA ? NW_all : xA);
  const int NB = NT > xA ? (int)((NT - xA + sp.slice_tiles - 1) / sp.slice_tiles) : 0;
  const int gw = warp * gridDim.x + blockIdx.x;
  auto slot_of = [&](int64_t x) {  // the range slot holding list tile x
    if (x < xA) return (int)((x * NW + NW - 1) / xA);
    return NW + (int)(((x - xA) * NB + NB - 1) / (NT - xA));
  };
  int64_t x0 = gw < NW ? xA * gw / NW : 0, x1 = gw < NW ? xA * (gw + 1) / NW : 0;
  int slot = gw;  // of the current range
  bool abort = false;

  struct Unit {
    int ri, b, h, n, C1, tail, tt, nt, k1, su;
    int64_t ustart;  // list index of the unit's tile 0
  };
  auto unit_of = [&](int64_t x) {  // the unit holding list tile x, and x's tile within it
    Unit u;
    u.ri = (int)(x / TPR);
    const int64_t rem = x - (int64_t)u.ri * TPR;
    int lo = 0, hi = B - 1;  // largest b with Hkv * pre[b] <= rem
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if ((int64_t)Hkv * s_pre[mid] <= rem) lo = mid;
      else hi = mid - 1;
    }
    u.b = lo;
    const int64_t rem2 = rem - (int64_t)Hkv * s_pre[lo];
    u.nt = s_nt[lo];
    u.h = (int)(rem2 / u.nt);
    u.ustart = x - (rem2 - (int64_t)u.h * u.nt);
    u.n = s_n[lo];
    u.C1 = u.n / s;
    u.tail = u.n - u.C1 * s;
    u.tt = (u.tail + 16) >> 4;  // tail tiles: the tail rows and the appended row
    u.k1 = s_k1[lo];
    const int li = sel_in_call ? sp.lead_of[u.ri] : -1;
    u.su = li >= 0 ? (li * B + u.b) * Hkv + u.h : -1;
    return u;
  };
  // waits (bounded) until every word this lane reads from selection unit
  // su's published words carries this call's tag: lane i of round r reads
  // word_of(32 r + i) for indices below cnt and hands it to put(index,
  // 16-bit value); false if the wait gave up
  auto read_published = [&](int su, int cnt, auto&& word_of, auto&& put) -> bool {
    const unsigned* pub = sp.sel_pub + (int64_t)su * recw;
    for (int i0 = 0; i0 < cnt; i0 += 32) {
      const int i = i0 + lane;
      unsigned v = i < cnt ? ld_relaxed_u32(pub + word_of(i)) : (tag << 16);
      if (__any_sync(0xffffffffu, (v >> 16) != tag)) {
        const uint64_t t0 = global_timer_ns();
        while (__any_sync(0xffffffffu, (v >> 16) != tag)) {
          if (global_timer_ns() - t0 > kWaitNs) {
            if (lane == 0) atomicOr(&g_mpc_status, kStatusWaitTimeout);
            return false;
          }
          __nanosleep(64);
          if (i < cnt && (v >> 16) != tag) v = ld_relaxed_u32(pub + word_of(i));
        }
      }
      if (i < cnt) put(i, v & 0xffffu);
    }
    __syncwarp();
    return true;
  };
  auto kv_off = [&](const Unit& u) {
    return (int64_t)p.refs.layer[u.ri] * p.cache_ls + (int64_t)(u.b * Hkv + u.h) * p.cap_tokens * D;
  };

  // ---- issue side: runs NST tiles ahead of the compute side
  Unit iu;
  iu.ustart = -1;
  iu.nt = 0;
  int64_t ix = x0;       // next list tile to issue
  int ci0 = 0, nci = 0;  // staged window of selected-cluster indices [ci0, ci0 + nci)
  int seq_i = 0;
  // ids of selected clusters of unit iu, staged in selb: cluster ci at
  // selb[ci - ci0] for ci in [ci0, ci0 + nci); an id outside [0, C_1)
  // (corrupt input) is reported and read as cluster 0
  auto check_ids = [&]() {
    for (int i = lane; i < nci; i += 32) {
      const int id = selb[i];
      if (id < 0 || id >= iu.C1) {
        atomicOr(&g_mpc_status, 4);
        selb[i] = 0;
      }
    }
    __syncwarp();
  };
  auto stage_ids = [&](int c0, int cnt) -> bool {
    cnt = min(cnt, kSelIds);
    if (iu.su >= 0) {
      if (!read_published(iu.su, cnt, [&](int i) { return 1 + c0 + i; },
                          [&](int i, unsigned v) { selb[i] = v == 0xffffu ? -1 : (int)v; }))
        return false;
    } else {
      const int* srow = p.sel + ((int64_t)(p.refs.group[iu.ri] * B + iu.b) * Hkv + iu.h) * p.sel_cap;
      for (int i = lane; i < cnt; i += 32) selb[i] = srow[c0 + i];
      __syncwarp();
    }
    ci0 = c0;
    nci = cnt;
    check_ids();
    return true;
  };
  auto issue_one = [&]() -> bool {
    if (ix >= x1 || abort) return false;
    const int64_t x = ix++;
    const bool first = x == x0 || x == iu.ustart + iu.nt;
    if (first) {
      iu = unit_of(x);
      nci = 0;
      if (iu.su >= 0) {
        // the unit's selected count and the ids this piece reads first, in
        // one poll of the words its team published
        const int t = (int)(x - iu.ustart);
        const int cA = t > iu.tt ? 16 * (t - iu.tt) / s : 0;
        const int cnt = max(0, min(iu.k1 - cA, kSelIds));
        int k1 = 0;
        if (!read_published(iu.su, 1 + cnt, [&](int i) { return i == 0 ? 0 : cA + i; },
                            [&](int i, unsigned v) {
                              if (i == 0) k1 = (int)v;
                              else selb[i - 1] = v == 0xffffu ? -1 : (int)v;
                            })) {
          abort = true;
          return false;
        }
        k1 = __shfl_sync(0xffffffffu, k1, 0);
        iu.k1 = min(k1, iu.k1);
        ci0 = cA;
        nci = max(0, min(cnt, iu.k1 - cA));
        check_ids();
      }
    }
    const int t = (int)(x - iu.ustart);
    const int slot = seq_i % NST;
    uint8_t* sK = ring + slot * STAGE;
    uint8_t* sV = sK + TILEB;
    const int64_t co = kv_off(iu);
    const uint8_t* kb = reinterpret_cast<const uint8_t*>((const bf16*)p.kc + co);
    const uint8_t* vb = reinterpret_cast<const uint8_t*>((const bf16*)p.vc + co);
    int nv = 0, cur = -1;
    if (t < iu.tt) {
      // tail rows (consecutive in the cache) and the appended row's slot
      const int a0 = 16 * t;
      const int ncache = max(0, min(16, iu.tail - a0));
      nv = min(16, iu.tail + 1 - a0);
      if (iu.tail >= a0 && iu.tail < a0 + 16) cur = iu.tail - a0;
      const int row0 = iu.C1 * s + a0;
      if (!fast && lane < 16) keys[slot * 16 + lane] = (int8_t)((row0 + lane) & 7);
      const uint8_t* gk = kb + (int64_t)row0 * ROWB;
      const uint8_t* gv = vb + (int64_t)row0 * ROWB;
      for (int i = lane; i < ncache * CH; i += 32) {
        cp_async16(sK + i * 16, gk + i * 16);
        cp_async16(sV + i * 16, gv + i * 16);
      }
    } else {
      const int a0 = 16 * (t - iu.tt);
      nv = max(0, min(16, iu.k1 * s - a0));  // 0: past the unit's last selected row
      if (nv > 0) {
        const int cA = a0 / s, cZ = (a0 + nv - 1) / s;  // clusters this tile reads
        if (cA < ci0 || cZ >= ci0 + nci) {
          if (!stage_ids(cA, iu.k1 - cA)) {
            abort = true;
            return false;
          }
        }
      }
      if (nv > 0 && fast) {
        const int src0 = selb[a0 / s - ci0] * s + (a0 % s);
        const uint8_t* gk = kb + (int64_t)src0 * ROWB;
        const uint8_t* gv = vb + (int64_t)src0 * ROWB;
        for (int i = lane; i < 16 * CH; i += 32) {
          cp_async16(sK + i * 16, gk + i * 16);
          cp_async16(sV + i * 16, gv + i * 16);
        }
      } else if (nv > 0) {
        const int r = lane & 15, a = a0 + r;
        int src = 0;
        if (r < nv) src = selb[a / s - ci0] * s + (a % s);
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
    if (first) {  // the unit's queries ride with its first tile
      const uint8_t* q = reinterpret_cast<const uint8_t*>((const bf16*)p.q + p.refs.layer[iu.ri] * p.q_ls +
                                                          ((int64_t)iu.b * p.Hq + iu.h * G) * D);
      for (int i = lane; i < G * D * 2 / 16; i += 32) cp_async16(sK + 2 * TILEB + i * 16, q + i * 16);
    }
    if (lane == 0) meta[slot] = nv | ((cur + 1) << 5) | (first ? 1 << 10 : 0);
    ++seq_i;
    return true;
  };

  // ---- compute side
  uint32_t qb[HN][KS][2];  // Q^T operand: k = channels, n = heads
  float o[KS][HN][4];      // O^T accumulators: m = channels, n = heads
  float m_run[HN][2], l_run[HN][2];
  Unit u;
  u.ustart = -1;
  u.nt = 0;
  const int r_tok = lane >> 2;       // token row of S^T (and +8)
  const int h_off = 2 * (lane & 3);  // first of this thread's two heads in an n-tile
  const int REC = G * (D + 4);       // record: per head max (log2), sum, 2 pad, o[D]
  float* recA = p.part;                               // [range slot]: a later piece's record
  float* recB = p.part + (int64_t)sp.rec_slots * REC;  // [range slot]: an owner's record

  // folds record rec (max, sum, o) into the registers by log-sum-exp
  auto fold = [&](const float* rec, bool staged, float (&lq)[HN][2]) {
    auto ld = [&](const float* a) { return staged ? *a : __ldcg(a); };
#pragma unroll
    for (int hn = 0; hn < HN; ++hn)
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int g = hn * 8 + h_off + e;
        if (g < G) {
          const float* rg = rec + g * (D + 4);
          const float mk = ld(rg), lk = ld(rg + 1);
          // explicit roundings: every merge path (inlined at several call
          // sites) computes the same bits, so outputs do not depend on which
          // piece of a unit finishes last
          const float M = fmaxf(m_run[hn][e], mk);
          const float wa = (m_run[hn][e] == kNegInf) ? 0.f : fast_exp2(m_run[hn][e] - M);
          const float wb = (mk == kNegInf) ? 0.f : fast_exp2(mk - M);
          m_run[hn][e] = M;
          lq[hn][e] = __fmaf_rn(lk, wb, __fmul_rn(lq[hn][e], wa));
#pragma unroll
          for (int mt = 0; mt < KS; ++mt) {
            o[mt][hn][e] = __fmaf_rn(wb, ld(rg + 4 + mt * 16 + r_tok), __fmul_rn(o[mt][hn][e], wa));
            o[mt][hn][2 + e] = __fmaf_rn(wb, ld(rg + 4 + mt * 16 + r_tok + 8), __fmul_rn(o[mt][hn][2 + e], wa));
          }
        }
      }
  };
  // sets the registers to record rec (as written by write_rec)
  auto load_rec = [&](const float* rec, float (&lq)[HN][2]) {
#pragma unroll
    for (int hn = 0; hn < HN; ++hn)
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int g = hn * 8 + h_off + e;
        if (g < G) {
          const float* rg = rec + g * (D + 4);
          m_run[hn][e] = __ldcg(rg);
          lq[hn][e] = __ldcg(rg + 1);
#pragma unroll
          for (int mt = 0; mt < KS; ++mt) {
            o[mt][hn][e] = __ldcg(rg + 4 + mt * 16 + r_tok);
            o[mt][hn][2 + e] = __ldcg(rg + 4 + mt * 16 + r_tok + 8);
          }
        }
      }
  };
  auto write_rec = [&](float* dst, const float (&lq)[HN][2]) {
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
  };

  // end of the warp's piece of unit u
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
    const int64_t uend = u.ustart + u.nt;
    const bool later = u.ustart < x0, owner = !later && uend > x1;
    bool write = !later && !owner;  // the whole unit is in this warp's range
    if (later || owner) {
      const int w0 = slot_of(u.ustart);
      const int nother = slot_of(uend - 1) - w0;  // pieces besides the owner's
      int* cnt = p.unit_counter + ((int64_t)u.ri * B + u.b) * Hkv + u.h;
      if (owner) {
        int done = 0;
        if (lane == 0) done = ld_acquire(cnt);
        done = __shfl_sync(0xffffffffu, done, 0);
        if (done == nother) {
          // every later piece has published: this piece is the last; stage
          // the later pieces' records (slots slot + 1 .. slot + nother,
          // contiguous) in the idle ring with one batch of copies and fold them
          if (lane == 0) *cnt = 0;
          const bool staged = nother * REC * 4 <= NST * STAGE;
          const float* recs = recA + (int64_t)(slot + 1) * REC;
          if (staged) {
            const uint8_t* src = reinterpret_cast<const uint8_t*>(recs);
            for (int i = lane; i < nother * REC / 4; i += 32) cp_async16(ring + i * 16, src + i * 16);
            cp_async_commit();
            cp_async_wait<0>();
            __syncwarp();
            recs = reinterpret_cast<const float*>(ring);
          }
          for (int k = 0; k < nother; ++k) fold(recs + (int64_t)k * REC, staged, lq);
          write = true;
        } else {
          write_rec(recB + (int64_t)slot * REC, lq);
          __syncwarp();
          int t = 0;
          if (lane == 0) t = atom_add_acq_rel(cnt, 1);
          if (__shfl_sync(0xffffffffu, t, 0) == nother) {  // the later pieces finished meanwhile
            if (lane == 0) *cnt = 0;
            for (int k = 1; k <= nother; ++k) fold(recA + (int64_t)(slot + k) * REC, false, lq);
            write = true;
          }
        }
      } else {
        write_rec(recA + (int64_t)slot * REC, lq);
        __syncwarp();
        int t = 0;
        if (lane == 0) t = atom_add_acq_rel(cnt, 1);
        if (__shfl_sync(0xffffffffu, t, 0) == nother) {
          // the last piece of the unit (rare: the owner usually ends last):
          // start from the owner's record and fold every later piece's, this
          // one's included, in piece order, as the owner would
          if (lane == 0) *cnt = 0;
          load_rec(recB + (int64_t)w0 * REC, lq);
          for (int k = 1; k <= nother; ++k) fold(recA + (int64_t)(w0 + k) * REC, false, lq);
          write = true;
        }
      }
    }
    if (write) {
      float* outp = p.out + p.refs.layer[u.ri] * p.out_ls + ((int64_t)u.b * p.Hq + u.h * G) * D;
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
    // the piece holding the appended row seals a full tail; the unit's
    // selection, which read the pyramid, is complete (its count was read)
    const int64_t tcur = u.ustart + (u.tail >> 4);
    if (p.refs.leader[u.ri] && u.tail + 1 == s && p.rmax != nullptr && tcur >= x0 && tcur < x1) {
      __syncwarp();
      seal_cluster<bf16, D>(p, p.refs.group[u.ri], u.b, u.h, u.C1, (const bf16*)p.kc + kv_off(u));
    }
  };

  while (true) {  // the warp's static range, then the slices it claims
  const int nj = (int)(x1 - x0);
  ix = x0;
  seq_i = 0;
  iu.ustart = -1;
  iu.nt = 0;
  bool have = false;
  for (int j = 0; j < NST; ++j) {
    issue_one();
    cp_async_commit();
  }
  for (int j = 0; j < nj && !abort; ++j) {
    const int slot = j % NST;
    uint8_t* sK = ring + slot * STAGE;
    uint8_t* sV = sK + TILEB;
    const int8_t* kk = keys + slot * 16;
    cp_async_wait<NST - 1>();  // this lane's copies of tile j have landed
    __syncwarp();
    if (j >= seq_i) break;  // its issue gave up (a wait ran out)
    const int mtw = meta[slot];
    const int nv = mtw & 31, cur_r = ((mtw >> 5) & 31) - 1;
    if ((mtw >> 10) & 1) {  // first tile of a unit piece
      if (have) flush();
      // (the issue side read the unit's published count before its first
      // tile, so its selection, which read the pyramid a seal updates, is done)
      u = unit_of(x0 + j);
      have = true;
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
    if (nv > 0) {
      if (cur_r >= 0 || nv < 16) {
        if (cur_r >= 0) {
          // the appended row goes from the inputs to the cache and to this tile
          const int64_t nb = p.refs.layer[u.ri] * p.kvn_ls + (int64_t)(u.b * Hkv + u.h) * D;
          const uint4* kn = reinterpret_cast<const uint4*>((const bf16*)p.k_new + nb);
          const uint4* vn = reinterpret_cast<const uint4*>((const bf16*)p.v_new + nb);
          bf16* kcw = (bf16*)p.kc + kv_off(u);
          bf16* vcw = (bf16*)p.vc + kv_off(u);
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
        float xs[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int tk = r_tok + (e >> 1) * 8;
          xs[e] = (tk < nv) ? (sc[hn][0][e] + sc[hn][1][e]) * p.scale_log2 : kNegInf;
        }
        float pr[4];
#pragma unroll
        for (int e = 0; e < 2; ++e) {  // this thread's two heads
          float mx = fmaxf(xs[e], xs[e + 2]);
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
          const float mnew = fmaxf(m_run[hn][e], mx);
          corr[hn][e] = (m_run[hn][e] == kNegInf) ? 0.f : fast_exp2(m_run[hn][e] - mnew);
          m_run[hn][e] = mnew;
          pr[e] = fast_exp2(xs[e] - mnew);
          pr[e + 2] = fast_exp2(xs[e + 2] - mnew);
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
    }
    __syncwarp();
    issue_one();
    cp_async_commit();  // one group per tile, empty near the end
  }
  cp_async_wait<0>();
  __syncwarp();
  if (have && !abort) flush();
  if (abort || NB == 0) break;
  int k = 0;
  if (lane == 0) k = atomicAdd(&sp.ctl[kCtlSliceClaim], 1);
  k = __shfl_sync(0xffffffffu, k, 0);
  if (k >= NB) break;
  x0 = xA + (NT - xA) * k / NB;
  x1 = xA + (NT - xA) * (k + 1) / NB;
  slot = NW + k;
  }
  // every slice is claimed; the last warp to leave resets the counter
  if (NB > 0 && lane == 0 && atomicAdd(&sp.ctl[kCtlWarpsDone], 1) == (int)(gridDim.x * WPC) - 1) {
    sp.ctl[kCtlSliceClaim] = 0;
    sp.ctl[kCtlWarpsDone] = 0;
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
