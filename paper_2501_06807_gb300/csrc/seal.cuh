// Decode-step seal of a full tail (App. A decode append; Sec. 3.3 summaries,
// hierarchical clustering): shared by the attention kernels.
#pragma once

#include "kernels.cuh"

namespace mpc {

// Called by one warp once the s rows of finest cluster c_new (cache rows
// [c_new s, c_new s + s) of `kcache`, the unit's key cache) are in place:
// writes its r_max / r_min / rep (and the mean key when a mean pyramid is
// kept) and merges it into every coarser level of the group's pyramid: a
// node that already held children takes the element-wise max / min with the
// new cluster and recomputes rep = alpha r_max + (1 - alpha) r_min; the mean
// of a node is the running mean over its finest clusters.  A pyramid row past
// a level's capacity is refused (flag 2).
template <typename T, int D>
__device__ void seal_cluster(const AttnParams& p, int group, int b, int h, int c_new, const T* kcache) {
  const int s = p.pyr.s;
  const int lane = threadIdx.x & 31;
  if (c_new >= p.pyr.cap[0]) {
    if (lane == 0) atomicOr(&g_mpc_status, 2);
    return;
  }
  constexpr int PER = D / 32;
  float mx[PER], mn[PER], sm[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) {
    mx[i] = kNegInf;
    mn[i] = -kNegInf;
    sm[i] = 0.f;
  }
#pragma unroll 8
  for (int r = c_new * s; r < c_new * s + s; ++r) {
    const T* row = kcache + (int64_t)r * D;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const int c = lane * PER + i;
      const float v = to_float<T>(row[swz<T>(r, c)]);
      mx[i] = fmaxf(mx[i], v);
      mn[i] = fminf(mn[i], v);
      sm[i] += v;
    }
  }
  const int64_t ubase = ((int64_t)(group * p.B + b) * p.Hkv + h) * p.pyr.rows;
  const float a = p.alpha, am = 1.f - p.alpha;
  int prod = 1;
  for (int l = 0; l < p.pyr.n_levels; ++l) {
    if (l > 0) prod *= p.pyr.fanout[l - 1];
    const int node = c_new / prod;
    const bool fresh = (c_new % prod) == 0;
    if (node >= p.pyr.cap[l]) {
      if (lane == 0) atomicOr(&g_mpc_status, 2);
      return;
    }
    float* Rx = p.rmax + (ubase + p.pyr.off[l] + node) * D;
    float* Rn = p.rmin + (ubase + p.pyr.off[l] + node) * D;
    float* Rp = p.rep + (ubase + p.pyr.off[l] + node) * D;
    float* Rm = p.mean ? p.mean + (ubase + p.pyr.off[l] + node) * D : nullptr;
    const int n_old = c_new - node * prod;  // finest clusters the node held before
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const int c = lane * PER + i;
      float x = mx[i], n = mn[i];
      if (!fresh) {
        x = fmaxf(x, Rx[c]);
        n = fminf(n, Rn[c]);
      }
      Rx[c] = x;
      Rn[c] = n;
      Rp[c] = fmaf(a, x, am * n);
      if (Rm) {  // running mean over the node's finest clusters
        const float m_new = sm[i] / (float)s;
        Rm[c] = fresh ? m_new : fmaf((float)n_old, Rm[c], m_new) / (float)(n_old + 1);
      }
    }
  }
}

}  // namespace mpc
