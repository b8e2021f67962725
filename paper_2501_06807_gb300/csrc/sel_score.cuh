// Cluster similarity of one staged summary row against the group's summed
// query (Eq. 3 with rep, the average-key baseline with the mean key, or the
// Eq. 2 bound with r_max / r_min), shared by the selection kernels so that a
// cluster gets the same fp32 score in either.
#pragma once

#include "common.cuh"

namespace mpc {

// Four lanes score one row: lane ql of the four holds channel chunks
// ql + 4 c (c < D / 16) of q in registers (`qv`, channel order) and reads the
// same chunks of the row.  The reads go in an order rotated by `rot` (the
// row's parity), so the 32 lanes of a warp-wide read hit 8 distinct 16-byte
// bank groups, but the products are accumulated in channel order, so the
// score does not depend on where the row is staged.  Returns this lane's
// partial sum; the caller adds the four lanes' partials (xor 1, then xor 2).
template <int D, bool BOUND>
__device__ __forceinline__ float row_partial(const float* row_a, const float* row_b, const float4 (&qv)[D / 16],
                                             int ql, int rot) {
  constexpr int V4 = D / 16;
  const float4* ra = reinterpret_cast<const float4*>(row_a);
  const float4* rb = reinterpret_cast<const float4*>(row_b);
  float4 va[V4], vb[V4];
#pragma unroll
  for (int j = 0; j < V4; ++j) {
    const int c = (j + rot) % V4;  // load j fetches chunk c
    va[j] = ra[ql + 4 * c];
    if (BOUND) vb[j] = rb[ql + 4 * c];
  }
  float ax = 0.f, ay = 0.f, az = 0.f, aw = 0.f;
#pragma unroll
  for (int c = 0; c < V4; ++c) {
    const int j0 = c, j1 = (c + V4 - 1) % V4;  // chunk c came from load c - rot
    const float4 v = rot ? va[j1] : va[j0];
    if (!BOUND) {
      ax = fmaf(v.x, qv[c].x, ax);
      ay = fmaf(v.y, qv[c].y, ay);
      az = fmaf(v.z, qv[c].z, az);
      aw = fmaf(v.w, qv[c].w, aw);
    } else {
      const float4 m = rot ? vb[j1] : vb[j0];
      ax += fmaxf(qv[c].x * v.x, qv[c].x * m.x);
      ay += fmaxf(qv[c].y * v.y, qv[c].y * m.y);
      az += fmaxf(qv[c].z * v.z, qv[c].z * m.z);
      aw += fmaxf(qv[c].w * v.w, qv[c].w * m.w);
    }
  }
  return (ax + ay) + (az + aw);
}

// 64-bit candidate key: orderable score, then the inverted id, so that all
// keys are distinct and a larger key is a larger score, then a smaller id.
__device__ __forceinline__ unsigned long long cand_key(uint32_t oscore, int id) {
  return ((unsigned long long)oscore << 32) | (unsigned long long)(0xffffffffu - (uint32_t)id);
}
__device__ __forceinline__ int cand_id(unsigned long long key) {
  return (int)(0xffffffffu - (uint32_t)(key & 0xffffffffull));
}

}  // namespace mpc
