// Cluster similarity of one staged summary row against the group's summed
// query (Eq. 3 with rep, the average-key baseline with the mean key, or the
// Eq. 2 bound with r_max / r_min), shared by the selection kernels so that a
// cluster gets the same fp32 score in either.
#pragma once

#include "common.cuh"

namespace mpc {

// Four lanes score one row: lane ql of the four reads channel chunks
// ql + 4 c (c < D / 16) of the row, in an order rotated by `rot` (the row's
// parity, fixed for a lane): load j fetches chunk (j + rot) % (D / 16), so
// the 32 lanes of a warp-wide read hit 8 distinct 16-byte bank groups.  `qv`
// holds the lane's chunks of q in that same load order (qv_load_order).
// Each chunk's four products are summed first (x, y, z, w), then the chunks
// in channel order, so the score does not depend on where the row is staged;
// only one float per chunk stays live (not the loaded rows), which keeps the
// 4-warp kernel within its register budget.  Returns this lane's partial
// sum; the caller adds the four lanes' partials (xor 1, then xor 2).
template <int D, bool BOUND>
__device__ __forceinline__ float row_partial(const float* row_a, const float* row_b, const float4 (&qv)[D / 16],
                                             int ql, int rot) {
  constexpr int V4 = D / 16;
  const float4* ra = reinterpret_cast<const float4*>(row_a);
  const float4* rb = reinterpret_cast<const float4*>(row_b);
  float pc[V4];  // pc[j]: the products of the chunk load j fetched
#pragma unroll
  for (int j = 0; j < V4; ++j) {
    const int c = (j + rot) % V4;
    const float4 v = ra[ql + 4 * c];
    const float4 q = qv[j];
    if (!BOUND) {
      pc[j] = fmaf(v.w, q.w, fmaf(v.z, q.z, fmaf(v.y, q.y, v.x * q.x)));
    } else {
      const float4 m = rb[ql + 4 * c];
      pc[j] = ((fmaxf(q.x * v.x, q.x * m.x) + fmaxf(q.y * v.y, q.y * m.y)) + fmaxf(q.z * v.z, q.z * m.z)) +
              fmaxf(q.w * v.w, q.w * m.w);
    }
  }
  // channel order: chunk c came from load (c - rot) mod V4
  float s = rot ? pc[V4 - 1] : pc[0];
#pragma unroll
  for (int c = 1; c < V4; ++c) s += rot ? pc[c - 1] : pc[c];
  return s;
}

// The lane's q chunks in row_partial's load order: qv[j] = chunk
// ql + 4 ((j + rot) % (D / 16)) of the summed query.
template <int D>
__device__ __forceinline__ void qv_load_order(float4 (&qv)[D / 16], const float* qsum, int ql, int rot) {
  constexpr int V4 = D / 16;
#pragma unroll
  for (int j = 0; j < V4; ++j) qv[j] = reinterpret_cast<const float4*>(qsum)[ql + 4 * ((j + rot) % V4)];
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
