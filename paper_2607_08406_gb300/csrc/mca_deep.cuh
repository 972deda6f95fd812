// Pieces of the deep MLP trial loop shared by the SIMT chain (mca_deep.cu) and the tensor-core
// chain (mca_deep_tc.cu): the candidate of trial tau + k, and the loss change of one sample.
#pragma once

#include "mca_device.cuh"
#include "mca_internal.h"

namespace mca {

// Float index of W[r][k] (256 x 256 layer) inside the split-weight image of the tensor-core chain:
// 16 chunks of 16 columns, each chunk 32 KB (hi 16 KB, then lo), core-matrix order inside
// (columns 4g .. 4g+3 of 256 rows form a 4 KB block). The lo part is 4096 floats further on.
__host__ __device__ __forceinline__ size_t deep_tc_image_index(int r, int k) {
  return (size_t)(k >> 4) * 8192 + (size_t)((k >> 2) & 3) * 1024 + (size_t)r * 4 + (size_t)(k & 3);
}

// Flat index of trial tau's weight from its first Philox word r0 (Eq. 1): uniform over all
// weights, or, under the current-layer schedule, uniform inside its stretch's layer.
__host__ __device__ __forceinline__ unsigned int deep_trial_index(const DeepArgs& a,
                                                                  unsigned long long tau,
                                                                  uint32_t r0) {
  if (a.stretch <= 0) return (unsigned int)(((unsigned long long)r0 * a.off[a.L]) >> 32);
  const int l = stretch_layer(a.seed, tau / (unsigned long long)a.stretch, a.L);
  return (unsigned int)(a.off[l] + (((unsigned long long)r0 * (a.off[l + 1] - a.off[l])) >> 32));
}

// Layer of candidate k's weight (proposal only, no memory reads besides the layer offsets).
__device__ __forceinline__ int deep_candidate_layer(const DeepArgs& a, int k) {
  unsigned int idx;
  if (a.n_explicit > 0) {
    idx = a.ex_idx[k];
  } else {
    const uint4 w = trial_words(a.seed, a.tau + (unsigned long long)k);
    idx = deep_trial_index(a, a.tau + (unsigned long long)k, w.x);
  }
  int l = 0;
  while (l + 1 < a.L && (unsigned long long)idx >= a.off[l + 1]) ++l;
  return l;
}

__device__ __forceinline__ DeepCand deep_candidate(const DeepArgs& a, int k) {
  unsigned int idx;
  uint32_t r1 = 0u;
  const bool ex = a.n_explicit > 0;
  float exv = 0.0f;
  if (ex) {
    idx = a.ex_idx[k];
    exv = a.ex_new[k];
  } else {
    const uint4 w = trial_words(a.seed, a.tau + (unsigned long long)k);
    idx = deep_trial_index(a, a.tau + (unsigned long long)k, w.x);
    r1 = w.y;
  }
  int l = 0;
  while (l + 1 < a.L && (unsigned long long)idx >= a.off[l + 1]) ++l;
  const unsigned long long off = idx - a.off[l];
  DeepCand c;
  c.idx = idx;
  c.layer = l;
  c.row = (int)(off / (unsigned long long)a.n_in[l]);
  c.col = (int)(off % (unsigned long long)a.n_in[l]);
  const Mutation m = draw_mutation(a.wk[l], a.w[l], a.code[l], a.wfix[l], a.sc[l], off, a.op, a.lo,
                                   a.hi, a.delta, a.bound, r1, ex, exv);
  c.oldw = m.oldw;
  c.neww = m.neww;
  c.new_code = m.new_code;
  c.valid = m.valid;
  c.delta = __fsub_rn(c.neww, c.oldw);
  return c;
}

// Loss change of sample n whose output fields become zz (changed: any field differs from the cached
// one). COMMIT writes the new output fields and loss.
template <bool COMMIT>
__device__ __forceinline__ float out_delta(const DeepArgs& a, int n, const float (&zz)[kMaxC],
                                           bool changed) {
  if (!changed) return 0.0f;
  const int Lo = a.L - 1;
  const float ln = sample_loss<-1, -1, kMaxC>(zz, a.C, a.y[n], a.g[Lo], a.act[Lo], a.loss);
  const float dl = ln - a.ell[n];
  if (COMMIT) {
#pragma unroll
    for (int c = 0; c < kMaxC; ++c)
      if (c < a.C) a.Z[Lo][(size_t)c * a.Np + n] = zz[c];
    a.ell[n] = ln;
  }
  return dl;
}

}  // namespace mca
