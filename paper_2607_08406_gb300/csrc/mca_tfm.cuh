// Pieces of the Transformer trial loop shared by the SIMT kernels (mca_tfm.cu) and the tensor-core
// kernels (mca_tfm_tc.cu): the stage a parameter feeds and the candidate of trial tau + k.
#pragma once

#include "mca_device.cuh"
#include "mca_internal.h"

namespace mca {

// Stage of parameter idx: -1 embeddings, b in [0, nL) block b, nL the final LN and head.
__device__ __forceinline__ int tfm_stage(const TfmArgs& a, unsigned long long idx) {
  if (idx < a.o_blk0) return -1;
  if (idx < a.o_lnf_g) return (int)((idx - a.o_blk0) / a.blk_size);
  return a.nL;
}

// Where the recomputation of a candidate in parameter idx of block `stage` starts (Section 2.4's
// cached forward at sub-block granularity; the tensor-core kernels): kRestartBlock, the block's
// input; kRestartFfn (LN2 gain or bias), the block's cached mid stream after its attention
// sub-block; kRestartUnit (W1, b1, W2, b2), one hidden unit of the block's feed-forward network,
// a rank-1 change of the block's output stream, after which block stage + 1 starts. The block's
// parameters are laid out ln1, attention, ln2, W1, b1, W2, b2, so the last two kinds are its tail.
enum TfmRestart { kRestartBlock = 0, kRestartFfn = 1, kRestartUnit = 2 };

__device__ __forceinline__ int tfm_restart(const TfmArgs& a, unsigned long long idx, int stage) {
  if (stage < 0 || stage >= a.nL) return kRestartBlock;
  const unsigned long long off = idx - a.o_blk0 - (unsigned long long)stage * a.blk_size;
  if (off < a.r_ln2g) return kRestartBlock;
  return off < a.r_w1 ? kRestartFfn : kRestartUnit;
}

// Whether the candidate leaves its block's attention sub-block (and so its mid stream) unchanged.
__device__ __forceinline__ bool tfm_ffn_param(const TfmArgs& a, unsigned long long idx, int stage) {
  return tfm_restart(a, idx, stage) != kRestartBlock;
}

// The batch's first trial, and its width (fewer at the end of a run whose batches run ahead of the
// host).
__device__ __forceinline__ unsigned long long tfm_batch_tau(const TfmArgs& a) {
  return a.tau_dev ? __ldcg(a.tau_dev) : a.tau;
}

__device__ __forceinline__ int tfm_batch_width(const TfmArgs& a, unsigned long long tau) {
  if (a.n_explicit > 0) return a.n_explicit;
  if (!a.tau_dev) return a.Kb;
  return tau >= a.tau_end ? 0 : (int)min((unsigned long long)a.Kb, a.tau_end - tau);
}

__device__ __forceinline__ DeepCand tfm_candidate(const TfmArgs& a, int k) {
  unsigned int idx;
  uint32_t r1 = 0u;
  const bool ex = a.n_explicit > 0;
  float exv = 0.0f;
  if (ex) {
    idx = a.ex_idx[k];
    exv = a.ex_new[k];
  } else {
    const uint4 w = trial_words(a.seed, tfm_batch_tau(a) + (unsigned long long)k);
    idx = (unsigned int)(((unsigned long long)w.x * a.P) >> 32);
    r1 = w.y;
  }
  const Mutation m = draw_mutation(MCA_W_FP32, a.params, nullptr, nullptr, 1.0f, idx, a.op, a.lo,
                                   a.hi, a.delta, a.bound, r1, ex, exv);
  DeepCand c;
  c.idx = idx;
  c.layer = tfm_stage(a, idx);
  c.row = idx < a.o_pos ? (int)(idx / (unsigned long long)a.d) : -1;   // token of a tok_emb entry
  c.col = 0;
  c.oldw = m.oldw;
  c.neww = m.neww;
  c.new_code = 0;
  c.valid = m.valid;
  c.delta = __fsub_rn(c.neww, c.oldw);
  return c;
}

}  // namespace mca
