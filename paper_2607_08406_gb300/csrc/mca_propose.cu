// Proposals of a run of trials (Eq. 1) as explicit candidates, for callers that take the decision
// outside a handle: the sample-sharded chain evaluates every trial of a batch on each shard's
// samples, adds the shards' loss changes and decides once for all shards (Eq. 2 is a sum over
// samples). Trial tau's flat index and new value come from the same Philox words and the same
// index and mutation rules as mca_run's kernels (mlp2_trial_index / deep_trial_index, which agree
// for two layers; draw_mutation), so a shard evaluates exactly the candidates mca_run would.
#include "mca_device.cuh"
#include "mca_internal.h"

namespace mca {

namespace {

__global__ void propose_kernel(ProposeArgs a) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= a.n) return;
  const unsigned long long tau = a.tau0 + (unsigned long long)k;
  const uint4 w = trial_words(a.seed, tau);
  unsigned int idx;
  if (a.stretch <= 0) {
    idx = (unsigned int)(((unsigned long long)w.x * a.off[a.L]) >> 32);
  } else {
    const int l = stretch_layer(a.seed, tau / (unsigned long long)a.stretch, a.L);
    idx = (unsigned int)(a.off[l] + (((unsigned long long)w.x * (a.off[l + 1] - a.off[l])) >> 32));
  }
  int l = 0;
  while (l + 1 < a.L && (unsigned long long)idx >= a.off[l + 1]) ++l;
  const unsigned long long off = idx - a.off[l];
  const Mutation m = draw_mutation(a.wk[l], a.w[l], a.code[l], a.wfix[l], a.sc[l], off, a.op, a.lo,
                                   a.hi, a.delta, a.bound, w.y, false, 0.0f);
  mca_trace_rec r;
  r.tau = tau;
  r.idx = idx;
  r.accept = 0;
  r.old_w = m.oldw;
  r.new_w = m.neww;
  r.valid = m.valid;
  r.forced = 0;
  r.dS = 0.0;
  r.S = 0.0;
  a.rec[k] = r;
  a.ex_idx[k] = idx;
  // a rejected proposal is evaluated as the no-op (its loss change is exactly 0 and is not used)
  a.ex_new[k] = m.valid ? m.neww : m.oldw;
}

}  // namespace

cudaError_t launch_propose(const ProposeArgs& a, cudaStream_t s) {
  if (a.n <= 0) return cudaSuccess;
  propose_kernel<<<(a.n + 127) / 128, 128, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace mca
