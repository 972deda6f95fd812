// Trial loop of the single-hidden-layer MCA path (input -> hidden -> output), Section 2.4, as one
// persistent cooperative kernel.
//
// Cached state (feature-major, so that a mutated neuron's field row is contiguous):
//   z1   [H x Np]   hidden local fields z1[j, n] = sum_i W1[j, i] x[n, i]
//   srec [N x 16]   per sample: output fields z2[0..C), the sample's loss, its label
//   X    CSR by input feature: the non-zero entries x[n, i] of feature i, ascending n
//
// A mutation of W1[j, i] changes z1[j, n] by delta * x[n, i] only where x[n, i] != 0 (a rank-1
// update restricted to feature i's non-zeros) and the output fields by W2[:, j] times neuron j's
// activation change. A mutation of W2[o, j] changes z2[o, n] by delta * f(z1[j, n]) for every n.
//
// Work split: the samples are cut into NR contiguous ranges and CTA r owns range r for the whole
// launch -- it is the only CTA that reads or writes z1[:, n] and srec[n] for n in its range, and it
// keeps the range's sample records in shared memory. Per batch of K candidates:
//   propose   every CTA draws all K proposals itself (Philox; no communication)
//   evaluate  each CTA sums l' - l over its own samples for every candidate, in fixed sub-chunks
//             (warp per sub-chunk, fixed lane order), and writes one partial per (candidate, range)
//   barrier   the only grid-wide synchronisation of a batch
//   decide    every CTA sums each candidate's NR partials in the same fixed order and takes the
//             lowest-index candidate with dS <= theta (Eq. 6: theta = 0; Eq. 7: the trial's
//             Metropolis threshold): the same answer in every CTA
//   commit    each CTA applies the accepted candidate to its own samples (no barrier needed: no
//             other CTA reads them) and writes the new weight value (the same value from all CTAs)
// Every partial depends only on (candidate, range), so dS and the trajectory do not depend on K.
#include <algorithm>
#include <cstdio>

#include "mca_device.cuh"
#include "mca_internal.h"

namespace mca {

struct Cand {
  unsigned long long bytes;  // compulsory DRAM bytes of evaluating this candidate (statistics)
  unsigned int idx;
  int layer, row, col;
  float oldw, neww, delta;
  int new_code;
  int valid;
  int gcnt;                  // entries over all samples; 0: nothing changes, dS = 0 exactly
  int ebeg, ecnt;            // this CTA's segment (CSR entries, or samples of the range)
  int sub0, nsub;            // this CTA's sub-chunks
};

__device__ __forceinline__ void fill_candidate(const Mlp2Args& a, unsigned int idx, uint32_t r1,
                                               bool explicit_value, float ex_new, int r, int s0,
                                               int s1, Cand& c) {
  const int layer = (unsigned long long)idx >= a.P1 ? 1 : 0;
  const unsigned long long off = idx - (layer ? a.P1 : 0ull);
  const int n_in = layer ? a.H : a.D;
  c.idx = idx;
  c.layer = layer;
  c.row = (int)(off / (unsigned long long)n_in);
  c.col = (int)(off % (unsigned long long)n_in);
  const Mutation mu = draw_mutation(layer ? a.wk2 : a.wk1, layer ? a.w2 : a.w1,
                                    layer ? a.code2 : a.code1, layer ? a.wfix2 : a.wfix1,
                                    layer ? a.sc2 : a.sc1, off, a.op, a.lo, a.hi, a.delta, a.bound,
                                    r1, explicit_value, ex_new);
  c.oldw = mu.oldw;
  c.neww = mu.neww;
  c.new_code = mu.new_code;
  c.valid = mu.valid;
  c.delta = __fsub_rn(c.neww, c.oldw);
  const int all = layer == 0 ? a.xs_off[c.col + 1] - a.xs_off[c.col] : a.N;
  // A zero change leaves every field bit-identical: dS = 0 exactly, nothing to evaluate.
  c.gcnt = (c.valid && c.delta != 0.0f) ? all : 0;
  c.bytes = 0ull;
  c.ebeg = 0;
  c.ecnt = 0;
  if (c.gcnt > 0) {
    if (layer == 0) {
      const int* ro = a.xs_roff + (size_t)c.col * (a.NR + 1) + r;
      c.ebeg = ro[0];
      c.ecnt = ro[1] - ro[0];
      c.bytes = 32ull * (unsigned long long)a.xs_sect[c.col] + 8ull * (unsigned long long)all;
    } else {
      c.ecnt = s1 - s0;
      c.bytes = 4ull * (unsigned long long)a.N;
    }
  }
  c.nsub = (c.ecnt + a.SUB - 1) / a.SUB;
}

// Sample records of this CTA's range: field f of range-local sample nl at rec[f * pitch + nl].
struct Recs {
  float* rec;
  int pitch;
};

// One entry of a first-layer candidate: range-local sample nl with input value x and cached field
// z; w holds W2[:, j]. Returns l' - l; COMMIT also writes the new hidden field (*zp) and record.
template <int ACT1, int ACT2, int LOSS, int NC, bool COMMIT>
__device__ __forceinline__ float entry_l1(const Mlp2Args& a, Recs R, float delta,
                                          const float (&w)[NC > 0 ? NC : kMaxC], int nl, float x,
                                          float z, float* zp) {
  const float zn = fmaf(delta, x, z);
  const float da = act<ACT1>(zn, a.g1, a.act1) - act<ACT1>(z, a.g1, a.act1);
  if (COMMIT) *zp = zn;
  if (da == 0.0f) return 0.0f;
  constexpr int M = NC > 0 ? NC : kMaxC;
  const int C = NC > 0 ? NC : a.C;
  float zz[M];
  float ell;
  int y;
  load_srec(R.rec, R.pitch, nl, zz, ell, y);
#pragma unroll
  for (int k = 0; k < M; ++k)
    if (k < C) zz[k] = fmaf(w[k], da, zz[k]);
  const float ln = sample_loss<ACT2, LOSS, M>(zz, C, y, a.g2, a.act2, a.loss);
  if (COMMIT) store_srec(R.rec, R.pitch, nl, zz, ln, y);
  return ln - ell;
}

// One sample of an output-layer candidate W2[o, j] (o = row, j's cached field z1[j, n] = z).
template <int ACT1, int ACT2, int LOSS, int NC, bool COMMIT>
__device__ __forceinline__ float entry_l2(const Mlp2Args& a, Recs R, float delta, int o, int nl,
                                          float z) {
  constexpr int M = NC > 0 ? NC : kMaxC;
  const int C = NC > 0 ? NC : a.C;
  const float av = act<ACT1>(z, a.g1, a.act1);
  float zz[M];
  float ell;
  int y;
  load_srec(R.rec, R.pitch, nl, zz, ell, y);
  float zo = 0.0f;
#pragma unroll
  for (int k = 0; k < M; ++k)
    if (k == o) zo = zz[k];
  const float zon = fmaf(delta, av, zo);
  if (zon == zo) return 0.0f;
#pragma unroll
  for (int k = 0; k < M; ++k)
    if (k == o) zz[k] = zon;
  const float ln = sample_loss<ACT2, LOSS, M>(zz, C, y, a.g2, a.act2, a.loss);
  if (COMMIT) store_srec(R.rec, R.pitch, nl, zz, ln, y);
  return ln - ell;
}

template <int NC>
__device__ __forceinline__ void load_w2c(const float* src, int C, float (&w)[NC > 0 ? NC : kMaxC]) {
  constexpr int M = NC > 0 ? NC : kMaxC;
#pragma unroll
  for (int k = 0; k < M; ++k) w[k] = (NC > 0 || k < C) ? src[k] : 0.0f;
}

// Warp-level sum of l' - l over sub-chunk q of candidate c's segment in this CTA's range. Lane l
// takes entries l, l + 32, ... of the sub-chunk in ascending order (four at a time, loads first).
template <int ACT1, int ACT2, int LOSS, int NC>
__device__ __forceinline__ float eval_sub(const Mlp2Args& a, Recs R, int s0, const Cand& c,
                                          const float* w2c, int q) {
  const int lane = threadIdx.x & 31;
  const int e_lo = q * a.SUB;
  const int e_hi = min(e_lo + a.SUB, c.ecnt);
  const float* zrow = a.z1 + (size_t)(c.layer == 0 ? c.row : c.col) * a.Np;
  const float delta = c.delta;
  const int layer = c.layer, o = c.row, ebeg = c.ebeg;
  float w[NC > 0 ? NC : kMaxC];
  load_w2c<NC>(w2c, a.C, w);
  float acc = 0.0f;
  for (int g = e_lo; g < e_hi; g += 128) {
    int nn[4];
    float xv[4], zv[4];
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int e = g + t * 32 + lane;
      nn[t] = -1;
      xv[t] = 0.0f;
      if (e < e_hi) {
        if (layer == 0) {
          nn[t] = __ldg(a.xs_n + ebeg + e);
          xv[t] = __ldg(a.xs_v + ebeg + e);
        } else {
          nn[t] = s0 + e;
        }
      }
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) zv[t] = nn[t] >= 0 ? zrow[nn[t]] : 0.0f;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      if (nn[t] < 0) continue;
      if (layer == 0)
        acc += entry_l1<ACT1, ACT2, LOSS, NC, false>(a, R, delta, w, nn[t] - s0, xv[t], zv[t],
                                                     nullptr);
      else
        acc += entry_l2<ACT1, ACT2, LOSS, NC, false>(a, R, delta, o, nn[t] - s0, zv[t]);
    }
  }
  return warp_sum(acc);
}

// Up to four sub-chunks of at most 128 entries each (the common case SUB == 128) at once: every lane
// issues the loads of all its entries (up to 16) before computing any, so one warp keeps up to 512
// gathers in flight. The per-sub-chunk lane order is the same as eval_sub's.
template <int ACT1, int ACT2, int LOSS, int NC>
__device__ __forceinline__ void eval_quad(const Mlp2Args& a, Recs R, int s0, const Cand* cs,
                                          const float (*w2c)[kMaxC], const int (&ks)[4],
                                          const int (&qs)[4], int nq, float (&out)[4]) {
  const int lane = threadIdx.x & 31;
  int nn[16];
  float xv[16], zv[16];
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const Cand& c = cs[ks[u]];
    const int e_lo = qs[u] * 128;
    const int e_hi = u < nq ? min(e_lo + 128, c.ecnt) : 0;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int e = e_lo + t * 32 + lane;
      const int sidx = u * 4 + t;
      nn[sidx] = -1;
      xv[sidx] = 0.0f;
      if (e < e_hi) {
        if (c.layer == 0) {
          nn[sidx] = __ldg(a.xs_n + c.ebeg + e);
          xv[sidx] = __ldg(a.xs_v + c.ebeg + e);
        } else {
          nn[sidx] = s0 + e;
        }
      }
    }
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const Cand& c = cs[ks[u]];
    const float* zrow = a.z1 + (size_t)(c.layer == 0 ? c.row : c.col) * a.Np;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int sidx = u * 4 + t;
      zv[sidx] = nn[sidx] >= 0 ? zrow[nn[sidx]] : 0.0f;
    }
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const Cand& c = cs[ks[u]];
    const float delta = c.delta;
    const int layer = c.layer, o = c.row;
    float w[NC > 0 ? NC : kMaxC];
    load_w2c<NC>(w2c[ks[u]], a.C, w);
    float acc = 0.0f;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int sidx = u * 4 + t;
      if (nn[sidx] < 0) continue;
      if (layer == 0)
        acc += entry_l1<ACT1, ACT2, LOSS, NC, false>(a, R, delta, w, nn[sidx] - s0, xv[sidx],
                                                     zv[sidx], nullptr);
      else
        acc += entry_l2<ACT1, ACT2, LOSS, NC, false>(a, R, delta, o, nn[sidx] - s0, zv[sidx]);
    }
    out[u] = warp_sum(acc);
  }
}

template <int ACT1, int ACT2, int LOSS, int NC>
__global__ void __launch_bounds__(kLoopThreads, 1) mlp2_trial_loop(Mlp2Args a) {
  extern __shared__ __align__(16) float s_records[];
  __shared__ Cand s_c[kKmax];
  __shared__ float s_w2c[kKmax][kMaxC];
  __shared__ float s_sub[kKmax * kMaxSubs];
  __shared__ float s_dS[kKmax];
  __shared__ unsigned int s_macc[kKmax / 32], s_mbad[kKmax / 32], s_mforced[kKmax / 32];
  __shared__ int s_flag, s_kstar, s_total, s_bvalid;
  __shared__ unsigned long long s_bbytes, s_tau_hi;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int r = blockIdx.x;
  const int s0 = min(r * a.RS, a.N), s1 = min(s0 + a.RS, a.N);
  const bool explicit_mode = a.n_explicit > 0;
  const Recs R = a.smem_records ? Recs{s_records, a.RS} : Recs{a.srec + s0, a.Np};
  if (a.smem_records) {
    const int ns = s1 - s0;
    for (int t = tid; t < kRecFields * ns; t += kLoopThreads) {
      const int f = t / ns, nl = t - f * ns;
      s_records[f * a.RS + nl] = a.srec[(size_t)f * a.Np + s0 + nl];
    }
  }

  // CTA 0, thread 0 carries the run statistics in registers for the whole launch.
  DevState* st = a.st;
  const bool stats_thread = r == 0 && tid == 0;
  double S = 0.0;
  unsigned long long n_trials = 0, n_acc = 0, n_cand = 0, n_batch = 0, n_waste = 0, n_forced = 0,
                     n_bytes = 0, n_trace = 0, ph0 = 0, ph1 = 0, ph2 = 0, ph3 = 0;
  if (stats_thread) {
    S = st->S;
    n_trace = st->trace_written;
  }
  unsigned int gen = 0;
  unsigned long long tau = a.tau0;
  if (tid == 0) s_tau_hi = a.tau0;
  // acceptance-rate estimate behind the batch width: the same in every CTA
  float rate_a = st->rate_acc, rate_t = st->rate_trials;
  const unsigned long long end = a.tau0 + a.n_trials;
  int buf = 0;
  __syncthreads();

  while (explicit_mode || tau < end) {
    const unsigned long long t_a = stats_thread ? globaltimer_ns() : 0ull;
    const int Kw = a.fixed_K ? a.K : batch_width(rate_a, rate_t, kWidthMlp2, a.K);
    const int Kb = explicit_mode ? a.n_explicit
                                 : (int)((end - tau) < (unsigned long long)Kw ? (end - tau) : Kw);
    // ---- propose: every CTA draws every candidate
    for (int k = tid; k < Kb; k += kLoopThreads) {
      Cand c;
      if (explicit_mode) {
        fill_candidate(a, a.ex_idx[k], 0u, true, a.ex_new[k], r, s0, s1, c);
      } else {
        const uint4 w = trial_words(a.seed, tau + (unsigned long long)k);
        const unsigned int idx =
            mlp2_trial_index(a.P, a.P1, a.seed, tau + (unsigned long long)k, w.x, a.stretch);
        fill_candidate(a, idx, w.y, false, 0.0f, r, s0, s1, c);
      }
      if (c.layer == 0 && c.gcnt > 0) {
#pragma unroll
        for (int q = 0; q < kMaxC; ++q)
          s_w2c[k][q] = q < a.C ? a.w2[(size_t)q * a.H + c.row] : 0.0f;
      }
      s_c[k] = c;
    }
    __syncthreads();
    if (warp == 0) {                 // exclusive scan of the sub-chunk counts; batch statistics
      int v[4], loc = 0;
      unsigned long long bytes = 0ull;
      int valid = 0;
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int k = lane * 4 + t;
        v[t] = k < Kb ? s_c[k].nsub : 0;
        loc += v[t];
        if (k < Kb) {
          // bytes of candidates not evaluated before in this launch (a candidate re-evaluated in
          // the next batch finds its data on chip)
          if (tau + (unsigned long long)k >= s_tau_hi) bytes += s_c[k].bytes;
          valid += s_c[k].valid;
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        bytes += __shfl_xor_sync(0xffffffffu, bytes, o);
        valid += __shfl_xor_sync(0xffffffffu, valid, o);
      }
      if (lane == 0) {
        s_bbytes = bytes;
        s_bvalid = valid;
      }
      int inc = loc;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += y;
      }
      int ex = inc - loc;
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int k = lane * 4 + t;
        if (k < Kb) s_c[k].sub0 = ex;
        ex += v[t];
      }
      if (lane == 31) s_total = inc;
    }
    __syncthreads();

    // ---- evaluate this CTA's samples: warp per sub-chunk (four at a time when SUB == 128)
    {
      const int total = s_total;
      int k = 0;
      if (a.SUB == 128) {
        for (int it0 = warp; it0 < total; it0 += 4 * kLoopWarps) {
          int ks[4], qs[4], nq = 0;
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int it = it0 + u * kLoopWarps;
            ks[u] = k;
            qs[u] = 0;
            if (it < total) {
              while (s_c[k].sub0 + s_c[k].nsub <= it) ++k;
              ks[u] = k;
              qs[u] = it - s_c[k].sub0;
              nq = u + 1;
            }
          }
          float v[4];
          eval_quad<ACT1, ACT2, LOSS, NC>(a, R, s0, s_c, s_w2c, ks, qs, nq, v);
          if (lane == 0) {
#pragma unroll
            for (int u = 0; u < 4; ++u)
              if (u < nq) s_sub[it0 + u * kLoopWarps] = v[u];
          }
        }
      } else {
        for (int it = warp; it < total; it += kLoopWarps) {
          while (s_c[k].sub0 + s_c[k].nsub <= it) ++k;
          const float v =
              eval_sub<ACT1, ACT2, LOSS, NC>(a, R, s0, s_c[k], s_w2c[k], it - s_c[k].sub0);
          if (lane == 0) s_sub[it] = v;
        }
      }
    }
    __syncthreads();
    float* part = a.partial + (size_t)buf * kKmax * a.NR;
    for (int k = tid; k < Kb; k += kLoopThreads) {
      float s = 0.0f;
      const int b = s_c[k].sub0, nb = s_c[k].nsub;
      for (int q = 0; q < nb; ++q) s += s_sub[b + q];
      part[(size_t)k * a.NR + r] = s;
    }
    const unsigned long long t_b = stats_thread ? globaltimer_ns() : 0ull;
    if (!grid_sync(a.bar, gridDim.x, gen, &st->err, &s_flag)) break;
    const unsigned long long t_c = stats_thread ? globaltimer_ns() : 0ull;

    // ---- dS of every candidate: the NR partials in a fixed order (lane-strided, compensated
    // fp32). A warp takes candidates warp, warp + 16, warp + 32, warp + 48 together, loads first.
    for (int k0 = warp; k0 < Kb; k0 += 4 * kLoopWarps) {
      float hi[4] = {0.0f, 0.0f, 0.0f, 0.0f}, lo[4] = {0.0f, 0.0f, 0.0f, 0.0f};
      for (int q0 = 0; q0 < a.NR; q0 += 32 * 8) {
        float v[4][8];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int k = k0 + u * kLoopWarps;
          const bool live = k < Kb && s_c[k].gcnt > 0;
#pragma unroll
          for (int m = 0; m < 8; ++m) {
            const int q = q0 + m * 32 + lane;
            v[u][m] = (live && q < a.NR) ? part[(size_t)k * a.NR + q] : 0.0f;
          }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
          for (int m = 0; m < 8; ++m) two_sum_add(hi[u], lo[u], v[u][m]);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int k = k0 + u * kLoopWarps;
        const float t = warp_sum_comp(hi[u], lo[u]);
        if (lane == 0 && k < Kb) s_dS[k] = s_c[k].valid ? t : __int_as_float(0x7fc00000);
      }
    }
    __syncthreads();
    if (explicit_mode) {
      if (r == 0)
        for (int k = tid; k < Kb; k += kLoopThreads) a.ex_out[k] = (double)s_dS[k];
      break;
    }

    // ---- decide (the same in every CTA): lowest-index candidate with dS <= theta (Eq. 6 / 7)
    if (warp < kKmax / 32) {
      bool acc = false, bad = false, forced = false;
      const int k = tid;
      if (k < Kb && s_c[k].valid) {
        const unsigned long long tk = tau + (unsigned long long)k;
        bool facc = false;
        if (a.nforce > 0) {          // binary search of the forced-decision list
          int lo = 0, hi = a.nforce;
          while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (a.ftau[mid] < tk)
              lo = mid + 1;
            else
              hi = mid;
          }
          if (lo < a.nforce && a.ftau[lo] == tk) {
            forced = true;
            facc = a.facc[lo] != 0;
          }
        }
        const float d = s_dS[k];
        if (forced) {
          acc = facc;
        } else {
          bad = !isfinite(d);
          acc = accept_change(d, a.strict, a.metro, a.seed, tk, a.msc);
        }
      }
      const unsigned int ma = __ballot_sync(0xffffffffu, acc);
      const unsigned int mb = __ballot_sync(0xffffffffu, bad);
      const unsigned int mf = __ballot_sync(0xffffffffu, forced);
      if (lane == 0) {
        s_macc[warp] = ma;
        s_mbad[warp] = mb;
        s_mforced[warp] = mf;
      }
    }
    __syncthreads();
    if (tid == 0) {
      int kstar = -1, kbad = -1;
      for (int w = 0; w < kKmax / 32 && kstar < 0; ++w)
        if (s_macc[w]) kstar = w * 32 + __ffs(s_macc[w]) - 1;
      for (int w = 0; w < kKmax / 32 && kbad < 0; ++w)
        if (s_mbad[w]) kbad = w * 32 + __ffs(s_mbad[w]) - 1;
      if (kbad >= 0 && (kstar < 0 || kbad <= kstar)) kstar = -2;
      s_kstar = kstar;
      if (stats_thread) {
        const int last = kstar >= 0 ? kstar : Kb - 1;
        if (a.trace_cap > 0) {
          for (int k = 0; k <= last; ++k) {
            mca_trace_rec rec;
            rec.tau = tau + (unsigned long long)k;
            rec.idx = s_c[k].idx;
            rec.accept = k == kstar ? 1 : 0;
            rec.old_w = s_c[k].oldw;
            rec.new_w = s_c[k].neww;
            rec.valid = s_c[k].valid;
            rec.forced = (int)((s_mforced[k >> 5] >> (k & 31)) & 1u);
            rec.dS = (double)s_dS[k];
            rec.S = S;
            a.trace[n_trace % (unsigned long long)a.trace_cap] = rec;
            ++n_trace;
          }
        }
        for (int w = 0; w < kKmax / 32; ++w) {
          unsigned int m = s_mforced[w];
          const int hi = last - w * 32;
          if (hi < 31) m &= hi < 0 ? 0u : ((2u << hi) - 1u);
          n_forced += (unsigned long long)__popc(m);
        }
        n_cand += (unsigned long long)s_bvalid;
        n_bytes += s_bbytes;
        ++n_batch;
        if (kstar >= 0) {
          n_trials += (unsigned long long)(kstar + 1);
          ++n_acc;
          n_waste += (unsigned long long)(Kb - kstar - 1);
          S += (double)s_dS[kstar];
          if (s_c[kstar].layer == 0 && s_c[kstar].gcnt > 0)
            n_bytes += 32ull * (unsigned long long)a.xs_sect[s_c[kstar].col];
        } else if (kstar == -1) {
          n_trials += (unsigned long long)Kb;
        }
      }
    }
    __syncthreads();
    const int kstar = s_kstar;
    const unsigned long long t_d = stats_thread ? globaltimer_ns() : 0ull;
    if (kstar == -2) {                // the same non-finite candidate in every CTA
      if (stats_thread) atomicCAS(&st->err, 0, (int)MCA_ERR_NUMERIC);
      break;
    }

    // ---- commit the accepted candidate to this CTA's samples (no writes on a reject)
    if (kstar >= 0) {
      const Cand& c = s_c[kstar];
      if (c.gcnt > 0) {
        if (c.layer == 0) {
          float* zrow = a.z1 + (size_t)c.row * a.Np;
          float w[NC > 0 ? NC : kMaxC];
          load_w2c<NC>(s_w2c[kstar], a.C, w);
          for (int e = tid; e < c.ecnt; e += kLoopThreads) {
            const int n = __ldg(a.xs_n + c.ebeg + e);
            const float x = __ldg(a.xs_v + c.ebeg + e);
            (void)entry_l1<ACT1, ACT2, LOSS, NC, true>(a, R, c.delta, w, n - s0, x, zrow[n],
                                                      zrow + n);
          }
        } else {
          const float* zrow = a.z1 + (size_t)c.col * a.Np;
          for (int e = tid; e < c.ecnt; e += kLoopThreads)
            (void)entry_l2<ACT1, ACT2, LOSS, NC, true>(a, R, c.delta, c.row, e, zrow[s0 + e]);
        }
      }
      if (tid == 0) {                 // every CTA writes the same value
        const unsigned long long off = c.idx - (c.layer ? a.P1 : 0ull);
        (c.layer ? a.w2 : a.w1)[off] = c.neww;
        const int wk = c.layer ? a.wk2 : a.wk1;
        if (wk != MCA_W_FP32) (c.layer ? a.code2 : a.code1)[off] = (signed char)c.new_code;
      }
      __syncthreads();
      if (tid == 0) s_tau_hi = max(s_tau_hi, tau + (unsigned long long)Kb);
      tau += (unsigned long long)(kstar + 1);
      rate_a = rate_a * kRateDecay + 1.0f;
      rate_t = rate_t * kRateDecay + (float)(kstar + 1);
    } else {
      if (tid == 0) s_tau_hi = max(s_tau_hi, tau + (unsigned long long)Kb);
      tau += (unsigned long long)Kb;
      rate_a = rate_a * kRateDecay;
      rate_t = rate_t * kRateDecay + (float)Kb;
    }
    if (stats_thread) {
      const unsigned long long t_e = globaltimer_ns();
      ph0 += t_b - t_a;
      ph1 += t_c - t_b;
      ph2 += t_d - t_c;
      ph3 += t_e - t_d;
    }
    buf ^= 1;
  }

  // ---- epilogue: sample records back to global memory, statistics to the device state
  if (a.smem_records && !explicit_mode) {
    __syncthreads();
    const int ns = s1 - s0;
    for (int t = tid; t < kRecFields * ns; t += kLoopThreads) {
      const int f = t / ns, nl = t - f * ns;
      a.srec[(size_t)f * a.Np + s0 + nl] = s_records[f * a.RS + nl];
    }
  }
  if (stats_thread && !explicit_mode) {
    st->S = S;
    st->trials += n_trials;
    st->accepts += n_acc;
    st->candidates += n_cand;
    st->batches += n_batch;
    st->wasted += n_waste;
    st->forced += n_forced;
    st->alg_bytes += n_bytes;
    st->trace_written = n_trace;
    st->phase_ns[0] += ph0;
    st->phase_ns[1] += ph1;
    st->phase_ns[2] += ph2;
    st->phase_ns[3] += ph3;
    st->rate_acc = rate_a;
    st->rate_trials = rate_t;
  }
}

// ------------------------------------------------------------------------------------------------
// Windowed trial loop. Same work split, order of sums and decisions as mlp2_trial_loop, but each CTA
// keeps a ring of kWS candidate slots: slot (t mod kWS) holds trial t's candidate for this CTA's range
// and, for first-layer candidates with at most kCap entries in the range, the gathered entries
// (range-local sample, activation change f(z + delta x) - f(z), new field z + delta x). A batch then
// evaluates and commits from shared memory only.
//
// The CTA's warps have two roles. kProdWarps producer warps prepare slots ahead of the batches
// (Philox, weight, CSR and z1 gathers), in trial order, never more than kWS trials ahead; they take
// no part in the batch's barriers, so their memory latency overlaps everything else. The other
// (consumer) warps run the batches: set-up, evaluation, the grid-wide exchange, decision, commit.
// A slot records how many commits this CTA had made when its preparation began (its epoch); every
// commit is appended to a log. Before a batch uses a slot, the log entries since its epoch are
// replayed: a commit of the same weight (its old value changed) or of a first-layer weight on the
// same hidden row (z1 changed) sends the slot back for preparation; a commit of its W2 column is
// patched in.
// ------------------------------------------------------------------------------------------------
struct WSlot {
  Cand c;
  unsigned long long ticket;  // trial + 1 once the slot is ready for it (written last)
  int state;                  // 1 entries cached (or nothing to evaluate), 2 read from global
  int epoch;                  // commits of this CTA before the slot's data were read
};

// One logged commit of the windowed loop.
struct CommitLog {
  unsigned int idx;
  int layer, row, col;
  float neww;
  int changes_z1;             // a first-layer commit with entries: its z1 row changed
};

// Per-phase device timers of the windowed loop (statistics only; each read of the global timer
// sits on the batch's critical path). Built in with -DMCA_PHASE_TIMERS=1.
#ifndef MCA_PHASE_TIMERS
#define MCA_PHASE_TIMERS 0
#endif
constexpr bool kPhaseTimers = MCA_PHASE_TIMERS != 0;
constexpr int kLogLen = 128;
static_assert(kLogLen > kWS, "a slot is used at most kWS commits after its preparation began");
constexpr int kProdWarps = 3;
constexpr int kConsWarps = kLoopWarps - kProdWarps;
constexpr int kConsThreads = kConsWarps * 32;

// Barrier of the consumer warps only (named barrier 1).
__device__ __forceinline__ void cons_sync() {
  asm volatile("bar.sync 1, %0;" ::"r"(kConsThreads) : "memory");
}

size_t mlp2_window_smem_bytes(int RS) {
  return sizeof(float) * (size_t)kRecFields * RS +
         (size_t)kWS * kCap * (sizeof(unsigned short) + 2 * sizeof(float));
}

// One cached entry: l' - l from the activation change da (COMMIT: also the new record).
template <int ACT2, int LOSS, int NC, bool COMMIT>
__device__ __forceinline__ float entry_cached(const Mlp2Args& a, Recs R,
                                              const float (&w)[NC > 0 ? NC : kMaxC], int nl,
                                              float da) {
  if (da == 0.0f) return 0.0f;
  constexpr int M = NC > 0 ? NC : kMaxC;
  const int C = NC > 0 ? NC : a.C;
  float zz[M];
  float ell;
  int y;
  load_srec(R.rec, R.pitch, nl, zz, ell, y);
#pragma unroll
  for (int k = 0; k < M; ++k)
    if (k < C) zz[k] = fmaf(w[k], da, zz[k]);
  const float ln = sample_loss<ACT2, LOSS, M>(zz, C, y, a.g2, a.act2, a.loss);
  if (COMMIT) store_srec(R.rec, R.pitch, nl, zz, ln, y);
  return ln - ell;
}

// l' - l of one cached entry without branches (0 exactly when da == 0), so that a lane can keep
// several entries in flight.
template <int ACT2, int LOSS, int NC>
__device__ __forceinline__ float cached_delta(const Mlp2Args& a, Recs R,
                                              const float (&w)[NC > 0 ? NC : kMaxC], int nl,
                                              float da) {
  constexpr int M = NC > 0 ? NC : kMaxC;
  const int C = NC > 0 ? NC : a.C;
  float zz[M];
  float ell;
  int y;
  load_srec(R.rec, R.pitch, nl, zz, ell, y);
#pragma unroll
  for (int k = 0; k < M; ++k)
    if (k < C) zz[k] = fmaf(w[k], da, zz[k]);
  const float ln = sample_loss<ACT2, LOSS, M>(zz, C, y, a.g2, a.act2, a.loss);
  return da == 0.0f ? 0.0f : ln - ell;
}

// Warp-level sum of l' - l over the cached entries [e_lo, e_hi) of a slot. Lane l takes entries
// l, l + 32, ... in ascending order, three at a time.
template <int ACT2, int LOSS, int NC>
__device__ __forceinline__ float eval_cached(const Mlp2Args& a, Recs R,
                                             const float (&w)[NC > 0 ? NC : kMaxC],
                                             const unsigned short* nl, const float* da, int e_lo,
                                             int e_hi) {
  const int lane = threadIdx.x & 31;
  float acc = 0.0f;
  for (int g = e_lo; g < e_hi; g += 96) {
    float v[3];
#pragma unroll
    for (int u = 0; u < 3; ++u) {
      const int e = g + u * 32 + lane;
      const bool in = e < e_hi;
      v[u] = cached_delta<ACT2, LOSS, NC>(a, R, w, in ? (int)nl[e] : 0, in ? da[e] : 0.0f);
    }
#pragma unroll
    for (int u = 0; u < 3; ++u) acc += v[u];
  }
  return warp_sum(acc);
}

// Warp prepares slot sl for trial t: proposal, W2 column, and (cacheable first-layer candidates)
// the gathered entries; then publishes it. `epoch` was read before any of the data.
template <int ACT1>
__device__ __forceinline__ void prepare_slot(const Mlp2Args& a, WSlot* slots, float (*w2c)[kMaxC],
                                             unsigned short* e_nl, float* e_da, float* e_zn,
                                             int sl, unsigned long long t, int epoch, int r, int s0,
                                             int s1) {
  const int lane = threadIdx.x & 31;
  if (lane == 0) {
    const uint4 w = trial_words(a.seed, t);
    const unsigned int idx = mlp2_trial_index(a.P, a.P1, a.seed, t, w.x, a.stretch);
    Cand c;
    fill_candidate(a, idx, w.y, false, 0.0f, r, s0, s1, c);
    slots[sl].c = c;
    slots[sl].epoch = epoch;
  }
  __syncwarp();
  const Cand c = slots[sl].c;
  if (c.layer == 0 && c.gcnt > 0) {
    for (int q = lane; q < kMaxC; q += 32)
      w2c[sl][q] = q < a.C ? a.w2[(size_t)q * a.H + c.row] : 0.0f;
  }
  int state = 2;
  if (c.gcnt == 0) {
    state = 1;
  } else if (c.layer == 0 && c.ecnt <= kCap) {
    const float* zrow = a.z1 + (size_t)c.row * a.Np;
    unsigned short* nl = e_nl + (size_t)sl * kCap;
    float* da = e_da + (size_t)sl * kCap;
    float* zn = e_zn + (size_t)sl * kCap;
    for (int e0 = 0; e0 < c.ecnt; e0 += 128) {
      int nn[4];
      float xv[4], zv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int e = e0 + u * 32 + lane;
        nn[u] = -1;
        xv[u] = 0.0f;
        if (e < c.ecnt) {
          nn[u] = __ldg(a.xs_n + c.ebeg + e);
          xv[u] = __ldg(a.xs_v + c.ebeg + e);
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) zv[u] = nn[u] >= 0 ? zrow[nn[u]] : 0.0f;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int e = e0 + u * 32 + lane;
        if (nn[u] < 0) continue;
        const float z2 = fmaf(c.delta, xv[u], zv[u]);
        nl[e] = (unsigned short)(nn[u] - s0);
        zn[e] = z2;
        da[e] = act<ACT1>(z2, a.g1, a.act1) - act<ACT1>(zv[u], a.g1, a.act1);
      }
    }
    state = 1;
  }
  __syncwarp();
  if (lane == 0) {
    slots[sl].state = state;
    st_release_cta_shared_u64(&slots[sl].ticket, t + 1ull);
  }
  __syncwarp();
}

// Acquires the slot's data when it is ready for trial t.
__device__ __forceinline__ bool slot_ready(const WSlot* slots, unsigned long long t) {
  return ld_acquire_cta_shared_u64(&slots[t % kWS].ticket) == t + 1ull;
}

// The warp replays the commits [slot epoch, epoch) on a ready slot, 32 log entries at a time.
// Returns false (in every lane) when the slot must be prepared again.
__device__ __forceinline__ bool revalidate(WSlot& s, float* w2c, const CommitLog* log, int epoch) {
  const int lane = threadIdx.x & 31;
  const int e0 = s.epoch;
  if (epoch - e0 >= kLogLen) return false;
  const unsigned int idx = s.c.idx;
  const int layer = s.c.layer, row = s.c.row;
  for (int base = e0; base < epoch; base += 32) {
    const int e = base + lane;
    bool stale = false, patch = false;
    int prow = 0;
    float pval = 0.0f;
    if (e < epoch) {
      const CommitLog& L = log[e % kLogLen];
      stale = L.idx == idx || (layer == 0 && L.layer == 0 && L.changes_z1 && L.row == row);
      patch = layer == 0 && L.layer == 1 && L.col == row;
      prow = L.row;
      pval = L.neww;
    }
    if (__any_sync(0xffffffffu, stale)) return false;
    unsigned int pm = __ballot_sync(0xffffffffu, patch);
    while (pm) {                       // in commit order: the latest value of a row wins
      const int j = __ffs(pm) - 1;
      pm &= pm - 1u;
      if (lane == j) w2c[prow] = pval;
      __syncwarp();
    }
  }
  __syncwarp();
  if (lane == 0) s.epoch = epoch;
  __syncwarp();
  return true;
}

// One lane brings a ready slot from epoch E - 1 to E with log entry L (commit E - 1). Returns false
// when the slot must be prepared again.
__device__ __forceinline__ bool replay_one(WSlot& o, float* w2c, const CommitLog& L, int E) {
  const Cand& c = o.c;
  if (L.idx == c.idx || (c.layer == 0 && L.layer == 0 && L.changes_z1 && L.row == c.row))
    return false;
  if (c.layer == 0 && L.layer == 1 && L.col == c.row) w2c[L.row] = L.neww;
  o.epoch = E;
  return true;
}

// Warp 0: the batch's slots and its sub-chunks (lane k and k + 32 for batch position k). The
// prefix over batch positions is taken bit plane by bit plane of the sub-chunk counts (at most
// kMaxSubs), with ballots, so that it costs a few dependent steps.
__device__ __forceinline__ void batch_scan(const WSlot* slots, int Kb, unsigned int sl_tau,
                                           int* bslot, int* sub0, int* nsub, unsigned char* map,
                                           int* total, int* bvalid, int* nlive) {
  static_assert(kMaxSubs < 16, "sub-chunk counts fit four bit planes");
  const int lane = threadIdx.x & 31;
  const unsigned int lt = (1u << lane) - 1u;
  int v[2] = {0, 0};
  bool val[2] = {false, false}, liv[2] = {false, false};
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int k = lane + 32 * h;
    if (k < Kb) {
      const int sl = (int)((sl_tau + (unsigned int)k) % (unsigned int)kWS);
      bslot[k] = sl;
      const Cand& c = slots[sl].c;
      v[h] = c.nsub;
      val[h] = c.valid != 0;
      liv[h] = c.valid && c.gcnt > 0;
    }
  }
  int ex[2] = {0, 0}, tot[2] = {0, 0};
#pragma unroll
  for (int b = 0; b < 4; ++b) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const unsigned int m = __ballot_sync(0xffffffffu, (v[h] >> b) & 1);
      ex[h] += __popc(m & lt) << b;
      tot[h] += __popc(m) << b;
    }
  }
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int k = lane + 32 * h;
    if (k < Kb) {
      const int e = ex[h] + (h ? tot[0] : 0);
      sub0[k] = e;
      nsub[k] = v[h];
      for (int q = 0; q < v[h]; ++q) map[e + q] = (unsigned char)k;
    }
  }
  const int nval = __popc(__ballot_sync(0xffffffffu, val[0])) +
                   __popc(__ballot_sync(0xffffffffu, val[1]));
  const int nliv = __popc(__ballot_sync(0xffffffffu, liv[0])) +
                   __popc(__ballot_sync(0xffffffffu, liv[1]));
  if (lane == 0) {
    *total = tot[0] + tot[1];
    *bvalid = nval;
    *nlive = nliv;
  }
}

// Compulsory bytes of the batch's candidates not evaluated before (statistics of CTA 0).
__device__ __forceinline__ unsigned long long batch_bytes(const WSlot* slots, unsigned long long tau,
                                                          int Kb, unsigned int sl_tau,
                                                          unsigned long long tau_hi) {
  const int lane = threadIdx.x & 31;
  unsigned long long bytes = 0ull;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int k = lane + 32 * h;
    if (k < Kb && tau + (unsigned long long)k >= tau_hi)
      bytes += slots[(sl_tau + (unsigned int)k) % (unsigned int)kWS].c.bytes;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) bytes += __shfl_xor_sync(0xffffffffu, bytes, o);
  return bytes;
}

template <int ACT1, int ACT2, int LOSS, int NC>
__global__ void __launch_bounds__(kLoopThreads, 1) mlp2_window_loop(Mlp2Args a) {
  extern __shared__ __align__(16) float s_dyn[];
  __shared__ WSlot s_slot[kWS];
  __shared__ float s_w2c[kWS][kMaxC];
  __shared__ float s_sub[kKmax * kMaxSubs];
  __shared__ CommitLog s_log[kLogLen];
  __shared__ int s_bslot[kKmax];       // batch position -> slot
  __shared__ int s_sub0[kKmax], s_nsub[kKmax];
  __shared__ float s_dS[kKmax];
  __shared__ unsigned char s_map[kKmax * kMaxSubs];   // sub-chunk -> batch position
  __shared__ unsigned int s_stale[2];
  __shared__ int s_flag, s_kstar, s_total, s_bvalid, s_nlive, s_fail, s_done, s_epoch, s_redo;
  __shared__ unsigned long long s_bbytes, s_tau_hi, s_next, s_cons_tau;
  float* s_records = s_dyn;
  unsigned short* e_nl = reinterpret_cast<unsigned short*>(s_dyn + kRecFields * a.RS);
  float* e_da = reinterpret_cast<float*>(e_nl + kWS * kCap);
  float* e_zn = e_da + kWS * kCap;
  constexpr int M = NC > 0 ? NC : kMaxC;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int r = blockIdx.x;
  const int s0 = min(r * a.RS, a.N), s1 = min(s0 + a.RS, a.N);
  const Recs R{s_records, a.RS};
  {
    const int ns = s1 - s0;
    for (int t = tid; t < kRecFields * ns; t += kLoopThreads) {
      const int f = t / ns, nl = t - f * ns;
      s_records[f * a.RS + nl] = a.srec[(size_t)f * a.Np + s0 + nl];
    }
  }
  for (int q = tid; q < kWS; q += kLoopThreads) s_slot[q].ticket = 0ull;
  DevState* st = a.st;
  unsigned long long tau = a.tau0;
  const unsigned long long end = a.tau0 + a.n_trials;
  if (tid == 0) {
    s_tau_hi = a.tau0;
    s_next = a.tau0;
    s_cons_tau = a.tau0;
    s_fail = 0;
    s_done = 0;
    s_epoch = 0;
  }
  __syncthreads();

  if (warp >= kConsWarps) {
    // ---- producers: prepare slots in trial order, at most kWS trials ahead of the batch
    for (;;) {
      unsigned long long t = 0ull;
      if (lane == 0) t = atomicAdd(&s_next, 1ull);
      t = __shfl_sync(0xffffffffu, t, 0);
      if (t >= end) break;
      int go = 1;
      if (lane == 0) {
        const unsigned long long w0 = globaltimer_ns();
        while (t >= *(volatile unsigned long long*)&s_cons_tau + (unsigned long long)kWS) {
          if (*(volatile int*)&s_done) {
            go = 0;
            break;
          }
          if (globaltimer_ns() - w0 > kBarrierTimeoutNs) {
            atomicCAS(&st->err, 0, (int)MCA_ERR_TIMEOUT);   // the consumers stop at their decision
            go = 0;
            break;
          }
          __nanosleep(64);
        }
      }
      if (!__shfl_sync(0xffffffffu, go, 0)) break;
      int epoch = 0;
      if (lane == 0) epoch = ld_acquire_cta_shared_s32(&s_epoch);
      __syncwarp();
      epoch = __shfl_sync(0xffffffffu, epoch, 0);
      prepare_slot<ACT1>(a, s_slot, s_w2c, e_nl, e_da, e_zn, (int)(t % kWS), t, epoch, r, s0, s1);
    }
  } else {
    // ---- consumers: the batches. The commit of batch b runs at the start of batch b + 1 on warps
    // 1.., overlapped with that batch's set-up on warp 0, which reads neither records nor z1.
    const bool stats_thread = r == 0 && tid == 0;
    const bool timer = kPhaseTimers && tid == 0;   // phase times of every CTA, mean over CTAs
    double S = 0.0;
    unsigned long long n_trials = 0, n_acc = 0, n_cand = 0, n_batch = 0, n_waste = 0, n_forced = 0,
                       n_bytes = 0, n_trace = 0, ph0 = 0, ph1 = 0, ph2 = 0, ph3 = 0, ph4 = 0,
                       n_starve = 0, n_reprep = 0;
    if (stats_thread) {
      S = st->S;
      n_trace = st->trace_written;
    }
    float rate_a = st->rate_acc, rate_t = st->rate_trials;
    unsigned int bidx = 0;
    int epoch = 0;                     // commits of this CTA so far (consumer copy of s_epoch)
    const int kmaxw = min(a.K, kWinBatch);
    unsigned int sl_tau = (unsigned int)(tau % kWS);   // slot of trial tau
    int pend = -1;                     // slot of the accepted candidate not yet committed

    for (;;) {
      const unsigned long long t_a = timer ? globaltimer_ns() : 0ull;
      const bool more = tau < end;
      int Kb = 0;
      if (more) {
        const int Kw = a.fixed_K ? kmaxw : batch_width_fast(rate_a, rate_t, kWidthMlp2, kmaxw);
        Kb = (int)((end - tau) < (unsigned long long)Kw ? (end - tau) : Kw);
      }
      const int E = epoch + (pend >= 0 ? 1 : 0);    // commits including the pending one
      if (warp == 0) {
        // ---- set-up: the batch's slots ready (bounded wait for the producers) and brought up to
        // E, lane k (and k + 32) for batch position k: a slot one commit behind is checked against
        // the pending candidate itself; the log entry is written afterwards
        CommitLog P;
        P.idx = ~0u;
        P.layer = P.row = P.col = -1;
        P.neww = 0.0f;
        P.changes_z1 = 0;
        if (pend >= 0) {
          const Cand& pc = s_slot[pend].c;
          P.idx = pc.idx;
          P.layer = pc.layer;
          P.row = pc.row;
          P.col = pc.col;
          P.neww = pc.neww;
          P.changes_z1 = pc.layer == 0 && pc.gcnt > 0;
        } else if (E > 0) {
          P = s_log[(E - 1) % kLogLen];      // no commit pending: commit E - 1 is logged
        }
        if (lane == 0)     // producers may fill slots up to kWS trials past the oldest in use
          *(volatile unsigned long long*)&s_cons_tau = pend >= 0 ? tau - 1ull : tau;
        bool full[2] = {false, false}, stale[2] = {false, false};
        int sl[2] = {0, 0};
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int k = lane + 32 * h;
          if (k >= Kb) continue;
          const unsigned long long t = tau + (unsigned long long)k;
          sl[h] = (int)((sl_tau + (unsigned int)k) % (unsigned int)kWS);
          if (!slot_ready(s_slot, t)) {
            const unsigned long long w0 = globaltimer_ns();
            unsigned int spins = 0;
            bool ok = true;
            while (!slot_ready(s_slot, t)) {
              if ((++spins & 63u) == 0u && globaltimer_ns() - w0 > kBarrierTimeoutNs) {
                atomicCAS(&st->err, 0, (int)MCA_ERR_TIMEOUT);
                *(volatile int*)&s_fail = 1;
                ok = false;
                break;
              }
            }
            if (kPhaseTimers) n_starve += globaltimer_ns() - w0;
            if (!ok) continue;
          }
          WSlot& o = s_slot[sl[h]];
          const int oe = o.epoch;
          if (oe == E - 1)
            stale[h] = !replay_one(o, s_w2c[sl[h]], P, E);
          else if (oe != E)
            full[h] = true;
        }
        if (pend >= 0 && lane == 0) s_log[epoch % kLogLen] = P;
        const unsigned int mf0 = __ballot_sync(0xffffffffu, full[0]);
        const unsigned int mf1 = __ballot_sync(0xffffffffu, full[1]);
        if (mf0 | mf1) {
          // older commits to replay (slots published after the last look): warp-wide, rare
          __syncwarp();
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            unsigned int m = h ? mf1 : mf0;
            while (m) {
              const int j = __ffs(m) - 1;
              m &= m - 1u;
              const int slj = __shfl_sync(0xffffffffu, sl[h], j);
              const bool okj = revalidate(s_slot[slj], s_w2c[slj], s_log, E);
              if (lane == j) stale[h] = !okj;
            }
          }
        }
        const unsigned int ms0 = __ballot_sync(0xffffffffu, stale[0]);
        const unsigned int ms1 = __ballot_sync(0xffffffffu, stale[1]);
        if (lane == 0) {
          s_stale[0] = ms0;
          s_stale[1] = ms1;
          s_redo = (ms0 | ms1) != 0u || *(volatile int*)&s_fail != 0;
        }
        if ((ms0 | ms1) == 0u)
          batch_scan(s_slot, Kb, sl_tau, s_bslot, s_sub0, s_nsub, s_map, &s_total, &s_bvalid,
                     &s_nlive);
      } else if (pend >= 0) {
        // ---- commit of the pending candidate to this CTA's samples (threads 32..)
        const int sl = pend;
        const Cand c = s_slot[sl].c;
        const int i0 = tid - 32, istride = kConsThreads - 32;
        if (c.gcnt > 0) {
          if (s_slot[sl].state == 1) {
            float w[M];
            load_w2c<NC>(s_w2c[sl], a.C, w);
            float* zrow = a.z1 + (size_t)c.row * a.Np + s0;
            const unsigned short* nl = e_nl + (size_t)sl * kCap;
            const float* da = e_da + (size_t)sl * kCap;
            const float* zn = e_zn + (size_t)sl * kCap;
            for (int e = i0; e < c.ecnt; e += istride) {
              zrow[nl[e]] = zn[e];
              (void)entry_cached<ACT2, LOSS, NC, true>(a, R, w, nl[e], da[e]);
            }
          } else if (c.layer == 0) {
            float* zrow = a.z1 + (size_t)c.row * a.Np;
            float w[M];
            load_w2c<NC>(s_w2c[sl], a.C, w);
            for (int e = i0; e < c.ecnt; e += istride) {
              const int n = __ldg(a.xs_n + c.ebeg + e);
              const float x = __ldg(a.xs_v + c.ebeg + e);
              (void)entry_l1<ACT1, ACT2, LOSS, NC, true>(a, R, c.delta, w, n - s0, x, zrow[n],
                                                        zrow + n);
            }
          } else {
            const float* zrow = a.z1 + (size_t)c.col * a.Np;
            for (int e = i0; e < c.ecnt; e += istride)
              (void)entry_l2<ACT1, ACT2, LOSS, NC, true>(a, R, c.delta, c.row, e, zrow[s0 + e]);
          }
        }
        if (tid == 32) {
          if (r == 0 && c.layer == 0 && c.gcnt > 0)   // hidden-field sectors written back
            n_bytes += 32ull * (unsigned long long)a.xs_sect[c.col];
          const unsigned long long off = c.idx - (c.layer ? a.P1 : 0ull);
          (c.layer ? a.w2 : a.w1)[off] = c.neww;
          const int wk = c.layer ? a.wk2 : a.wk1;
          if (wk != MCA_W_FP32) (c.layer ? a.code2 : a.code1)[off] = (signed char)c.new_code;
        }
      }
      // CTA 0 clears the buffer of batch bidx + 1, which is also that of batch bidx - 2: every CTA
      // has added its share of batch bidx - 1, so every CTA has finished waiting on batch
      // bidx - 2. Warp 1 fences the clearing before the barrier that precedes CTA 0's additions
      // to batch bidx, for which every CTA waits before it adds to batch bidx + 1.
      if (r == 0 && warp == 1) {
        unsigned long long* z = a.accum + (size_t)((bidx + 1) % 3) * kAccStride;
        z[lane] = 0ull;
        z[lane + 32] = 0ull;
        if (lane == 0) z[kArrivalWord] = 0ull;
      }
      cons_sync();
      if (pend >= 0) {
        // every consumer's writes of the commit precede the new epoch that producers read
        ++epoch;
        if (tid == 0) st_release_cta_shared_s32(&s_epoch, epoch);
        pend = -1;
      }
      if (!more) break;
      if (s_redo) {
        if (*(volatile int*)&s_fail) break;
        // slots a commit invalidated, prepared again now that the commit is complete (rare)
        if (warp == 0) {
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            unsigned int m = s_stale[h];
            while (m) {
              const int j = __ffs(m) - 1;
              m &= m - 1u;
              const int k = j + 32 * h;
              const unsigned long long t = tau + (unsigned long long)k;
              prepare_slot<ACT1>(a, s_slot, s_w2c, e_nl, e_da, e_zn,
                                 (int)((sl_tau + (unsigned int)k) % (unsigned int)kWS), t, epoch,
                                 r, s0, s1);
              if (lane == 0) ++n_reprep;
            }
          }
          batch_scan(s_slot, Kb, sl_tau, s_bslot, s_sub0, s_nsub, s_map, &s_total, &s_bvalid,
                     &s_nlive);
        }
        cons_sync();
      }
      const unsigned long long t_s = timer ? globaltimer_ns() : 0ull;
      // ---- evaluate: warp per sub-chunk; cached slots from shared memory, the rest from global
      {
        const int total = s_total;
        for (int it = warp; it < total; it += kConsWarps) {
          const int k = s_map[it];
          const int sl = s_bslot[k];
          const Cand& c = s_slot[sl].c;
          const int q = it - s_sub0[k];
          float v;
          if (s_slot[sl].state == 1) {
            float w[M];
            load_w2c<NC>(s_w2c[sl], a.C, w);
            const int e_lo = q * a.SUB, e_hi = min(e_lo + a.SUB, c.ecnt);
            v = eval_cached<ACT2, LOSS, NC>(a, R, w, e_nl + (size_t)sl * kCap,
                                            e_da + (size_t)sl * kCap, e_lo, e_hi);
          } else {
            v = eval_sub<ACT1, ACT2, LOSS, NC>(a, R, s0, c, s_w2c[sl], q);
          }
          if (lane == 0) s_sub[it] = v;
        }
      }
      const unsigned long long t_v = timer ? globaltimer_ns() : 0ull;
      if (r == 0 && warp == 1) __threadfence();    // the clearing above
      cons_sync();
      // this range's loss change of every candidate, added into the candidate's packed 64-bit
      // word: bits 56..63 count the CTAs that have added, bits 48..55 those whose share was not
      // finite or not below 2^19 in magnitude, bits 0..47 the sum over the other CTAs of
      // (share in units of 2^-20) + 2^39. Integer sums are exact and independent of the order of
      // arrival, so dS is the same in every CTA and for every batch width; the count is the
      // batch's only grid-wide wait, and one load of the word gives everything.
      unsigned long long* acc = a.accum + (size_t)(bidx % 3) * kAccStride;
      for (int k = tid; k < Kb; k += kConsThreads) {
        const Cand& c = s_slot[s_bslot[k]].c;
        if (!c.valid || c.gcnt == 0) continue;
        float sum = 0.0f;
        for (int q = 0; q < s_nsub[k]; ++q) sum += s_sub[s_sub0[k] + q];
        unsigned long long w = 1ull << 56;
        if (isfinite(sum) && fabsf(sum) < 0x1p19f)
          w += (1ull << 39) + (unsigned long long)__float2ll_rn(sum * 0x1p20f);
        else
          w += 1ull << 48;
        atomicAdd(acc + k, w);
      }
      // a batch without a live candidate still synchronises (on the arrival word), so that no
      // CTA runs more than one batch ahead of the clearing of the rotating buffers
      if (tid == 0 && s_nlive == 0) atomicAdd(acc + kArrivalWord, 1ull << 56);
      const unsigned long long t_b = timer ? globaltimer_ns() : 0ull;
      // ---- warp 0 waits until every CTA has added to every live candidate (bounded), then
      // decides
      if (warp == 0) {
        const unsigned long long need = (unsigned long long)gridDim.x;
        int ok = 1;
        unsigned long long v[2] = {0ull, 0ull};
        bool live[2], poll[2];
        const unsigned long long* pa[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int k = lane + 32 * h;
          live[h] = false;
          if (k < Kb) {
            const Cand& c = s_slot[s_bslot[k]].c;
            live[h] = c.valid && c.gcnt > 0;
          }
          poll[h] = live[h];
          pa[h] = acc + k;
        }
        if (s_nlive == 0 && lane == 0) {
          poll[0] = true;
          pa[0] = acc + kArrivalWord;
        }
        // the clock is read only once the wait has lasted 64 polls (and for the phase timers)
        unsigned long long w0 = kPhaseTimers ? globaltimer_ns() : 0ull;
        unsigned int spins = 0;
        for (;;) {
          bool mine = true;
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            if (poll[h] && (v[h] >> 56) < need) {
              v[h] = ld_acquire_gpu_u64(pa[h]);
              mine = mine && (v[h] >> 56) >= need;
            }
          }
          if (__all_sync(0xffffffffu, mine)) break;
          int stop = 0;
          if (lane == 0 && (++spins & 63u) == 0u) {
            const unsigned long long now = globaltimer_ns();
            if (spins == 64u && !kPhaseTimers) w0 = now;
            if (ld_volatile_int(&st->err) != 0) {
              stop = 1;
            } else if (now - w0 > kBarrierTimeoutNs) {
              atomicCAS(&st->err, 0, (int)MCA_ERR_TIMEOUT);
              stop = 1;
            }
          }
          if (__shfl_sync(0xffffffffu, stop, 0)) {
            ok = 0;
            break;
          }
        }
        // decide in the same warp (the same in every CTA): lowest-index candidate with
        // dS <= theta (Eq. 6 / Eq. 7); decisions forced by the caller take precedence; a
        // non-finite dS at or before the first acceptance stops the run
        unsigned int mask_a[2], mask_b[2], mask_f[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int k = lane + 32 * h;
          bool accept = false, bad = false, forced = false;
          if (k < Kb) {
            const Cand& c = s_slot[s_bslot[k]].c;
            float d = 0.0f;
            const unsigned long long nbad = (v[h] >> 48) & 255ull;
            if (!c.valid || (live[h] && nbad != 0ull)) {
              d = __int_as_float(0x7fc00000);
            } else if (live[h]) {
              const long long q =
                  (long long)(v[h] & ((1ull << 48) - 1ull)) - (long long)(need << 39);
              d = __ll2float_rn(q) * 0x1p-20f;
            }
            s_dS[k] = d;
            if (c.valid) {
              const unsigned long long tk = tau + (unsigned long long)k;
              bool facc = false;
              if (a.nforce > 0) {
                int lo = 0, hi = a.nforce;
                while (lo < hi) {
                  const int mid = (lo + hi) >> 1;
                  if (a.ftau[mid] < tk)
                    lo = mid + 1;
                  else
                    hi = mid;
                }
                if (lo < a.nforce && a.ftau[lo] == tk) {
                  forced = true;
                  facc = a.facc[lo] != 0;
                }
              }
              if (forced) {
                accept = facc;
              } else {
                bad = !isfinite(d);
                accept = accept_change(d, a.strict, a.metro, a.seed, tk, a.msc);
              }
            }
          }
          mask_a[h] = __ballot_sync(0xffffffffu, accept);
          mask_b[h] = __ballot_sync(0xffffffffu, bad);
          mask_f[h] = __ballot_sync(0xffffffffu, forced);
        }
        __syncwarp();
        if (lane == 0) {
          if (kPhaseTimers) ph2 += globaltimer_ns() - w0;
          s_flag = ok;                 // an error elsewhere ends this CTA's next wait
          int kstar = mask_a[0] ? __ffs(mask_a[0]) - 1 : (mask_a[1] ? 31 + __ffs(mask_a[1]) : -1);
          const int kbad =
              mask_b[0] ? __ffs(mask_b[0]) - 1 : (mask_b[1] ? 31 + __ffs(mask_b[1]) : -1);
          if (kbad >= 0 && (kstar < 0 || kbad <= kstar)) kstar = -2;
          s_kstar = kstar;
          if (stats_thread && ok) {
            const int last = kstar >= 0 ? kstar : Kb - 1;
            if (a.trace_cap > 0) {
              for (int k = 0; k <= last; ++k) {
                const Cand& c = s_slot[s_bslot[k]].c;
                mca_trace_rec rec;
                rec.tau = tau + (unsigned long long)k;
                rec.idx = c.idx;
                rec.accept = k == kstar ? 1 : 0;
                rec.old_w = c.oldw;
                rec.new_w = c.neww;
                rec.valid = c.valid;
                rec.forced = (int)((mask_f[k >> 5] >> (k & 31)) & 1u);
                rec.dS = (double)s_dS[k];
                rec.S = S;
                a.trace[n_trace % (unsigned long long)a.trace_cap] = rec;
                ++n_trace;
              }
            }
#pragma unroll
            for (int w = 0; w < 2; ++w) {
              unsigned int m = mask_f[w];
              const int hi = last - w * 32;
              if (hi < 31) m &= hi < 0 ? 0u : ((2u << hi) - 1u);
              n_forced += (unsigned long long)__popc(m);
            }
            n_cand += (unsigned long long)s_bvalid;
            ++n_batch;
            if (kstar >= 0) {
              n_trials += (unsigned long long)(kstar + 1);
              ++n_acc;
              n_waste += (unsigned long long)(Kb - kstar - 1);
              S += (double)s_dS[kstar];
            } else if (kstar == -1) {
              n_trials += (unsigned long long)Kb;
            }
          }
        }
      } else if (warp <= 3) {
        if (warp == 1 && r == 0) {
          const unsigned long long bb = batch_bytes(s_slot, tau, Kb, sl_tau, s_tau_hi);
          if (lane == 0) s_bbytes = bb;
        }
        // warps 1..3 bring the published slots past the batch up to date meanwhile, one slot per
        // lane (a few commits behind: replayed by the lane; further: warp-wide)
        const int j = Kb + lane + 32 * (warp - 1);
        const unsigned long long t = tau + (unsigned long long)j;
        bool full = false;
        int slj = 0;
        if (j < kWS && t < end) {
          slj = (int)((sl_tau + (unsigned int)j) % (unsigned int)kWS);
          if (slot_ready(s_slot, t)) {
            WSlot& o = s_slot[slj];
            const int lag = epoch - o.epoch;
            if (lag > 4) {
              full = true;
            } else {
              for (int e = o.epoch; e < epoch; ++e)
                if (!replay_one(o, s_w2c[slj], s_log[e % kLogLen], e + 1)) break;
            }
          }
        }
        unsigned int m = __ballot_sync(0xffffffffu, full);
        while (m) {
          const int jj = __ffs(m) - 1;
          m &= m - 1u;
          const int sj = __shfl_sync(0xffffffffu, slj, jj);
          (void)revalidate(s_slot[sj], s_w2c[sj], s_log, epoch);
        }
      }
      cons_sync();
      if (!s_flag) break;
      const int kstar = s_kstar;
      if (stats_thread) n_bytes += s_bbytes;
      if (timer) {
        const unsigned long long t_c = globaltimer_ns();
        ph0 += t_s - t_a;
        ph1 += t_v - t_s;
        ph4 += t_b - t_v;
        ph3 += t_c - t_b;
      }
      if (kstar == -2) {
        if (stats_thread) atomicCAS(&st->err, 0, (int)MCA_ERR_NUMERIC);
        break;
      }
      if (tid == 0) s_tau_hi = max(s_tau_hi, tau + (unsigned long long)Kb);
      const int adv = kstar >= 0 ? kstar + 1 : Kb;
      if (kstar >= 0) {
        pend = s_bslot[kstar];
        rate_a = rate_a * kRateDecay + 1.0f;
      } else {
        rate_a = rate_a * kRateDecay;
      }
      rate_t = rate_t * kRateDecay + (float)adv;
      tau += (unsigned long long)adv;
      sl_tau = (sl_tau + (unsigned int)adv) % (unsigned int)kWS;
      ++bidx;
    }
    if (tid == 0) *(volatile int*)&s_done = 1;
    if (timer) {
      const unsigned long long g = (unsigned long long)gridDim.x;
      atomicAdd(&st->phase_ns[0], ph0 / g);
      atomicAdd(&st->phase_ns[1], ph1 / g);
      atomicAdd(&st->phase_ns[2], ph2 / g);
      atomicAdd(&st->phase_ns[3], ph3 / g);
      atomicAdd(&st->phase_ns[4], ph4 / g);
    }
    if (lane == 0 && (n_starve | n_reprep)) {
      atomicAdd(&st->phase_ns[6], n_starve / (unsigned long long)gridDim.x);
      atomicAdd(&st->phase_ns[7], n_reprep);
    }
    if (r == 0 && tid == 32 && n_bytes) atomicAdd(&st->alg_bytes, n_bytes);
    if (stats_thread) {
      st->S = S;
      st->trials += n_trials;
      st->accepts += n_acc;
      st->candidates += n_cand;
      st->batches += n_batch;
      st->wasted += n_waste;
      st->forced += n_forced;
      atomicAdd(&st->alg_bytes, n_bytes);
      st->trace_written = n_trace;
      st->rate_acc = rate_a;
      st->rate_trials = rate_t;
    }
  }

  __syncthreads();
  {
    const int ns = s1 - s0;
    for (int t = tid; t < kRecFields * ns; t += kLoopThreads) {
      const int f = t / ns, nl = t - f * ns;
      a.srec[(size_t)f * a.Np + s0 + nl] = s_records[f * a.RS + nl];
    }
  }
}

// Kernel variants with 10 classes: (tanh, sigmoid, MSE), (tanh, identity, CE), (Gaussian, sigmoid,
// MSE); and a generic one that switches on transfer functions, loss and class count at run time.
using LoopFn = void (*)(Mlp2Args);

template <int A1, int A2, int LS, int NC>
static LoopFn loop_variant(bool window) {
  return window ? mlp2_window_loop<A1, A2, LS, NC> : mlp2_trial_loop<A1, A2, LS, NC>;
}

static LoopFn pick_loop(const Mlp2Args& a) {
  const bool w = a.window && a.n_explicit == 0;
  if (a.C == 10) {
    if (a.act1 == MCA_ACT_TANH && a.act2 == MCA_ACT_SIGMOID && a.loss == MCA_LOSS_MSE_ONEHOT)
      return loop_variant<MCA_ACT_TANH, MCA_ACT_SIGMOID, MCA_LOSS_MSE_ONEHOT, 10>(w);
    if (a.act1 == MCA_ACT_TANH && a.act2 == MCA_ACT_IDENTITY && a.loss == MCA_LOSS_SOFTMAX_CE)
      return loop_variant<MCA_ACT_TANH, MCA_ACT_IDENTITY, MCA_LOSS_SOFTMAX_CE, 10>(w);
    if (a.act1 == MCA_ACT_GAUSSIAN && a.act2 == MCA_ACT_SIGMOID && a.loss == MCA_LOSS_MSE_ONEHOT)
      return loop_variant<MCA_ACT_GAUSSIAN, MCA_ACT_SIGMOID, MCA_LOSS_MSE_ONEHOT, 10>(w);
  }
  return loop_variant<-1, -1, -1, -1>(w);
}

size_t mlp2_loop_smem_bytes(const Mlp2Args& a) {
  if (a.window && a.n_explicit == 0) return mlp2_window_smem_bytes(a.RS);
  return a.smem_records ? (size_t)a.RS * kRecFields * sizeof(float) : 0;
}

int mlp2_loop_max_grid(const Mlp2Args& a, int num_sms) {
  const LoopFn loop = pick_loop(a);
  const size_t smem = mlp2_loop_smem_bytes(a);
  if (smem > 0 && cudaFuncSetAttribute((const void*)loop,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem) != cudaSuccess)
    return 0;
  int occ = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, loop, kLoopThreads, smem) !=
      cudaSuccess)
    return 0;
  return occ * num_sms;
}

cudaError_t launch_mlp2_loop(const Mlp2Args& a, cudaStream_t s) {
  const LoopFn loop = pick_loop(a);
  const size_t smem = mlp2_loop_smem_bytes(a);
  if (smem > 0) {
    cudaError_t e = cudaFuncSetAttribute((const void*)loop,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  Mlp2Args args = a;
  void* params[] = {&args};
  return cudaLaunchCooperativeKernel((const void*)loop, dim3(a.NR), dim3(kLoopThreads), params,
                                     smem, s);
}

}  // namespace mca
