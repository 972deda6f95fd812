// Kernels of the single-hidden-layer MCA path (input -> hidden -> output), Section 2.4.
//
// Cached state (feature-major so that a mutated neuron's field row is contiguous):
//   z1   [H x Np]   hidden local fields z1[j, n] = sum_i W1[j, i] x[n, i]
//   srec [N x 16]   per sample: output fields z2[0..C), the sample's loss, its label
//   X    CSR by feature: the non-zero entries x[n, i] of each input feature i, ascending n
//
// One trial = one candidate (Eq. 1). A mutation of W1[j, i] changes z1[j, n] by delta * x[n, i]
// only where x[n, i] != 0 (a rank-1 update restricted to feature i's non-zeros), and the output
// fields by W2[:, j] times the hidden activation change (Section 2.4). A mutation of W2[o, j]
// changes z2[o, n] by delta * f(z1[j, n]) for every sample.
//
// The trial loop is one persistent cooperative kernel. Per batch of K candidates:
//   propose   every CTA draws all K proposals itself (Philox, no communication)
//   evaluate  work items = fixed chunks of kChunk entries of each candidate; each item's partial
//             loss change goes to its own slot (no atomics), so dS_k does not depend on K or grid
//   barrier
//   decide    every CTA sums each candidate's chunk partials in the same fixed order and takes
//             the lowest-index candidate with dS <= 0 (Eq. 6) -- the same answer everywhere
//   commit    only if one was accepted: its chunks rewrite z1 row j and the touched sample
//             records; CTA 0 writes the weight, S, statistics and trace; then a second barrier.
#include <algorithm>
#include <cstdio>

#include "mca_device.cuh"
#include "mca_internal.h"

namespace mca {

struct Cand {
  unsigned int idx;
  int layer, row, col;
  float oldw, neww, delta;
  int new_code;
  int valid;
  int start, cnt, nch;
};

__device__ __forceinline__ void fill_candidate(const Mlp2Args& a, unsigned int idx, uint32_t r1,
                                               bool explicit_value, float ex_new, Cand& c) {
  const int layer = (unsigned long long)idx >= a.P1 ? 1 : 0;
  const unsigned long long off = idx - (layer ? a.P1 : 0ull);
  const int n_in = layer ? a.H : a.D;
  c.idx = idx;
  c.layer = layer;
  c.row = (int)(off / (unsigned long long)n_in);
  c.col = (int)(off % (unsigned long long)n_in);
  const int wk = layer ? a.wk2 : a.wk1;
  const float* weff = layer ? a.w2 : a.w1;
  const signed char* code = layer ? a.code2 : a.code1;
  const float* wfix = layer ? a.wfix2 : a.wfix1;
  const float sc = layer ? a.sc2 : a.sc1;
  c.valid = 1;
  c.new_code = 0;
  c.oldw = weff[off];
  if (explicit_value) {
    c.neww = ex_new;
  } else if (wk == MCA_W_TERNARY_I8) {
    const int oc = code[off];
    const int nc = (int)(((unsigned long long)r1 * 3ull) >> 32) - 1;
    c.oldw = __fmul_rn(sc, (float)oc);
    c.neww = __fmul_rn(sc, (float)nc);
    c.new_code = nc;
  } else if (wk == MCA_W_MASKED_FP32) {
    const int om = code[off];
    const int nm = 1 - om;
    const float w = wfix[off];
    c.oldw = om ? w : 0.0f;
    c.neww = nm ? w : 0.0f;
    c.new_code = nm;
  } else {
    const float u = unit24(r1);
    if (a.op == MCA_OP_PERTURB) {
      const float rr = __fsub_rn(__fmul_rn(2.0f, u), 1.0f);
      c.neww = __fadd_rn(c.oldw, __fmul_rn(a.delta, rr));
    } else {
      c.neww = __fadd_rn(a.lo, __fmul_rn(__fsub_rn(a.hi, a.lo), u));
    }
    if (a.bound > 0.0f && !(fabsf(c.neww) < a.bound)) c.valid = 0;
  }
  c.delta = __fsub_rn(c.neww, c.oldw);
  if (layer == 0) {
    c.start = a.xs_off[c.col];
    c.cnt = a.xs_off[c.col + 1] - c.start;
  } else {
    c.start = 0;
    c.cnt = a.N;
  }
  // A zero change leaves every field bit-identical: dS = 0 exactly, nothing to evaluate.
  c.nch = (c.valid && c.delta != 0.0f) ? (c.cnt + a.CH - 1) / a.CH : 0;
}

// Load one sample record: fields into z[0..C), loss and label.
__device__ __forceinline__ void load_srec(const float* srec, int n, float (&z)[kMaxC], float& ell,
                                          int& y) {
  const float4* p = reinterpret_cast<const float4*>(srec + (size_t)n * kSR);
  const float4 v0 = p[0], v1 = p[1], v2 = p[2], v3 = p[3];
  z[0] = v0.x; z[1] = v0.y; z[2] = v0.z; z[3] = v0.w;
  z[4] = v1.x; z[5] = v1.y; z[6] = v1.z; z[7] = v1.w;
  z[8] = v2.x; z[9] = v2.y; z[10] = v2.z; z[11] = v2.w;
  z[12] = v3.x; z[13] = v3.y;
  z[14] = 0.0f; z[15] = 0.0f;
  ell = v3.z;
  y = __float_as_int(v3.w);
}

__device__ __forceinline__ void store_srec(float* srec, int n, const float (&z)[kMaxC], float ell,
                                           int y) {
  float4* p = reinterpret_cast<float4*>(srec + (size_t)n * kSR);
  p[0] = make_float4(z[0], z[1], z[2], z[3]);
  p[1] = make_float4(z[4], z[5], z[6], z[7]);
  p[2] = make_float4(z[8], z[9], z[10], z[11]);
  p[3] = make_float4(z[12], z[13], ell, __int_as_float(y));
}

// Chunk `chunk` of a first-layer candidate: entries [start + chunk*CH, ...) of feature col.
// Returns this thread's share of sum(l' - l). COMMIT: also write the new fields and losses.
template <int ACT1, int ACT2, int LOSS, bool COMMIT>
__device__ __forceinline__ float l1_chunk(const Mlp2Args& a, const Cand& c, const float* w2c,
                                          int chunk) {
  const int e0 = c.start + chunk * a.CH;
  const int e1 = min(e0 + a.CH, c.start + c.cnt);
  float* zrow = a.z1 + (size_t)c.row * a.Np;
  int nn[kPerThread];
  float xv[kPerThread], zv[kPerThread];
#pragma unroll
  for (int r = 0; r < kPerThread; ++r) {
    const int e = e0 + threadIdx.x + r * kLoopThreads;
    nn[r] = -1;
    if (e < e1) {
      nn[r] = __ldg(a.xs_n + e);
      xv[r] = __ldg(a.xs_v + e);
    }
  }
#pragma unroll
  for (int r = 0; r < kPerThread; ++r) zv[r] = nn[r] >= 0 ? zrow[nn[r]] : 0.0f;
  float acc = 0.0f;
#pragma unroll
  for (int r = 0; r < kPerThread; ++r) {
    if (nn[r] < 0) continue;
    const float zn = fmaf(c.delta, xv[r], zv[r]);
    const float da = act<ACT1>(zn, a.g1, a.act1) - act<ACT1>(zv[r], a.g1, a.act1);
    if (COMMIT) zrow[nn[r]] = zn;
    if (da != 0.0f) {
      float z[kMaxC];
      float ell;
      int y;
      load_srec(a.srec, nn[r], z, ell, y);
#pragma unroll
      for (int k = 0; k < kMaxC; ++k)
        if (k < a.C) z[k] = fmaf(w2c[k], da, z[k]);
      const float ln = sample_loss<ACT2, LOSS, kMaxC>(z, a.C, y, a.g2, a.act2, a.loss);
      acc += ln - ell;
      if (COMMIT) store_srec(a.srec, nn[r], z, ln, y);
    }
  }
  return acc;
}

// Chunk of an output-layer candidate W2[o, j]: samples [chunk*CH, ...).
template <int ACT1, int ACT2, int LOSS, bool COMMIT>
__device__ __forceinline__ float l2_chunk(const Mlp2Args& a, const Cand& c, int chunk) {
  const int n0 = chunk * a.CH;
  const int n1 = min(n0 + a.CH, a.N);
  const float* zrow = a.z1 + (size_t)c.col * a.Np;
  const int o = c.row;
  float zv[kPerThread];
#pragma unroll
  for (int r = 0; r < kPerThread; ++r) {
    const int n = n0 + threadIdx.x + r * kLoopThreads;
    zv[r] = n < n1 ? zrow[n] : 0.0f;
  }
  float acc = 0.0f;
#pragma unroll
  for (int r = 0; r < kPerThread; ++r) {
    const int n = n0 + threadIdx.x + r * kLoopThreads;
    if (n >= n1) continue;
    const float av = act<ACT1>(zv[r], a.g1, a.act1);
    float z[kMaxC];
    float ell;
    int y;
    load_srec(a.srec, n, z, ell, y);
    float zo = 0.0f;
#pragma unroll
    for (int k = 0; k < kMaxC; ++k)
      if (k == o) zo = z[k];
    const float zon = fmaf(c.delta, av, zo);
    if (zon != zo) {
#pragma unroll
      for (int k = 0; k < kMaxC; ++k)
        if (k == o) z[k] = zon;
      const float ln = sample_loss<ACT2, LOSS, kMaxC>(z, a.C, y, a.g2, a.act2, a.loss);
      acc += ln - ell;
      if (COMMIT) store_srec(a.srec, n, z, ln, y);
    }
  }
  return acc;
}

template <int ACT1, int ACT2, int LOSS>
__global__ void __launch_bounds__(kLoopThreads, 1) mlp2_trial_loop(Mlp2Args a) {
  __shared__ Cand s_c[kKmax];
  __shared__ float s_w2c[kKmax][kMaxC];
  __shared__ int s_pre[kKmax + 1];
  __shared__ double s_dS[kKmax];
  __shared__ float s_red[32];
  __shared__ int s_flag, s_kstar;

  unsigned int gen = 0;
  unsigned long long tau = a.tau0;
  const unsigned long long end = a.tau0 + a.n_trials;
  const bool explicit_mode = a.n_explicit > 0;
  int fcur = 0;
  if (threadIdx.x == 0)
    while (fcur < a.nforce && a.ftau[fcur] < tau) ++fcur;
  int buf = 0;
  const size_t pstride = (size_t)kKmax * a.maxch;

  while (explicit_mode || tau < end) {
    const int Kb = explicit_mode ? a.n_explicit
                                 : (int)((end - tau) < (unsigned long long)a.K ? (end - tau) : a.K);
    // ---- propose (every CTA, redundantly)
    for (int k = threadIdx.x; k < Kb; k += blockDim.x) {
      Cand c;
      if (explicit_mode) {
        fill_candidate(a, a.ex_idx[k], 0u, true, a.ex_new[k], c);
      } else {
        const uint4 r = trial_words(a.seed, tau + (unsigned long long)k);
        const unsigned int idx = (unsigned int)(((unsigned long long)r.x * a.P) >> 32);
        fill_candidate(a, idx, r.y, false, 0.0f, c);
      }
      s_c[k] = c;
      if (c.layer == 0) {
#pragma unroll
        for (int q = 0; q < kMaxC; ++q)
          s_w2c[k][q] = q < a.C ? a.w2[(size_t)q * a.H + c.row] : 0.0f;
      }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int t = 0;
      for (int k = 0; k < Kb; ++k) {
        s_pre[k] = t;
        t += s_c[k].nch;
      }
      s_pre[Kb] = t;
    }
    __syncthreads();
    const int total = s_pre[Kb];
    float* part = a.partial + (size_t)buf * pstride;

    // ---- evaluate: items blockIdx.x, blockIdx.x + gridDim.x, ...
    int k = 0;
    for (int it = blockIdx.x; it < total; it += gridDim.x) {
      while (s_pre[k + 1] <= it) ++k;
      const int ch = it - s_pre[k];
      const Cand& c = s_c[k];
      float v = c.layer == 0 ? l1_chunk<ACT1, ACT2, LOSS, false>(a, c, s_w2c[k], ch)
                             : l2_chunk<ACT1, ACT2, LOSS, false>(a, c, ch);
      v = block_sum(v, s_red);
      if (threadIdx.x == 0) part[(size_t)k * a.maxch + ch] = v;
    }
    if (!grid_sync(a.bar, gridDim.x, gen, &a.st->err, &s_flag)) return;

    // ---- per-candidate loss change, fixed order over chunks
    for (int kk = threadIdx.x; kk < Kb; kk += blockDim.x) {
      double s = 0.0;
      const int nch = s_c[kk].nch;
      for (int ch = 0; ch < nch; ++ch) s += (double)part[(size_t)kk * a.maxch + ch];
      s_dS[kk] = s_c[kk].valid ? s : __longlong_as_double(0x7ff8000000000000ll);
    }
    __syncthreads();
    if (explicit_mode) {
      if (blockIdx.x == 0)
        for (int kk = threadIdx.x; kk < Kb; kk += blockDim.x) a.ex_out[kk] = s_dS[kk];
      return;
    }

    // ---- decide (identical in every CTA): lowest-index candidate with dS <= 0 (Eq. 6)
    if (threadIdx.x == 0) {
      int kstar = -1, nonfinite = 0, forced_here = 0;
      for (int kk = 0; kk < Kb; ++kk) {
        const unsigned long long tk = tau + (unsigned long long)kk;
        while (fcur < a.nforce && a.ftau[fcur] < tk) ++fcur;
        const bool forced = fcur < a.nforce && a.ftau[fcur] == tk;
        const double d = s_dS[kk];
        bool acc;
        if (!s_c[kk].valid) {
          acc = false;
        } else if (forced) {
          acc = a.facc[fcur] != 0;
          forced_here++;
        } else {
          if (!isfinite(d)) nonfinite = 1;
          acc = a.strict ? (d < 0.0) : (d <= 0.0);
        }
        if (blockIdx.x == 0 && a.trace_cap > 0) {
          const unsigned long long slot = a.st->trace_written % (unsigned long long)a.trace_cap;
          mca_trace_rec rec;
          rec.tau = tk;
          rec.idx = s_c[kk].idx;
          rec.accept = acc ? 1 : 0;
          rec.old_w = s_c[kk].oldw;
          rec.new_w = s_c[kk].neww;
          rec.valid = s_c[kk].valid;
          rec.forced = forced ? 1 : 0;
          rec.dS = d;
          rec.S = a.st->S;
          a.trace[slot] = rec;
          a.st->trace_written += 1ull;
        }
        if (acc) {
          kstar = kk;
          break;
        }
      }
      s_kstar = nonfinite ? -2 : kstar;
      if (blockIdx.x == 0) {
        DevState* st = a.st;
        st->batches += 1ull;
        st->forced += (unsigned long long)forced_here;
        // compulsory DRAM bytes: per evaluated first-layer candidate the z1 sectors its feature's
        // entries touch plus the entries (index + value); per output-layer candidate one z1 row
        unsigned long long bytes = 0ull;
        for (int kk = 0; kk < Kb; ++kk) {
          const Cand& c = s_c[kk];
          st->candidates += c.valid ? 1ull : 0ull;
          if (c.nch > 0)
            bytes += c.layer == 0 ? 32ull * (unsigned long long)a.xs_sect[c.col] + 8ull * c.cnt
                                  : 4ull * (unsigned long long)a.N;
        }
        if (kstar >= 0 && s_c[kstar].nch > 0 && s_c[kstar].layer == 0)
          bytes += 32ull * (unsigned long long)a.xs_sect[s_c[kstar].col];   // z1 write-back
        st->alg_bytes += bytes;
        if (kstar >= 0) {
          st->trials += (unsigned long long)(kstar + 1);
          st->accepts += 1ull;
          st->wasted += (unsigned long long)(Kb - kstar - 1);
          st->S += s_dS[kstar] == s_dS[kstar] ? s_dS[kstar] : 0.0;
        } else {
          st->trials += (unsigned long long)Kb;
        }
        if (nonfinite) atomicCAS(&st->err, 0, (int)MCA_ERR_NUMERIC);
      }
    }
    __syncthreads();
    const int kstar = s_kstar;
    if (kstar == -2) return;       // every CTA sees the same non-finite candidate and leaves

    // ---- commit the accepted candidate (no writes at all on a reject)
    if (kstar >= 0) {
      const Cand& c = s_c[kstar];
      for (int ch = blockIdx.x; ch < c.nch; ch += gridDim.x) {
        if (c.layer == 0)
          (void)l1_chunk<ACT1, ACT2, LOSS, true>(a, c, s_w2c[kstar], ch);
        else
          (void)l2_chunk<ACT1, ACT2, LOSS, true>(a, c, ch);
      }
      if (blockIdx.x == 0 && threadIdx.x == 0) {
        const unsigned long long off = c.idx - (c.layer ? a.P1 : 0ull);
        float* weff = c.layer ? a.w2 : a.w1;
        weff[off] = c.neww;
        const int wk = c.layer ? a.wk2 : a.wk1;
        if (wk != MCA_W_FP32) (c.layer ? a.code2 : a.code1)[off] = (signed char)c.new_code;
      }
      if (!grid_sync(a.bar, gridDim.x, gen, &a.st->err, &s_flag)) return;
      tau += (unsigned long long)(kstar + 1);
    } else {
      tau += (unsigned long long)Kb;
    }
    buf ^= 1;
  }
}

// ------------------------------------------------------------------------------------------------
// Full forward pass (resync): z1 = W1 X^T (SGEMM), then output fields, losses and S.
// ------------------------------------------------------------------------------------------------

// XT[i, n] = X[n, i] for n < N, 0 in the padding columns.
__global__ void transpose_pad_kernel(const float* __restrict__ X, int N, int D,
                                     float* __restrict__ XT, int Np) {
  __shared__ float tile[32][33];
  const int n0 = blockIdx.x * 32, i0 = blockIdx.y * 32;
  for (int r = threadIdx.y; r < 32; r += blockDim.y) {
    const int n = n0 + r, i = i0 + threadIdx.x;
    tile[r][threadIdx.x] = (n < N && i < D) ? X[(size_t)n * D + i] : 0.0f;
  }
  __syncthreads();
  for (int r = threadIdx.y; r < 32; r += blockDim.y) {
    const int i = i0 + r, n = n0 + threadIdx.x;
    if (i < D && n < Np) XT[(size_t)i * Np + n] = tile[threadIdx.x][r];
  }
}

__global__ void csr_count_kernel(const float* __restrict__ XT, int Np, int N, int* cnt) {
  const float* row = XT + (size_t)blockIdx.x * Np;
  int c = 0;
  for (int n0 = 0; n0 < N; n0 += blockDim.x) {
    const int n = n0 + threadIdx.x;
    c += __syncthreads_count(n < N && row[n] != 0.0f);
  }
  if (threadIdx.x == 0) cnt[blockIdx.x] = c;
}

// One CTA per feature; block-wide compaction keeps entries in ascending sample order.
__global__ void csr_fill_kernel(const float* __restrict__ XT, int Np, int N, const int* off,
                                int* xs_n, float* xs_v) {
  __shared__ int wcount[32];
  __shared__ int s_base;
  const float* row = XT + (size_t)blockIdx.x * Np;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  if (threadIdx.x == 0) s_base = off[blockIdx.x];
  __syncthreads();
  for (int n0 = 0; n0 < N; n0 += blockDim.x) {
    const int n = n0 + threadIdx.x;
    const float v = n < N ? row[n] : 0.0f;
    const bool nz = v != 0.0f;
    const unsigned int m = __ballot_sync(0xffffffffu, nz);
    if (lane == 0) wcount[warp] = __popc(m);
    __syncthreads();
    int before = 0, tot = 0;
    for (int w = 0; w < nw; ++w) {
      if (w < warp) before += wcount[w];
      tot += wcount[w];
    }
    const int pos = s_base + before + __popc(m & ((1u << lane) - 1u));
    if (nz) {
      xs_n[pos] = n;
      xs_v[pos] = v;
    }
    __syncthreads();
    if (threadIdx.x == 0) s_base += tot;
    __syncthreads();
  }
}

// Distinct 32-byte sectors (8 samples) of a z1 row holding feature i's entries.
__global__ void csr_sectors_kernel(const int* __restrict__ off, const int* __restrict__ xs_n,
                                   int* sect) {
  const int s = off[blockIdx.x], e = off[blockIdx.x + 1];
  int c = 0;
  for (int p0 = s; p0 < e; p0 += blockDim.x) {
    const int p = p0 + threadIdx.x;
    c += __syncthreads_count(p < e && (p == s || (xs_n[p] >> 3) != (xs_n[p - 1] >> 3)));
  }
  if (threadIdx.x == 0) sect[blockIdx.x] = c;
}

__global__ void count_nonfinite_kernel(const float* __restrict__ p, size_t n, int* out) {
  int bad = 0;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x)
    bad |= !isfinite(p[i]);
  if (__syncthreads_or(bad) && threadIdx.x == 0) atomicOr(out, 1);
}

__global__ void init_layer_kernel(int wkind, float scale, const float* __restrict__ src,
                                  const signed char* __restrict__ mask, size_t n, float* w_eff,
                                  signed char* code, float* wfix) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x) {
    const float v = src[i];
    if (wkind == MCA_W_TERNARY_I8) {
      const int t = (int)v;
      code[i] = (signed char)t;
      w_eff[i] = __fmul_rn(scale, (float)t);
    } else if (wkind == MCA_W_MASKED_FP32) {
      const int m = mask ? (mask[i] != 0) : 1;
      wfix[i] = v;
      code[i] = (signed char)m;
      w_eff[i] = m ? v : 0.0f;
    } else {
      w_eff[i] = v;
    }
  }
}

// C[M x Ncol] = A[M x K] * B[K x Ncol], row-major, fp32 FMA in ascending k. Ncol % 128 == 0,
// ldb and ldc multiples of 4. 128x128 tile per CTA, 256 threads, 8x8 outputs per thread.
__global__ void __launch_bounds__(256) sgemm_nn_kernel(int M, int Ncol, int K,
                                                       const float* __restrict__ A, int lda,
                                                       const float* __restrict__ B, int ldb,
                                                       float* __restrict__ C, int ldc) {
  constexpr int BM = 128, BN = 128, BK = 8;
  __shared__ __align__(16) float As[BK][BM];
  __shared__ __align__(16) float Bs[BK][BN];
  const int tid = threadIdx.x;
  const int bm = blockIdx.y * BM, bn = blockIdx.x * BN;
  const int tr = tid / 16, tc = tid % 16;
  float acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.0f;
  const int arow = tid / 2, akk = (tid % 2) * 4;
  const int bkk = tid / 32, bcol = (tid % 32) * 4;
  for (int k0 = 0; k0 < K; k0 += BK) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int m = bm + arow, kk = k0 + akk + q;
      As[akk + q][arow] = (m < M && kk < K) ? A[(size_t)m * lda + kk] : 0.0f;
    }
    {
      const int kk = k0 + bkk;
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (kk < K) v = *reinterpret_cast<const float4*>(B + (size_t)kk * ldb + bn + bcol);
      *reinterpret_cast<float4*>(&Bs[bkk][bcol]) = v;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      float ra[8], rb[8];
      const float4 a0 = *reinterpret_cast<const float4*>(&As[kk][tr * 4]);
      const float4 a1 = *reinterpret_cast<const float4*>(&As[kk][64 + tr * 4]);
      const float4 b0 = *reinterpret_cast<const float4*>(&Bs[kk][tc * 4]);
      const float4 b1 = *reinterpret_cast<const float4*>(&Bs[kk][64 + tc * 4]);
      ra[0] = a0.x; ra[1] = a0.y; ra[2] = a0.z; ra[3] = a0.w;
      ra[4] = a1.x; ra[5] = a1.y; ra[6] = a1.z; ra[7] = a1.w;
      rb[0] = b0.x; rb[1] = b0.y; rb[2] = b0.z; rb[3] = b0.w;
      rb[4] = b1.x; rb[5] = b1.y; rb[6] = b1.z; rb[7] = b1.w;
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(ra[i], rb[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int m = bm + (i < 4 ? tr * 4 + i : 64 + tr * 4 + (i - 4));
    if (m >= M) continue;
    float* crow = C + (size_t)m * ldc + bn;
    *reinterpret_cast<float4*>(crow + tc * 4) =
        make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
    *reinterpret_cast<float4*>(crow + 64 + tc * 4) =
        make_float4(acc[i][4], acc[i][5], acc[i][6], acc[i][7]);
  }
}

// Output fields z2[:, n] = W2 f(z1[:, n]) (ascending j), the sample's loss, and its label.
template <int ACT1, int ACT2, int LOSS>
__global__ void __launch_bounds__(128) mlp2_outputs_kernel(Mlp2Args a, const int* __restrict__ y) {
  constexpr int TJ = 64;
  __shared__ float w2s[kMaxC][TJ];
  const int n = blockIdx.x * blockDim.x + threadIdx.x;
  float acc[kMaxC];
#pragma unroll
  for (int k = 0; k < kMaxC; ++k) acc[k] = 0.0f;
  for (int j0 = 0; j0 < a.H; j0 += TJ) {
    __syncthreads();
    for (int t = threadIdx.x; t < kMaxC * TJ; t += blockDim.x) {
      const int k = t / TJ, jj = t % TJ;
      w2s[k][jj] = (k < a.C && j0 + jj < a.H) ? a.w2[(size_t)k * a.H + j0 + jj] : 0.0f;
    }
    __syncthreads();
    if (n < a.N) {
      const int jn = min(TJ, a.H - j0);
      for (int jj = 0; jj < jn; ++jj) {
        const float av = act<ACT1>(a.z1[(size_t)(j0 + jj) * a.Np + n], a.g1, a.act1);
#pragma unroll
        for (int k = 0; k < kMaxC; ++k)
          if (k < a.C) acc[k] = fmaf(w2s[k][jj], av, acc[k]);
      }
    }
  }
  if (n < a.N) {
    const int yn = y[n];
    const float ln = sample_loss<ACT2, LOSS, kMaxC>(acc, a.C, yn, a.g2, a.act2, a.loss);
    store_srec(a.srec, n, acc, ln, yn);
  }
}

// S = sum_n loss_n in fp64, one CTA, fixed order.
__global__ void __launch_bounds__(1024) sum_loss_kernel(const float* __restrict__ srec, int N,
                                                        DevState* st) {
  __shared__ double red[32];
  double s = 0.0;
  for (int n = threadIdx.x; n < N; n += blockDim.x) s += (double)srec[(size_t)n * kSR + kSR - 2];
  s = block_sum_d(s, red);
  if (threadIdx.x == 0) st->S = s;
}

// ------------------------------------------------------------------------------------------------
// Launchers
// ------------------------------------------------------------------------------------------------
cudaError_t launch_transpose_pad(const float* X, int N, int D, float* XT, int Np, cudaStream_t s) {
  dim3 grid((Np + 31) / 32, (D + 31) / 32), block(32, 8);
  transpose_pad_kernel<<<grid, block, 0, s>>>(X, N, D, XT, Np);
  return cudaGetLastError();
}

cudaError_t launch_csr_count(const float* XT, int Np, int N, int D, int* cnt, cudaStream_t s) {
  csr_count_kernel<<<D, 256, 0, s>>>(XT, Np, N, cnt);
  return cudaGetLastError();
}

cudaError_t launch_csr_fill(const float* XT, int Np, int N, int D, const int* off, int* xs_n,
                            float* xs_v, cudaStream_t s) {
  csr_fill_kernel<<<D, 1024, 0, s>>>(XT, Np, N, off, xs_n, xs_v);
  return cudaGetLastError();
}

cudaError_t launch_csr_sectors(const int* off, const int* xs_n, int D, int* sect, cudaStream_t s) {
  csr_sectors_kernel<<<D, 256, 0, s>>>(off, xs_n, sect);
  return cudaGetLastError();
}

cudaError_t launch_count_nonfinite(const float* p, size_t n, int* out, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  const int grid = (int)std::min<size_t>(4096, (n + 255) / 256);
  count_nonfinite_kernel<<<grid, 256, 0, s>>>(p, n, out);
  return cudaGetLastError();
}

cudaError_t launch_init_layer(int wkind, float scale, const float* src, const signed char* mask,
                              size_t n, float* w_eff, signed char* code, float* wfix,
                              cudaStream_t s) {
  const int grid = (int)std::min<size_t>(4096, (n + 255) / 256);
  init_layer_kernel<<<grid, 256, 0, s>>>(wkind, scale, src, mask, n, w_eff, code, wfix);
  return cudaGetLastError();
}

cudaError_t launch_sgemm_nn(int M, int Ncol, int K, const float* A, int lda, const float* B,
                            int ldb, float* C, int ldc, cudaStream_t s) {
  dim3 grid(Ncol / 128, (M + 127) / 128);
  sgemm_nn_kernel<<<grid, 256, 0, s>>>(M, Ncol, K, A, lda, B, ldb, C, ldc);
  return cudaGetLastError();
}

cudaError_t launch_sum_loss(const float* srec, int N, DevState* st, cudaStream_t s) {
  sum_loss_kernel<<<1, 1024, 0, s>>>(srec, N, st);
  return cudaGetLastError();
}

// Kernel variants: (tanh, sigmoid, MSE), (tanh, identity, CE), (Gaussian, sigmoid, MSE), and a
// generic one that switches on the transfer functions and loss at run time.
using LoopFn = void (*)(Mlp2Args);
using OutFn = void (*)(Mlp2Args, const int*);

static void pick(const Mlp2Args& a, LoopFn* loop, OutFn* out) {
  if (a.act1 == MCA_ACT_TANH && a.act2 == MCA_ACT_SIGMOID && a.loss == MCA_LOSS_MSE_ONEHOT) {
    *loop = mlp2_trial_loop<MCA_ACT_TANH, MCA_ACT_SIGMOID, MCA_LOSS_MSE_ONEHOT>;
    *out = mlp2_outputs_kernel<MCA_ACT_TANH, MCA_ACT_SIGMOID, MCA_LOSS_MSE_ONEHOT>;
  } else if (a.act1 == MCA_ACT_TANH && a.act2 == MCA_ACT_IDENTITY &&
             a.loss == MCA_LOSS_SOFTMAX_CE) {
    *loop = mlp2_trial_loop<MCA_ACT_TANH, MCA_ACT_IDENTITY, MCA_LOSS_SOFTMAX_CE>;
    *out = mlp2_outputs_kernel<MCA_ACT_TANH, MCA_ACT_IDENTITY, MCA_LOSS_SOFTMAX_CE>;
  } else if (a.act1 == MCA_ACT_GAUSSIAN && a.act2 == MCA_ACT_SIGMOID &&
             a.loss == MCA_LOSS_MSE_ONEHOT) {
    *loop = mlp2_trial_loop<MCA_ACT_GAUSSIAN, MCA_ACT_SIGMOID, MCA_LOSS_MSE_ONEHOT>;
    *out = mlp2_outputs_kernel<MCA_ACT_GAUSSIAN, MCA_ACT_SIGMOID, MCA_LOSS_MSE_ONEHOT>;
  } else {
    *loop = mlp2_trial_loop<-1, -1, -1>;
    *out = mlp2_outputs_kernel<-1, -1, -1>;
  }
}

cudaError_t launch_mlp2_outputs(const Mlp2Args& a, const int* y, cudaStream_t s) {
  LoopFn loop;
  OutFn out;
  pick(a, &loop, &out);
  out<<<(a.N + 127) / 128, 128, 0, s>>>(a, y);
  return cudaGetLastError();
}

int mlp2_loop_max_grid(const Mlp2Args& a, int num_sms) {
  LoopFn loop;
  OutFn out;
  pick(a, &loop, &out);
  int occ = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, loop, kLoopThreads, 0) != cudaSuccess)
    return 0;
  return occ * num_sms;
}

cudaError_t launch_mlp2_loop(const Mlp2Args& a, int grid, cudaStream_t s) {
  LoopFn loop;
  OutFn out;
  pick(a, &loop, &out);
  Mlp2Args args = a;
  void* params[] = {&args};
  return cudaLaunchCooperativeKernel((const void*)loop, dim3(grid), dim3(kLoopThreads), params, 0,
                                     s);
}

}  // namespace mca
