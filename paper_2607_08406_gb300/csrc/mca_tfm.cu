// Character-level Transformer path of the MCA trial loop (Section 2.5): pre-LN GPT blocks.
//
// One CTA recomputes one sequence (T tokens x d features) from the first stage the mutated
// parameter feeds, with the residual stream, the per-head queries / keys / values, the attention
// probabilities and the FFN hidden chunk all in shared memory:
//   x = tok_emb[token] + pos_emb[t]                                  (stage 0)
//   per block:  h = LN1(x);  x += Wo concat_h softmax(q k^T / sqrt(dh), causal) v + bo
//               h = LN2(x);  x += W2 act(W1 h + b1) + b2
//   final:      logits = W_head LNf(x) + b_head;  loss = sum_t CE(logits_t, next token)
// Parameters are read from the flat array through a one-element patch (index midx reads mval), so a
// candidate's forward is exactly the forward with W'. The residual stream entering every block is
// cached per sequence; a rejected candidate writes nothing.
//
// Per batch: tfm_eval (grid K x B, one partial loss change per candidate and sequence), tfm_decide
// (one CTA, fixed-order sums, Eq. 6 or Eq. 7), tfm_commit (grid B: the accepted candidate with
// writes).
#include <algorithm>
#include <cstdio>

#include "mca_device.cuh"
#include "mca_internal.h"
#include "mca_tfm.cuh"

namespace mca {

__host__ __device__ inline int tfm_region_floats(int T, int /*d*/, int dh, int V) {
  const int att = T * dh + T * (dh + 1) + T * dh + T * T;
  const int ffn = T * kTfmFC;
  const int head = T * V;
  return std::max(att, std::max(ffn, head));
}

size_t tfm_smem_bytes(int T, int d, int dh, int V) {
  return sizeof(float) * ((size_t)2 * T * d + tfm_region_floats(T, d, dh, V) + 16 * 128);
}

__device__ __forceinline__ float ldp(const TfmArgs& a, unsigned long long i,
                                     unsigned long long midx, float mval) {
  return i == midx ? mval : a.params[i];
}

// Row-wise layer norm of x [T][d] into h (warp per row).
__device__ __forceinline__ void ln_rows(const TfmArgs& a, const float* x, float* h,
                                        unsigned long long og, unsigned long long ob,
                                        unsigned long long midx, float mval) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int d = a.d;
  for (int t = warp; t < a.T; t += kTfmThreads / 32) {
    float s = 0.0f;
    for (int c = lane; c < d; c += 32) s += x[t * d + c];
    const float mean = warp_sum(s) / (float)d;
    float v = 0.0f;
    for (int c = lane; c < d; c += 32) {
      const float e = x[t * d + c] - mean;
      v = fmaf(e, e, v);
    }
    const float rstd = rsqrtf(warp_sum(v) / (float)d + a.eps);
    for (int c = lane; c < d; c += 32)
      h[t * d + c] = (x[t * d + c] - mean) * rstd * ldp(a, og + c, midx, mval) +
                     ldp(a, ob + c, midx, mval);
  }
}

// acc[i][j] += sum_k A[(w + 16 i) * lda + k] * W(n = lane + 32 j, k) for rows < M, n < N, k < K;
// W(n, k) = params[wbase + n * ldw + k] (patched). The tile of W is staged in Ws [16][128].
template <int NJ>
__device__ __forceinline__ void gemm_w(const TfmArgs& a, const float* A, int lda, int M, int K,
                                       unsigned long long wbase, int ldw, int N, float* Ws,
                                       unsigned long long midx, float mval,
                                       float (&acc)[4][NJ]) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int k0 = 0; k0 < K; k0 += 16) {
    const int kn = min(16, K - k0);
    for (int e = tid; e < 16 * N; e += kTfmThreads) {
      const int n = e >> 4, kk = e & 15;
      Ws[kk * 128 + n] =
          kk < kn ? ldp(a, wbase + (unsigned long long)n * ldw + k0 + kk, midx, mval) : 0.0f;
    }
    __syncthreads();
    for (int kk = 0; kk < kn; ++kk) {
      float av[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int r = warp + 16 * i;
        av[i] = r < M ? A[r * lda + k0 + kk] : 0.0f;
      }
#pragma unroll
      for (int j = 0; j < NJ; ++j) {
        const float wv = Ws[kk * 128 + lane + 32 * j];
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[i][j] = fmaf(av[i], wv, acc[i][j]);
      }
    }
    __syncthreads();
  }
}

// out[r][n] = act(acc + bias[n]) for the thread's tile (act < 0: identity); out row stride ldo.
template <int NJ>
__device__ __forceinline__ void store_tile(const TfmArgs& a, const float (&acc)[4][NJ], int M,
                                           int N, float* out, int ldo, unsigned long long bbase,
                                           int act, unsigned long long midx, float mval) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int j = 0; j < NJ; ++j) {
    const int n = lane + 32 * j;
    if (n >= N) continue;
    const float bv = ldp(a, bbase + n, midx, mval);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int r = warp + 16 * i;
      if (r >= M) continue;
      const float v = acc[i][j] + bv;
      out[r * ldo + n] = act >= 0 ? act_rt(act, v, a.g) : v;
    }
  }
}

// One pre-LN block on the residual stream xs [T][d] (in place).
__device__ void tfm_block(const TfmArgs& a, int b, float* xs, float* hs, float* R, float* Ws,
                          unsigned long long midx, float mval) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int T = a.T, d = a.d, dh = a.dh, F = a.F;
  const unsigned long long base = a.o_blk0 + (unsigned long long)b * a.blk_size;
  float* qs = R;                       // [T][dh]
  float* ks = qs + T * dh;             // [T][dh + 1]
  float* vs = ks + T * (dh + 1);       // [T][dh]
  float* ps = vs + T * dh;             // [T][T]
  const float scale = rsqrtf((float)dh);

  ln_rows(a, xs, hs, base + a.r_ln1g, base + a.r_ln1b, midx, mval);
  __syncthreads();
  float oacc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) oacc[i][j] = 0.0f;
  for (int hh = 0; hh < a.H; ++hh) {
    const unsigned long long roff = (unsigned long long)hh * dh * d;   // first row of this head
    {
      float acc[4][1] = {{0.0f}, {0.0f}, {0.0f}, {0.0f}};
      gemm_w<1>(a, hs, d, T, d, base + a.r_wq + roff, d, dh, Ws, midx, mval, acc);
      store_tile<1>(a, acc, T, dh, qs, dh, base + a.r_bq + hh * dh, -1, midx, mval);
    }
    {
      float acc[4][1] = {{0.0f}, {0.0f}, {0.0f}, {0.0f}};
      gemm_w<1>(a, hs, d, T, d, base + a.r_wk + roff, d, dh, Ws, midx, mval, acc);
      store_tile<1>(a, acc, T, dh, ks, dh + 1, base + a.r_bk + hh * dh, -1, midx, mval);
    }
    {
      float acc[4][1] = {{0.0f}, {0.0f}, {0.0f}, {0.0f}};
      gemm_w<1>(a, hs, d, T, d, base + a.r_wv + roff, d, dh, Ws, midx, mval, acc);
      store_tile<1>(a, acc, T, dh, vs, dh, base + a.r_bv + hh * dh, -1, midx, mval);
    }
    __syncthreads();
    // scores and causal softmax (warp per query row)
    {
      float sc[4][2];
#pragma unroll
      for (int i = 0; i < 4; ++i) sc[i][0] = sc[i][1] = 0.0f;
      for (int c = 0; c < dh; ++c) {
        float qv[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int t1 = warp + 16 * i;
          qv[i] = t1 < T ? qs[t1 * dh + c] : 0.0f;
        }
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const int t2 = lane + 32 * j;
          const float kv = t2 < T ? ks[t2 * (dh + 1) + c] : 0.0f;
#pragma unroll
          for (int i = 0; i < 4; ++i) sc[i][j] = fmaf(qv[i], kv, sc[i][j]);
        }
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int t1 = warp + 16 * i;
        if (t1 >= T) continue;
        float v[2];
        float m = -INFINITY;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const int t2 = lane + 32 * j;
          v[j] = (t2 <= t1 && t2 < T) ? sc[i][j] * scale : -INFINITY;
          m = fmaxf(m, v[j]);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        float e[2], s = 0.0f;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const int t2 = lane + 32 * j;
          e[j] = (t2 <= t1 && t2 < T) ? __expf(v[j] - m) : 0.0f;
          s += e[j];
        }
        s = warp_sum(s);
        const float inv = 1.0f / s;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const int t2 = lane + 32 * j;
          if (t2 < T) ps[t1 * T + t2] = e[j] * inv;
        }
      }
    }
    __syncthreads();
    // attention output of the head into qs (queries are no longer needed)
    {
      float av[4][2];
#pragma unroll
      for (int i = 0; i < 4; ++i) av[i][0] = av[i][1] = 0.0f;
      for (int t2 = 0; t2 < T; ++t2) {
        float pv[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int t1 = warp + 16 * i;
          pv[i] = t1 < T ? ps[t1 * T + t2] : 0.0f;
        }
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const int c = lane + 32 * j;
          const float vv = c < dh ? vs[t2 * dh + c] : 0.0f;
#pragma unroll
          for (int i = 0; i < 4; ++i) av[i][j] = fmaf(pv[i], vv, av[i][j]);
        }
      }
      __syncthreads();
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int t1 = warp + 16 * i;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const int c = lane + 32 * j;
          if (t1 < T && c < dh) qs[t1 * dh + c] = av[i][j];
        }
      }
    }
    __syncthreads();
    // output projection of this head's slice: oacc += att_h Wo[:, hh dh : (hh+1) dh]^T
    gemm_w<4>(a, qs, dh, T, dh, base + a.r_wo + (unsigned long long)hh * dh, d, d, Ws, midx, mval,
              oacc);
  }
  // residual
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int c = lane + 32 * j;
    if (c >= d) continue;
    const float bo = ldp(a, base + a.r_bo + c, midx, mval);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int t = warp + 16 * i;
      if (t < T) xs[t * d + c] += oacc[i][j] + bo;
    }
  }
  __syncthreads();
  // feed-forward network in hidden chunks of kTfmFC
  ln_rows(a, xs, hs, base + a.r_ln2g, base + a.r_ln2b, midx, mval);
  __syncthreads();
  float facc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) facc[i][j] = 0.0f;
  float* us = R;
  for (int f0 = 0; f0 < F; f0 += kTfmFC) {
    const int fc = min(kTfmFC, F - f0);
    {
      float acc[4][4];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.0f;
      gemm_w<4>(a, hs, d, T, d, base + a.r_w1 + (unsigned long long)f0 * d, d, fc, Ws, midx, mval,
                acc);
      store_tile<4>(a, acc, T, fc, us, kTfmFC, base + a.r_b1 + f0, a.act, midx, mval);
    }
    __syncthreads();
    gemm_w<4>(a, us, kTfmFC, T, fc, base + a.r_w2 + f0, F, d, Ws, midx, mval, facc);
  }
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int c = lane + 32 * j;
    if (c >= d) continue;
    const float b2 = ldp(a, base + a.r_b2 + c, midx, mval);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int t = warp + 16 * i;
      if (t < T) xs[t * d + c] += facc[i][j] + b2;
    }
  }
  __syncthreads();
}

template <int MODE>
__global__ void __launch_bounds__(kTfmThreads, 1) tfm_seq_kernel(TfmArgs a) {
  extern __shared__ __align__(16) float sm[];
  __shared__ DeepCand s_c;
  __shared__ int s_tok[kTfmMaxT + 1];
  __shared__ float s_rowv[kTfmMaxT];
  __shared__ int s_skip;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int T = a.T, d = a.d, V = a.V;
  float* xs = sm;
  float* hs = xs + T * d;
  float* R = hs + T * d;
  float* Ws = R + tfm_region_floats(T, d, a.dh, V);
  const int k = MODE == kTfmEval ? blockIdx.x : 0;
  const int s = MODE == kTfmEval ? blockIdx.y : blockIdx.x;
  if (MODE == kTfmCommit && a.ctl->kstar < 0) return;
  if (tid == 0) {
    if (MODE == kTfmEval) {
      s_c = tfm_candidate(a, k);
    } else if (MODE == kTfmCommit) {
      s_c = a.ctl->acc;
    } else {
      DeepCand c;
      c.idx = 0xffffffffu;
      c.layer = -1;
      c.row = -1;
      c.col = 0;
      c.oldw = c.neww = 0.0f;
      c.delta = 1.0f;
      c.new_code = 0;
      c.valid = 1;
      s_c = c;
    }
  }
  for (int t = tid; t <= T; t += kTfmThreads) s_tok[t] = a.tokens[(size_t)s * (T + 1) + t];
  __syncthreads();
  const DeepCand c = s_c;
  float* part = a.partial + (size_t)k * a.B + s;
  if (!c.valid || c.delta == 0.0f) {
    if (MODE == kTfmEval && tid == 0) *part = 0.0f;
    return;
  }
  if (MODE != kTfmForward && c.row >= 0) {     // a tok_emb entry: sequences without that token
    if (tid == 0) {
      int skip = 1;
      for (int t = 0; t < T; ++t) skip &= s_tok[t] != c.row;
      s_skip = skip;
    }
    __syncthreads();
    if (s_skip) {
      if (MODE == kTfmEval && tid == 0) *part = 0.0f;
      return;
    }
  }
  const unsigned long long midx = MODE == kTfmForward ? ~0ull : (unsigned long long)c.idx;
  const float mval = c.neww;
  const size_t seq_stride = (size_t)T * d;
  int b0;
  if (MODE == kTfmForward || c.layer < 0) {
    b0 = 0;
    for (int e = tid; e < T * d; e += kTfmThreads) {
      const int t = e / d, cc = e - t * d;
      xs[e] = ldp(a, a.o_tok + (unsigned long long)s_tok[t] * d + cc, midx, mval) +
              ldp(a, a.o_pos + (unsigned long long)t * d + cc, midx, mval);
    }
    if (MODE != kTfmEval) {
      float* dst = a.X + (size_t)s * seq_stride;
      __syncthreads();
      for (int e = tid; e < T * d; e += kTfmThreads) dst[e] = xs[e];
    }
  } else {
    b0 = c.layer;
    const float* src = a.X + ((size_t)b0 * a.B + s) * seq_stride;
    for (int e = tid; e < T * d; e += kTfmThreads) xs[e] = src[e];
  }
  __syncthreads();
  for (int b = b0; b < a.nL; ++b) {
    tfm_block(a, b, xs, hs, R, Ws, midx, mval);
    if (MODE != kTfmEval) {
      float* dst = a.X + ((size_t)(b + 1) * a.B + s) * seq_stride;
      for (int e = tid; e < T * d; e += kTfmThreads) dst[e] = xs[e];
    }
  }
  // final layer norm, head, next-character cross-entropy
  ln_rows(a, xs, hs, a.o_lnf_g, a.o_lnf_b, midx, mval);
  __syncthreads();
  {
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] = 0.0f;
    gemm_w<4>(a, hs, d, T, d, a.o_wh, d, V, Ws, midx, mval, acc);
    store_tile<4>(a, acc, T, V, R, V, a.o_bh, -1, midx, mval);
  }
  __syncthreads();
  for (int t = warp; t < T; t += kTfmThreads / 32) {
    const float* z = R + t * V;
    float m = -INFINITY;
    for (int v = lane; v < V; v += 32) m = fmaxf(m, z[v]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float se = 0.0f;
    for (int v = lane; v < V; v += 32) se += __expf(z[v] - m);
    se = warp_sum(se);
    if (lane == 0) s_rowv[t] = (__logf(se) + m) - z[s_tok[t + 1]];
  }
  __syncthreads();
  if (tid == 0) {
    float l = 0.0f;
    for (int t = 0; t < T; ++t) l += s_rowv[t];
    if (MODE == kTfmEval)
      *part = l - a.ell[s];
    else
      a.ell[s] = l;
  }
}

// FLOPs of recomputing one sequence from stage b0 (-1 = embeddings) to the loss; restart: where
// the tensor-core kernels start inside block b0 (kRestartFfn: its feed-forward sub-block;
// kRestartUnit: block b0 + 1, the rank-1 step before it not counted).
__device__ __forceinline__ unsigned long long tfm_seq_flops(const TfmArgs& a, int b0, int restart) {
  const unsigned long long T = a.T, d = a.d, F = a.F, H = a.H, dh = a.dh, V = a.V;
  const unsigned long long attn = 3ull * T * d * d + 2ull * H * T * T * dh + T * d * d;
  const unsigned long long blk = attn + 2ull * T * d * F;
  int nb = a.nL - (b0 < 0 ? 0 : b0);
  if (restart == kRestartUnit) --nb;
  return 2ull * ((unsigned long long)(nb > 0 ? nb : 0) * blk -
                 (restart == kRestartFfn ? attn : 0ull) + T * d * V);
}

// One CTA: dS per candidate (fixed order over sequences, compensated fp32), the decision (Eq. 6),
// trace, statistics and the accepted parameter's new value.
__global__ void __launch_bounds__(kKmax) tfm_decide_kernel(TfmArgs a) {
  __shared__ DeepCand s_c[kKmax];
  __shared__ float s_dS[kKmax];
  __shared__ int s_take[kKmax];
  __shared__ float s_sum[kKmax];
  __shared__ float s_buf[(kKmax / 32) * 256];
  __shared__ unsigned int s_macc[kKmax / 32], s_mbad[kKmax / 32], s_mforced[kKmax / 32];
  const int k = threadIdx.x, lane = k & 31, warp = k >> 5;
  const unsigned long long tau = tfm_batch_tau(a);
  const int Kb = tfm_batch_width(a, tau);
  bool acc = false, bad = false, forced = false;
  if (k < Kb) {
    const DeepCand c = tfm_candidate(a, k);
    s_c[k] = c;
    s_take[k] = c.valid && c.delta != 0.0f;
  }
  __syncthreads();
  ordered_row_sums(a.partial, a.B, Kb, s_take, s_sum, s_buf);
  if (k < Kb) {
    const DeepCand c = s_c[k];
    const float d = c.valid ? s_sum[k] : __int_as_float(0x7fc00000);
    s_dS[k] = d;
    if (a.n_explicit > 0) {
      a.ex_out[k] = (double)d;
    } else if (c.valid) {
      const unsigned long long tk = tau + (unsigned long long)k;
      bool facc = false;
      if (a.nforce > 0) {
        int lo2 = 0, hi2 = a.nforce;
        while (lo2 < hi2) {
          const int mid = (lo2 + hi2) >> 1;
          if (a.ftau[mid] < tk)
            lo2 = mid + 1;
          else
            hi2 = mid;
        }
        if (lo2 < a.nforce && a.ftau[lo2] == tk) {
          forced = true;
          facc = a.facc[lo2] != 0;
        }
      }
      if (forced) {
        acc = facc;
      } else {
        bad = !isfinite(d);
        acc = accept_change(d, a.strict, a.metro, a.seed, tk, a.msc);
      }
    }
  }
  if (a.n_explicit > 0) return;
  const unsigned int ma = __ballot_sync(0xffffffffu, acc);
  const unsigned int mb = __ballot_sync(0xffffffffu, bad);
  const unsigned int mf = __ballot_sync(0xffffffffu, forced);
  if (lane == 0) {
    s_macc[warp] = ma;
    s_mbad[warp] = mb;
    s_mforced[warp] = mf;
  }
  __syncthreads();
  if (k != 0) return;
  int kstar = -1, kbad = -1;
  for (int w = 0; w < kKmax / 32 && kstar < 0; ++w)
    if (s_macc[w]) kstar = w * 32 + __ffs(s_macc[w]) - 1;
  for (int w = 0; w < kKmax / 32 && kbad < 0; ++w)
    if (s_mbad[w]) kbad = w * 32 + __ffs(s_mbad[w]) - 1;
  if (kbad >= 0 && (kstar < 0 || kbad <= kstar)) kstar = -2;
  DevState* st = a.st;
  const int last = kstar >= 0 ? kstar : Kb - 1;
  if (a.trace_cap > 0 && kstar != -2) {
    const double S = st->S;
    for (int q = 0; q <= last; ++q) {
      mca_trace_rec rec;
      rec.tau = tau + (unsigned long long)q;
      rec.idx = s_c[q].idx;
      rec.accept = q == kstar ? 1 : 0;
      rec.old_w = s_c[q].oldw;
      rec.new_w = s_c[q].neww;
      rec.valid = s_c[q].valid;
      rec.forced = (int)((s_mforced[q >> 5] >> (q & 31)) & 1u);
      rec.dS = (double)s_dS[q];
      rec.S = S;
      a.trace[st->trace_written % (unsigned long long)a.trace_cap] = rec;
      st->trace_written += 1ull;
    }
  }
  DeepCtl* ctl = a.ctl;
  ctl->kstar = kstar;
  if (kstar == -2) {
    atomicCAS(&st->err, 0, (int)MCA_ERR_NUMERIC);
    ctl->consumed = 0;
    return;
  }
  if (Kb == 0) {                 // a batch past the end of a run whose batches run ahead
    ctl->consumed = 0;
    return;
  }
  for (int w = 0; w < kKmax / 32; ++w) {
    unsigned int m = s_mforced[w];
    const int hi = last - w * 32;
    if (hi < 31) m &= hi < 0 ? 0u : ((2u << hi) - 1u);
    if (m) atomicAdd(&st->forced, (unsigned long long)__popc(m));
  }
  // (the statistics below are reductions without a returned value, so this thread does not wait
  // for their reads)
  unsigned long long ncand = 0, flops = 0;
  for (int q = 0; q < Kb; ++q) {
    ncand += s_c[q].valid ? 1ull : 0ull;
    if (s_c[q].valid && s_c[q].delta != 0.0f)
      flops += tfm_seq_flops(a, s_c[q].layer,
                             a.tc ? tfm_restart(a, s_c[q].idx, s_c[q].layer) : kRestartBlock) *
               (unsigned long long)a.B;
  }
  atomicAdd(&st->candidates, ncand);
  atomicAdd(&st->alg_flops, flops);
  atomicAdd(&st->batches, 1ull);
  if (kstar >= 0) {
    const DeepCand& c = s_c[kstar];
    ctl->acc = c;
    ctl->consumed = kstar + 1;
    atomicAdd(&st->trials, (unsigned long long)(kstar + 1));
    atomicAdd(&st->accepts, 1ull);
    atomicAdd(&st->wasted, (unsigned long long)(Kb - kstar - 1));
    atomicAdd(&st->S, (double)s_dS[kstar]);
    a.params[c.idx] = c.neww;
  } else {
    ctl->consumed = Kb;
    atomicAdd(&st->trials, (unsigned long long)Kb);
  }
  if (a.tau_dev) *a.tau_dev = tau + (unsigned long long)(kstar >= 0 ? kstar + 1 : Kb);
}

template <int MODE>
static cudaError_t launch_seq(const TfmArgs& a, dim3 grid, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute((const void*)tfm_seq_kernel<MODE>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)a.smem);
  if (e != cudaSuccess) return e;
  tfm_seq_kernel<MODE><<<grid, kTfmThreads, a.smem, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_tfm_eval(const TfmArgs& a, cudaStream_t s) {
  if (a.tc) return launch_tfm_tc_eval(a, s);
  const int Kb = a.n_explicit > 0 ? a.n_explicit : a.Kb;
  return launch_seq<kTfmEval>(a, dim3(Kb, a.B), s);
}

cudaError_t launch_tfm_commit(const TfmArgs& a, cudaStream_t s) {
  if (a.tc) return launch_tfm_tc_commit(a, s);
  return launch_seq<kTfmCommit>(a, dim3(a.B), s);
}

cudaError_t launch_tfm_forward(const TfmArgs& a, cudaStream_t s) {
  if (a.tc) return launch_tfm_tc_forward(a, s);
  return launch_seq<kTfmForward>(a, dim3(a.B), s);
}

cudaError_t launch_tfm_decide(const TfmArgs& a, cudaStream_t s) {
  tfm_decide_kernel<<<1, kKmax, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace mca
