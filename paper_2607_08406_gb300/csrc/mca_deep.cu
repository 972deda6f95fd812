// Deep MLP path of the MCA trial loop (three or more weight layers; the 24 x 256 tanh net).
//
// Cached state: the fields Z_l = W_l a_{l-1} of every layer for all samples ([n_out x Np],
// feature-major) and every sample's loss. A candidate W_l[j, i] -> W_l[j, i] + delta changes
//   row j of layer l:      z'_l[j, n]  = z_l[j, n] + delta a_{l-1}[i, n]            (Section 2.4)
//   layer l+1 (rank-1):    Z'_{l+1}    = Z_{l+1} + W_{l+1}[:, j] (f(z'_l[j]) - f(z_l[j]))
//   layers m >= l+2:       Z'_m        = Z_m + W_m (f(Z'_{m-1}) - f(Z_{m-1}))
// i.e. the dense recomputation from l+2 on is carried as a change: a sample whose activations did not
// change contributes exactly zero, and the commit writes exactly what the evaluation computed.
//
// Per batch the host launches three kernels:
//   deep_eval     grid (K, tiles): CTA (k, t) runs candidate k's chain over tile t's kDeepTS samples,
//                 the change matrix staying in shared memory from layer to layer, and writes one
//                 partial loss change per (candidate, tile) -- a fixed computation, independent of K
//   deep_decide   one CTA: fixed-order (compensated fp32) sums, lowest-index candidate with
//                 dS <= theta (Eq. 6: theta = 0; Eq. 7: the trial's Metropolis threshold), trace,
//                 statistics, weight update
//   deep_commit   grid (tiles): the accepted candidate's chain with writes
#include <algorithm>
#include <cstdio>

#include "mca_deep.cuh"
#include "mca_device.cuh"
#include "mca_internal.h"

namespace mca {

template <bool COMMIT>
__global__ void __launch_bounds__(kDeepThreads) deep_chain_kernel(DeepArgs a) {
  extern __shared__ __align__(16) float sm[];
  float* Ds = sm;                                   // [kDeepMaxWidth][kDeepTS] activation changes
  float* Ws = sm + kDeepMaxWidth * kDeepTS;         // [kDeepKC][kDeepMaxWidth] weight tile
  __shared__ DeepCand s_cand;
  __shared__ float s_da[kDeepTS];
  __shared__ float s_red[32];
  const int tid = threadIdx.x;
  const int k = COMMIT ? 0 : blockIdx.x;
  const int tile = COMMIT ? blockIdx.x : blockIdx.y;
  const int n0 = tile * kDeepTS;
  if (COMMIT && a.ctl->kstar < 0) return;
  if (tid == 0) s_cand = COMMIT ? a.ctl->acc : deep_candidate(a, k);
  __syncthreads();
  const DeepCand c = s_cand;
  float* part = a.partial + (size_t)k * a.ntiles + tile;
  if (!c.valid || c.delta == 0.0f) {
    if (!COMMIT && tid == 0) *part = 0.0f;
    return;
  }
  const int L = a.L, l = c.layer, j = c.row, i = c.col;
  const int Np = a.Np, N = a.N;
  float dl = 0.0f;

  // ---- row j of layer l
  if (tid < kDeepTS) {
    const int n = n0 + tid;
    float da = 0.0f;
    if (n < N) {
      const float v = l == 0 ? a.XT[(size_t)i * Np + n]
                             : act_rt(a.act[l - 1], a.Z[l - 1][(size_t)i * Np + n], a.g[l - 1]);
      float* zp = a.Z[l] + (size_t)j * Np + n;
      const float z = *zp;
      const float zn = fmaf(c.delta, v, z);
      if (l == L - 1) {                              // an output weight: output field j changes
        float zz[kMaxC];
#pragma unroll
        for (int q = 0; q < kMaxC; ++q)
          zz[q] = q < a.C ? a.Z[l][(size_t)q * Np + n] : 0.0f;
#pragma unroll
        for (int q = 0; q < kMaxC; ++q)
          if (q == j) zz[q] = zn;
        dl = out_delta<COMMIT>(a, n, zz, zn != z);
      } else {
        da = act_rt(a.act[l], zn, a.g[l]) - act_rt(a.act[l], z, a.g[l]);
        if (COMMIT) *zp = zn;
      }
    }
    s_da[tid] = da;
  }
  __syncthreads();

  if (l < L - 1) {
    // ---- layer l+1: rank-1 change through column j of W_{l+1}
    const int m1 = l + 1;
    const float* W1 = a.w[m1];
    const int K1 = a.n_in[m1];
    if (m1 == L - 1) {
      if (tid < kDeepTS) {
        const int n = n0 + tid;
        const float da = s_da[tid];
        if (n < N && da != 0.0f) {
          float zz[kMaxC];
          bool changed = false;
#pragma unroll
          for (int q = 0; q < kMaxC; ++q) {
            if (q < a.C) {
              const float zo = a.Z[m1][(size_t)q * Np + n];
              zz[q] = fmaf(W1[(size_t)q * K1 + j], da, zo);
              changed |= zz[q] != zo;
            } else {
              zz[q] = 0.0f;
            }
          }
          dl = out_delta<COMMIT>(a, n, zz, changed);
        }
      }
    } else {
      const int M = a.n_out[m1];
      for (int e = tid; e < M * kDeepTS; e += kDeepThreads) {
        const int r = e / kDeepTS, t = e - r * kDeepTS, n = n0 + t;
        const float da = s_da[t];
        float d = 0.0f;
        if (n < N && da != 0.0f) {
          float* zp = a.Z[m1] + (size_t)r * Np + n;
          const float zo = *zp;
          const float zn = fmaf(W1[(size_t)r * K1 + j], da, zo);
          if (COMMIT) *zp = zn;
          d = act_rt(a.act[m1], zn, a.g[m1]) - act_rt(a.act[m1], zo, a.g[m1]);
        }
        Ds[r * kDeepTS + t] = d;
      }
      __syncthreads();

      // ---- layers l+2 .. L-2: Z'_m = Z_m + W_m D, D <- f(Z'_m) - f(Z_m)
      const int ty = tid >> 4, tx = tid & 15;
      for (int m = l + 2; m < L - 1; ++m) {
        const float* Wm = a.w[m];
        const int Mm = a.n_out[m], Km = a.n_in[m];
        float acc[16][4];
#pragma unroll
        for (int q = 0; q < 16; ++q)
#pragma unroll
          for (int cc = 0; cc < 4; ++cc) acc[q][cc] = 0.0f;
        for (int k0 = 0; k0 < Km; k0 += kDeepKC) {
          const int kn = min(kDeepKC, Km - k0);
          if (tid < Mm) {
            const float* src = Wm + (size_t)tid * Km + k0;
            if (kn == kDeepKC && (Km & 3) == 0) {
#pragma unroll
              for (int v4 = 0; v4 < kDeepKC / 4; ++v4) {
                const float4 w4 = *reinterpret_cast<const float4*>(src + 4 * v4);
                Ws[(4 * v4 + 0) * kDeepMaxWidth + tid] = w4.x;
                Ws[(4 * v4 + 1) * kDeepMaxWidth + tid] = w4.y;
                Ws[(4 * v4 + 2) * kDeepMaxWidth + tid] = w4.z;
                Ws[(4 * v4 + 3) * kDeepMaxWidth + tid] = w4.w;
              }
            } else {
              for (int kk = 0; kk < kn; ++kk) Ws[kk * kDeepMaxWidth + tid] = src[kk];
            }
          }
          __syncthreads();
          for (int kk = 0; kk < kn; ++kk) {
            const float4 b = *reinterpret_cast<const float4*>(&Ds[(k0 + kk) * kDeepTS + tx * 4]);
            const float* wr = &Ws[kk * kDeepMaxWidth + ty * 16];
            float av[16];
#pragma unroll
            for (int v4 = 0; v4 < 4; ++v4) {
              const float4 w4 = *reinterpret_cast<const float4*>(wr + 4 * v4);
              av[4 * v4 + 0] = w4.x;
              av[4 * v4 + 1] = w4.y;
              av[4 * v4 + 2] = w4.z;
              av[4 * v4 + 3] = w4.w;
            }
#pragma unroll
            for (int q = 0; q < 16; ++q) {
              acc[q][0] = fmaf(av[q], b.x, acc[q][0]);
              acc[q][1] = fmaf(av[q], b.y, acc[q][1]);
              acc[q][2] = fmaf(av[q], b.z, acc[q][2]);
              acc[q][3] = fmaf(av[q], b.w, acc[q][3]);
            }
          }
          __syncthreads();
        }
        // epilogue: new fields and the next change matrix (rows >= Mm are never read)
        float* Zm = a.Z[m];
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          const int r = ty * 16 + q;
          if (r < Mm) {
            const int t0 = tx * 4;
            const float4 zo4 = *reinterpret_cast<const float4*>(Zm + (size_t)r * Np + n0 + t0);
            const float zo[4] = {zo4.x, zo4.y, zo4.z, zo4.w};
#pragma unroll
            for (int cc = 0; cc < 4; ++cc) {
              const int n = n0 + t0 + cc;
              const float zn = zo[cc] + acc[q][cc];
              float d = 0.0f;
              if (n < N && zn != zo[cc]) {
                d = act_rt(a.act[m], zn, a.g[m]) - act_rt(a.act[m], zo[cc], a.g[m]);
                if (COMMIT) Zm[(size_t)r * Np + n] = zn;
              }
              Ds[r * kDeepTS + t0 + cc] = d;
            }
          }
        }
        __syncthreads();
      }

      // ---- output layer: Z'_{L-1} = Z_{L-1} + W_{L-1} D, loss
      {
        const int mo = L - 1;
        const int Ko = a.n_in[mo];
        const float* Wo = a.w[mo];
        for (int e = tid; e < a.C * Ko; e += kDeepThreads) Ws[e] = Wo[e];
        __syncthreads();
        if (tid < kDeepTS) {
          const int n = n0 + tid;
          if (n < N) {
            float zz[kMaxC];
            bool changed = false;
#pragma unroll
            for (int q = 0; q < kMaxC; ++q) {
              if (q < a.C) {
                float s = 0.0f;
                const float* wq = Ws + q * Ko;
                for (int kk = 0; kk < Ko; ++kk) s = fmaf(wq[kk], Ds[kk * kDeepTS + tid], s);
                const float zo = a.Z[mo][(size_t)q * Np + n];
                zz[q] = zo + s;
                changed |= zz[q] != zo;
              } else {
                zz[q] = 0.0f;
              }
            }
            dl = out_delta<COMMIT>(a, n, zz, changed);
          }
        }
      }
    }
  }
  if (!COMMIT) {
    const float tot = block_sum(dl, s_red);
    if (tid == 0) *part = tot;
  }
}

// One CTA: dS per candidate (fixed order over tiles, compensated fp32), the decision (Eq. 6),
// trace, statistics, and the accepted weight's new value.
__global__ void __launch_bounds__(kKmax) deep_decide_kernel(DeepArgs a) {
  __shared__ DeepCand s_c[kKmax];
  __shared__ float s_dS[kKmax];
  __shared__ int s_take[kKmax];
  __shared__ float s_sum[kKmax];
  __shared__ float s_buf[(kKmax / 32) * 256];
  __shared__ unsigned int s_macc[kKmax / 32], s_mbad[kKmax / 32], s_mforced[kKmax / 32];
  const int k = threadIdx.x, lane = k & 31, warp = k >> 5;
  const int Kb = a.n_explicit > 0 ? a.n_explicit : a.Kb;
  bool acc = false, bad = false, forced = false;
  if (k < Kb) {
    const DeepCand c = deep_candidate(a, k);
    s_c[k] = c;
    s_take[k] = c.valid && c.delta != 0.0f;
  }
  __syncthreads();
  ordered_row_sums(a.partial, a.ntiles, Kb, s_take, s_sum, s_buf);
  if (k < Kb) {
    const DeepCand c = s_c[k];
    const float d = c.valid ? s_sum[k] : __int_as_float(0x7fc00000);
    s_dS[k] = d;
    if (a.n_explicit > 0) {
      a.ex_out[k] = (double)d;
    } else if (c.valid) {
      const unsigned long long tk = a.tau + (unsigned long long)k;
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
      rec.tau = a.tau + (unsigned long long)q;
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
  for (int w = 0; w < kKmax / 32; ++w) {
    unsigned int m = s_mforced[w];
    const int hi = last - w * 32;
    if (hi < 31) m &= hi < 0 ? 0u : ((2u << hi) - 1u);
    if (m) atomicAdd(&st->forced, (unsigned long long)__popc(m));
  }
  // (the statistics below are reductions without a returned value, so this thread does not wait
  // for their reads)
  // FLOPs of the evaluated chains: row update (2 per sample), rank-1 into layer l+1
  // (2 n_out[l+1] per sample), dense layers m = l+2 .. L-1 (2 n_out[m] n_in[m] per sample)
  unsigned long long ncand = 0, flops = 0;
  for (int q = 0; q < Kb; ++q) {
    const DeepCand& c = s_c[q];
    ncand += c.valid ? 1ull : 0ull;
    if (!c.valid || c.delta == 0.0f) continue;
    unsigned long long per = 2ull;
    if (c.layer + 1 < a.L) per += 2ull * (unsigned long long)a.n_out[c.layer + 1];
    for (int m = c.layer + 2; m < a.L; ++m)
      per += 2ull * (unsigned long long)a.n_out[m] * (unsigned long long)a.n_in[m];
    flops += per * (unsigned long long)a.N;
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
    const int l = c.layer;
    const unsigned long long off = c.idx - a.off[l];
    a.w[l][off] = c.neww;
    if (a.wk[l] != MCA_W_FP32) a.code[l][off] = (signed char)c.new_code;
    if (a.whi[l] != nullptr) {                      // split image of the tensor-core chain
      const float h = tf32_rna(c.neww);
      const size_t o = deep_tc_image_index(c.row, c.col);
      a.whi[l][o] = h;
      a.whi[l][o + 4096] = tf32_rna(c.neww - h);
    }
  } else {
    ctl->consumed = Kb;
    atomicAdd(&st->trials, (unsigned long long)Kb);
  }
}

// Per-sample losses from the output fields, and nothing else (S is summed by sum_loss_kernel).
__global__ void deep_losses_kernel(DeepArgs a) {
  const int n = blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= a.N) return;
  const int Lo = a.L - 1;
  float zz[kMaxC];
#pragma unroll
  for (int q = 0; q < kMaxC; ++q) zz[q] = q < a.C ? a.Z[Lo][(size_t)q * a.Np + n] : 0.0f;
  a.ell[n] = sample_loss<-1, -1, kMaxC>(zz, a.C, a.y[n], a.g[Lo], a.act[Lo], a.loss);
}

static size_t chain_smem() {
  return sizeof(float) * (size_t)(kDeepMaxWidth * kDeepTS + kDeepKC * kDeepMaxWidth);
}

cudaError_t launch_deep_eval(const DeepArgs& a, cudaStream_t s) {
  if (a.tc) return launch_deep_eval_tc(a, s);
  const int Kb = a.n_explicit > 0 ? a.n_explicit : a.Kb;
  cudaError_t e = cudaFuncSetAttribute((const void*)deep_chain_kernel<false>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)chain_smem());
  if (e != cudaSuccess) return e;
  deep_chain_kernel<false><<<dim3(Kb, a.ntiles), kDeepThreads, chain_smem(), s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_deep_decide(const DeepArgs& a, cudaStream_t s) {
  deep_decide_kernel<<<1, kKmax, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_deep_commit(const DeepArgs& a, cudaStream_t s) {
  if (a.tc) return launch_deep_commit_tc(a, s);
  cudaError_t e = cudaFuncSetAttribute((const void*)deep_chain_kernel<true>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)chain_smem());
  if (e != cudaSuccess) return e;
  deep_chain_kernel<true><<<a.ntiles, kDeepThreads, chain_smem(), s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_deep_losses(const DeepArgs& a, cudaStream_t s) {
  deep_losses_kernel<<<(a.N + 127) / 128, 128, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace mca
