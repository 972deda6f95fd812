// Full forward pass of the single-hidden-layer net and the creation-time data preparation:
// X -> feature-major XT, the CSR of X by input feature (plus per-range offsets and sector counts),
// parameter initialisation, z1 = W1 X^T (SIMT SGEMM), output fields, per-sample losses and S.
#include <algorithm>
#include <cstdio>

#include "mca_device.cuh"
#include "mca_internal.h"

namespace mca {

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

// roff[i * (NR + 1) + r] = first entry of feature i whose sample is >= r * RS (binary search over
// the feature's ascending sample list); roff[i * (NR + 1) + NR] = end of the feature's entries.
__global__ void csr_range_offsets_kernel(const int* __restrict__ off, const int* __restrict__ xs_n,
                                         int NR, int RS, int* roff) {
  const int i = blockIdx.x;
  const int b = off[i], e = off[i + 1];
  for (int r = threadIdx.x; r <= NR; r += blockDim.x) {
    int lo = b, hi = e;
    if (r < NR) {
      const long long s = (long long)r * RS;
      while (lo < hi) {
        const int mid = lo + ((hi - lo) >> 1);
        if (xs_n[mid] < s)
          lo = mid + 1;
        else
          hi = mid;
      }
    } else {
      lo = e;
    }
    roff[(size_t)i * (NR + 1) + r] = lo;
  }
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
// ACTB: the B operand enters as act(B) (the previous layer's activations from its fields).
template <bool ACTB>
__global__ void __launch_bounds__(256) sgemm_nn_kernel(int M, int Ncol, int K,
                                                       const float* __restrict__ A, int lda,
                                                       const float* __restrict__ B, int ldb,
                                                       float* __restrict__ C, int ldc, int bact,
                                                       float bg) {
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
      if (kk < K) {
        v = *reinterpret_cast<const float4*>(B + (size_t)kk * ldb + bn + bcol);
        if (ACTB) {
          v.x = act_rt(bact, v.x, bg);
          v.y = act_rt(bact, v.y, bg);
          v.z = act_rt(bact, v.z, bg);
          v.w = act_rt(bact, v.w, bg);
        }
      }
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
    store_srec(a.srec, a.Np, n, acc, ln, yn);
  }
}

// S = sum_n loss_n in fp64, one CTA, fixed order.
__global__ void __launch_bounds__(1024) sum_loss_kernel(const float* __restrict__ ell, int N,
                                                        DevState* st) {
  __shared__ double red[32];
  double s = 0.0;
  for (int n = threadIdx.x; n < N; n += blockDim.x) s += (double)ell[n];
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

cudaError_t launch_csr_range_offsets(const int* off, const int* xs_n, int D, int NR, int RS,
                                     int* roff, cudaStream_t s) {
  csr_range_offsets_kernel<<<D, 256, 0, s>>>(off, xs_n, NR, RS, roff);
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
  sgemm_nn_kernel<false><<<grid, 256, 0, s>>>(M, Ncol, K, A, lda, B, ldb, C, ldc, 0, 0.0f);
  return cudaGetLastError();
}

// Fields of deep layer l from the previous layer (or X for l = 0): Z_l = W_l act_{l-1}(Z_{l-1}).
cudaError_t launch_deep_forward_layer(const DeepArgs& a, int l, cudaStream_t s) {
  const int M = a.n_out[l], K = a.n_in[l];
  dim3 grid(a.Np / 128, (M + 127) / 128);
  if (l == 0)
    sgemm_nn_kernel<false><<<grid, 256, 0, s>>>(M, a.Np, K, a.w[0], K, a.XT, a.Np, a.Z[0], a.Np, 0,
                                                0.0f);
  else
    sgemm_nn_kernel<true><<<grid, 256, 0, s>>>(M, a.Np, K, a.w[l], K, a.Z[l - 1], a.Np, a.Z[l],
                                               a.Np, a.act[l - 1], a.g[l - 1]);
  return cudaGetLastError();
}

cudaError_t launch_sum_loss(const float* ell, int N, DevState* st, cudaStream_t s) {
  sum_loss_kernel<<<1, 1024, 0, s>>>(ell, N, st);
  return cudaGetLastError();
}

// Output-field kernel variants, matching the trial-loop variants.
using OutFn = void (*)(Mlp2Args, const int*);

static OutFn pick_outputs(const Mlp2Args& a) {
  if (a.act1 == MCA_ACT_TANH && a.act2 == MCA_ACT_SIGMOID && a.loss == MCA_LOSS_MSE_ONEHOT)
    return mlp2_outputs_kernel<MCA_ACT_TANH, MCA_ACT_SIGMOID, MCA_LOSS_MSE_ONEHOT>;
  if (a.act1 == MCA_ACT_TANH && a.act2 == MCA_ACT_IDENTITY && a.loss == MCA_LOSS_SOFTMAX_CE)
    return mlp2_outputs_kernel<MCA_ACT_TANH, MCA_ACT_IDENTITY, MCA_LOSS_SOFTMAX_CE>;
  if (a.act1 == MCA_ACT_GAUSSIAN && a.act2 == MCA_ACT_SIGMOID && a.loss == MCA_LOSS_MSE_ONEHOT)
    return mlp2_outputs_kernel<MCA_ACT_GAUSSIAN, MCA_ACT_SIGMOID, MCA_LOSS_MSE_ONEHOT>;
  return mlp2_outputs_kernel<-1, -1, -1>;
}

cudaError_t launch_mlp2_outputs(const Mlp2Args& a, const int* y, cudaStream_t s) {
  pick_outputs(a)<<<(a.N + 127) / 128, 128, 0, s>>>(a, y);
  return cudaGetLastError();
}

}  // namespace mca
