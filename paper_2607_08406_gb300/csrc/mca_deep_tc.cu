// Deep MLP path on the 5th-generation tensor cores: the dense part of a candidate's chain,
//   Z'_m = Z_m + W_m (f(Z'_{m-1}) - f(Z_{m-1})),   m = l+2 .. L-2   (Section 2.4),
// as error-compensated 3xTF32 tcgen05 MMAs with the accumulator in tensor memory.
//
// One CTA per (candidate, tile of kTcTS = 128 samples), 512 threads. Per dense layer the CTA computes
// the transposed change D^T[samples x 256] = A[samples x 256] W_m^T, where A holds the previous
// layer's activation changes split as A = A_hi + A_lo (each rounded to tf32) and W_m = W_hi + W_lo
// (kept split in global memory, updated with every commit):
//   D = A_lo W_hi^T + A_hi W_lo^T + A_hi W_hi^T      (the A_lo W_lo^T term, ~2^-22 relative, dropped)
// Tensor memory (512 columns): D in columns [0, 256) (lane = sample, column = output feature),
// A_hi in columns [256, 512) (the A operand of two of the three MMAs). A_lo lives in shared memory
// (128 KB); W streams through three 32 KB stages of 16-wide K chunks (hi + lo), each filled by one
// bulk copy, in a ring run by one thread (full / empty mbarriers) that reaches across layer
// boundaries. All operands are K-major without swizzle: 8-row x 16-byte core matrices.
//
// The epilogue (all 16 warps; warp w reads tensor-memory lanes 32 (w mod 4) .. + 31 and a quarter of
// the features) adds D to the cached fields, forms the next activation change f(z') - f(z) (exactly 0
// where a field did not change), and writes its hi part to tensor memory and its lo part to shared
// memory for the next layer; after the last dense layer it accumulates the output layer instead.
// Every per-(candidate, tile) loss change depends only on that pair: the trajectory does not depend
// on the batch width. COMMIT writes the fields exactly as the evaluation computed them.
#include <cstdio>

#include "mca_deep.cuh"
#include "mca_device.cuh"
#include "mca_internal.h"
#include "mca_tc.cuh"

namespace mca {
namespace {

constexpr int kTcThreads = 512;
constexpr int kParts = kTcThreads / 128;     // feature parts per sample (warps sharing a lane quarter)
constexpr int kTcW = 256;                  // width of the dense layers
constexpr int kPartW = kTcW / kParts;
constexpr int kTcKC = 16;                  // K chunk of a W stage
constexpr int kTcChunks = kTcW / kTcKC;
constexpr int kAloBytes = kTcTS * kTcW * 4;          // 128 KB
constexpr int kWHalfBytes = kTcW * kTcKC * 4;        // 16 KB: one of hi / lo of one chunk
constexpr int kWStageBytes = 2 * kWHalfBytes;        // 32 KB
constexpr int kStages = 3;
constexpr int kTcSmem = kAloBytes + kStages * kWStageBytes;
// core-matrix strides (bytes): A_lo: K groups 2 KB apart, sample groups 128 B apart;
// W stage: K groups 4 KB apart, row groups 128 B apart. The split weights of a layer are kept in
// global memory as kTcChunks consecutive 32 KB stage images (hi then lo), so that one bulk copy
// fills a stage.
constexpr uint32_t kAloLBO = (kTcTS / 8) * 128, kAloSBO = 128;
constexpr uint32_t kWLBO = (kTcW / 8) * 128, kWSBO = 128;
// kind::tf32, D fp32, A and B tf32 K-major, M = 128, N = 256
constexpr uint32_t kIdesc = tc_idesc_tf32(kTcTS, kTcW);

static_assert(kTcSmem + 2048 <= 227 * 1024, "shared memory of the chain kernel");

// One thread: stage st <- the 32 KB image of one chunk, completion counted on mbarrier full.
__device__ __forceinline__ void load_stage(uint32_t dst, const void* src, uint64_t* full) {
  bulk_load(dst, src, (uint32_t)kWStageBytes, full);
}

// A_lo element (sample s, feature k) in shared memory: 16 consecutive features of one sample as
// four 16-byte stores.
__device__ __forceinline__ void store_alo16(unsigned char* alo, int s, int f0, const float (&v)[16]) {
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    const int k = f0 + 4 * g;
    *reinterpret_cast<float4*>(alo + (size_t)(k >> 2) * kAloLBO + (size_t)s * 16) =
        make_float4(v[4 * g], v[4 * g + 1], v[4 * g + 2], v[4 * g + 3]);
  }
}

__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

// Field rows of one layer for this tile into L2 (thread t: row t, four 128-byte lines).
__device__ __forceinline__ void prefetch_tile(const float* Zm, int Np, int n0, int tid) {
#pragma unroll
  for (int p = 0; p < kTcTS / 32; ++p) prefetch_l2(Zm + (size_t)tid * Np + n0 + 32 * p);
}

// ACTH: transfer function of the hidden layers (-1: read per layer at run time).
template <bool COMMIT, int ACTH>
__global__ void __launch_bounds__(kTcThreads, 1) deep_chain_tc_kernel(DeepArgs a) {
  extern __shared__ __align__(1024) unsigned char tsm[];
  unsigned char* alo = tsm;                                   // A_lo
  unsigned char* wst = tsm + kAloBytes;                       // W stages
  __shared__ DeepCand s_cand;
  __shared__ float s_da[kTcTS];
  __shared__ float s_red[32];
  __shared__ __align__(8) uint64_t s_full[kStages], s_empty[kStages];
  __shared__ uint32_t s_tmem;
  __shared__ int s_fail;
  __shared__ int s_k;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int k = 0, tile = COMMIT ? blockIdx.x : 0;
  if (COMMIT && a.ctl->kstar < 0) return;
  if (!COMMIT) {
    // Longest chains first: CTAs start in linear block order, so the linear index is mapped to
    // (candidate rank, tile) with the candidates ranked by the depth of their dense chain (the
    // mutated layer, from the proposal alone), ties by index. Every CTA computes the same ranking.
    const int Kb = gridDim.x;
    const int lid = blockIdx.x + blockIdx.y * gridDim.x;
    const int rank = lid / a.ntiles;
    tile = lid - rank * a.ntiles;
    if (tid < Kb) {
      const int my = deep_candidate_layer(a, tid);
      int rk = 0;
      for (int q = 0; q < Kb; ++q) {
        const int lq = deep_candidate_layer(a, q);
        rk += (lq < my || (lq == my && q < tid)) ? 1 : 0;     // shallower layer = longer chain
      }
      if (rk == rank) s_k = tid;
    }
    __syncthreads();
    k = s_k;
  }
  const int n0 = tile * kTcTS;
  if (tid == 0) {
    s_cand = COMMIT ? a.ctl->acc : deep_candidate(a, k);
    s_fail = 0;
  }
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
  if (l + 1 < L - 1 && a.n_out[l + 1] == kTcW && tid < kTcW)
    prefetch_tile(a.Z[l + 1], Np, n0, tid);

  // ---- row j of layer l (thread s = sample)
  if (tid < kTcTS) {
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

  if (l == L - 2) {
    // ---- layer l+1 is the output layer: rank-1 change of the output fields
    if (tid < kTcTS) {
      const int n = n0 + tid;
      const float da = s_da[tid];
      const float* W1 = a.w[L - 1];
      if (n < N && da != 0.0f) {
        float zz[kMaxC];
        bool changed = false;
#pragma unroll
        for (int q = 0; q < kMaxC; ++q) {
          if (q < a.C) {
            const float zo = a.Z[L - 1][(size_t)q * Np + n];
            zz[q] = fmaf(W1[(size_t)q * a.n_in[L - 1] + j], da, zo);
            changed |= zz[q] != zo;
          } else {
            zz[q] = 0.0f;
          }
        }
        dl = out_delta<COMMIT>(a, n, zz, changed);
      }
    }
  } else if (l < L - 2) {
    const bool dense = l + 2 <= L - 2;
    const int qd = warp & 3, hf = warp >> 2;         // lane quarter, feature part
    const int s = qd * 32 + lane, n = n0 + s;
    const bool live = n < N;
    const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
    uint32_t tmem = 0;
    if (dense) {
      if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;"
                     ::"r"(smem_u32(&s_tmem)));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
      }
      if (tid == 0) {
        for (int q = 0; q < kStages; ++q) {
          asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&s_full[q])));
          asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&s_empty[q])));
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        // the first two chunks of the first dense layer load during the rank-1 step
        const unsigned char* w0 = reinterpret_cast<const unsigned char*>(a.whi[l + 2]);
        const uint32_t sw0 = smem_u32(wst);
        for (int q = 0; q < kStages - 1 && q < (L - 2 - (l + 2) + 1) * kTcChunks; ++q)
          load_stage(sw0 + (uint32_t)(q * kWStageBytes), w0 + (size_t)q * kWStageBytes, &s_full[q]);
      }
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncthreads();
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      tmem = s_tmem;
    }
    // output-layer accumulation of this thread's feature half (after the last change matrix)
    float outp[kMaxC];
#pragma unroll
    for (int q = 0; q < kMaxC; ++q) outp[q] = 0.0f;
    const float* Wout = a.w[L - 1];
    const int Kout = a.n_in[L - 1];

    // ---- layer l+1: rank-1 change through column j of W_{l+1}; its activation change is the
    // first A (dense) or feeds the output layer directly (l = L-3)
    {
      const int m1 = l + 1;
      const float* W1 = a.w[m1];
      const int K1 = a.n_in[m1];
      const float da = s_da[s];
      float* Zm = a.Z[m1];
      const bool moves = live && da != 0.0f;
      for (int f0 = hf * kPartW; f0 < (hf + 1) * kPartW; f0 += 16) {
        float hi[16], lo[16], zo[16], wv[16];
#pragma unroll
        for (int q = 0; q < 16; ++q) {          // loads first (n < Np: always in the array)
          wv[q] = W1[(size_t)(f0 + q) * K1 + j];
          zo[q] = Zm[(size_t)(f0 + q) * Np + n];
        }
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          const int f = f0 + q;
          const float zn = fmaf(wv[q], da, zo[q]);
          const bool ch = moves && zn != zo[q];
          const float an = act<ACTH>(zn, a.g[m1], a.act[m1]);
          const float ao = act<ACTH>(zo[q], a.g[m1], a.act[m1]);
          const float d = ch ? an - ao : 0.0f;
          if (COMMIT && ch) Zm[(size_t)f * Np + n] = zn;
          if (dense) {
            hi[q] = tf32_rna(d);
            lo[q] = tf32_rna(d - hi[q]);
          } else {
#pragma unroll
            for (int o = 0; o < kMaxC; ++o)
              if (o < a.C) outp[o] = fmaf(Wout[(size_t)o * Kout + f], d, outp[o]);
          }
        }
        if (dense) {
          tmem_st16(tmem + lane_base + 256u + (uint32_t)f0, hi);
          store_alo16(alo, s, f0, lo);
        }
      }
    }

    // ---- dense layers m = l+2 .. L-2 on the tensor cores
    if (dense) {
      const uint32_t sw = smem_u32(wst), salo = smem_u32(alo);
      const int nchunks = (L - 2 - (l + 2) + 1) * kTcChunks;   // chunks of all dense layers
      for (int m = l + 2; m <= L - 2; ++m) {
        const int li = m - (l + 2);
        if (tid < kTcW) prefetch_tile(a.Z[m], Np, n0, tid);
        // the previous step's A (tensor memory, shared memory) complete before the MMAs read it
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncthreads();
        if (tid == 0) {
          // one thread: wait for a chunk, issue its MMAs, release its stage, refill two ahead
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          for (int cidx = 0; cidx < kTcChunks; ++cidx) {
            const int gc = li * kTcChunks + cidx, st = gc % kStages;
            if (!mbar_wait(&s_full[st], (uint32_t)(gc / kStages) & 1u)) {
              s_fail = 1;
              break;
            }
#pragma unroll
            for (int ks = 0; ks < kTcKC / 8; ++ks) {
              const int g = cidx * (kTcKC / 8) + ks;       // K step of 8 over the layer
              const uint64_t dalo = umma_desc(salo + (uint32_t)g * 2u * kAloLBO, kAloLBO, kAloSBO);
              const uint32_t wb = sw + (uint32_t)(st * kWStageBytes) + (uint32_t)ks * 2u * kWLBO;
              const uint64_t dwhi = umma_desc(wb, kWLBO, kWSBO);
              const uint64_t dwlo = umma_desc(wb + kWHalfBytes, kWLBO, kWSBO);
              const uint32_t tahi = tmem + 256u + (uint32_t)(g * 8);
              mma_ss(tmem, dalo, dwhi, kIdesc, g > 0 ? 1u : 0u);
              mma_ts(tmem, tahi, dwlo, kIdesc, 1u);
              mma_ts(tmem, tahi, dwhi, kIdesc, 1u);
            }
            umma_commit(&s_empty[st]);
            // chunk gc + 2 goes to the stage chunk gc - 1 used, once its MMAs are done
            const int nc = gc + kStages - 1;
            if (nc < nchunks) {
              const int ns = nc % kStages;
              if (gc >= 1 && !mbar_wait(&s_empty[ns], (uint32_t)((gc - 1) / kStages) & 1u)) {
                s_fail = 1;
                break;
              }
              const int nl = l + 2 + nc / kTcChunks, nci = nc % kTcChunks;
              load_stage(sw + (uint32_t)(ns * kWStageBytes),
                         reinterpret_cast<const unsigned char*>(a.whi[nl]) +
                             (size_t)nci * kWStageBytes,
                         &s_full[ns]);
            }
          }
        }
        // every MMA of the layer done: the last chunk's commit (commits complete in order)
        {
          const int gl = li * kTcChunks + kTcChunks - 1;
          if (!mbar_wait(&s_empty[gl % kStages], (uint32_t)(gl / kStages) & 1u)) s_fail = 1;
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        __syncthreads();
        if (s_fail) break;                            // the same value in every thread here

        // epilogue: new fields, the next A (or the output layer after the last dense layer)
        const bool last = m == L - 2;
        float* Zm = a.Z[m];
        for (int f0 = hf * kPartW; f0 < (hf + 1) * kPartW; f0 += 16) {
          float zo[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) zo[q] = Zm[(size_t)(f0 + q) * Np + n];
          float dv[16];
          tmem_ld16(tmem + lane_base + (uint32_t)f0, dv);
          float hi[16], lo[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const int f = f0 + q;
            const float zn = zo[q] + dv[q];
            const bool ch = live && zn != zo[q];
            const float an = act<ACTH>(zn, a.g[m], a.act[m]);
            const float ao = act<ACTH>(zo[q], a.g[m], a.act[m]);
            const float d = ch ? an - ao : 0.0f;
            if (COMMIT && ch) Zm[(size_t)f * Np + n] = zn;
            if (!last) {
              hi[q] = tf32_rna(d);
              lo[q] = tf32_rna(d - hi[q]);
            } else {
#pragma unroll
              for (int o = 0; o < kMaxC; ++o)
                if (o < a.C) outp[o] = fmaf(Wout[(size_t)o * Kout + f], d, outp[o]);
            }
          }
          if (!last) {
            tmem_st16(tmem + lane_base + 256u + (uint32_t)f0, hi);
            store_alo16(alo, s, f0, lo);
          }
        }
      }
    }

    // ---- output layer: the feature parts of each sample, in a fixed order
    float* xo = reinterpret_cast<float*>(wst);        // W stages are free now
    __syncthreads();
    if (hf >= 1) {
#pragma unroll
      for (int o = 0; o < kMaxC; ++o) xo[((hf - 1) * kMaxC + o) * kTcTS + s] = outp[o];
    }
    __syncthreads();
    if (hf == 0) {
#pragma unroll
      for (int p = 1; p < kParts; ++p)
#pragma unroll
        for (int o = 0; o < kMaxC; ++o) outp[o] += xo[((p - 1) * kMaxC + o) * kTcTS + s];
    }
    if (hf == 0 && live) {
      float zz[kMaxC];
      bool changed = false;
#pragma unroll
      for (int o = 0; o < kMaxC; ++o) {
        if (o < a.C) {
          const float zo = a.Z[L - 1][(size_t)o * Np + n];
          zz[o] = zo + outp[o];
          changed |= zz[o] != zo;
        } else {
          zz[o] = 0.0f;
        }
      }
      dl = out_delta<COMMIT>(a, n, zz, changed);
    }
    if (dense) {
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncthreads();
      if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem));
      if (tid == 0 && s_fail) atomicCAS(&a.st->err, 0, (int)MCA_ERR_TIMEOUT);
    }
  }
  if (!COMMIT) {
    const float tot = block_sum(dl, s_red);
    if (tid == 0) *part = tot;
  }
}

// W_hi = tf32(W), W_lo = tf32(W - W_hi) for every dense layer, stored as the stage images the
// chain kernel copies (chunk c: hi then lo, core-matrix order).
__global__ void deep_split_kernel(DeepArgs a) {
  const int m = blockIdx.y + 1;
  if (m > a.L - 2 || a.whi[m] == nullptr) return;
  const int n = kTcW * kTcW;
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < n; e += gridDim.x * blockDim.x) {
    const int r = e / kTcW, k = e % kTcW;
    const float w = a.w[m][e];
    const float h = tf32_rna(w);
    const size_t o = deep_tc_image_index(r, k);
    a.whi[m][o] = h;
    a.whi[m][o + kWHalfBytes / 4] = tf32_rna(w - h);
  }
}

}  // namespace

cudaError_t launch_deep_split(const DeepArgs& a, cudaStream_t s) {
  if (a.L < 3) return cudaSuccess;
  deep_split_kernel<<<dim3(64, a.L - 2), 256, 0, s>>>(a);
  return cudaGetLastError();
}

// The hidden layers' common transfer function, if every layer 1 .. L-2 has the same one.
static int hidden_act(const DeepArgs& a) {
  for (int m = 1; m <= a.L - 2; ++m)
    if (a.act[m] != a.act[1]) return -1;
  return a.act[1] == MCA_ACT_TANH ? MCA_ACT_TANH : -1;
}

template <bool COMMIT>
static cudaError_t launch_tc(const DeepArgs& a, dim3 grid, cudaStream_t s) {
  const void* fn = hidden_act(a) == MCA_ACT_TANH
                       ? (const void*)deep_chain_tc_kernel<COMMIT, MCA_ACT_TANH>
                       : (const void*)deep_chain_tc_kernel<COMMIT, -1>;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kTcSmem);
  if (e != cudaSuccess) return e;
  DeepArgs args = a;
  void* params[] = {&args};
  return cudaLaunchKernel(fn, grid, dim3(kTcThreads), params, kTcSmem, s);
}

cudaError_t launch_deep_eval_tc(const DeepArgs& a, cudaStream_t s) {
  const int Kb = a.n_explicit > 0 ? a.n_explicit : a.Kb;
  return launch_tc<false>(a, dim3(Kb, a.ntiles), s);
}

cudaError_t launch_deep_commit_tc(const DeepArgs& a, cudaStream_t s) {
  return launch_tc<true>(a, dim3(a.ntiles), s);
}

}  // namespace mca
