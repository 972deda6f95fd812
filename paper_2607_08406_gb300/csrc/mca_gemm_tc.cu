// Fields of a whole layer on the 5th-generation tensor cores: the forward pass over all samples
// (Section 2.1) that creation, mca_resync, mca_set_params and the channel trials run,
//   Z[M x Np] = W[M x K] act(B)[K x Np]       (feature-major fields, ld = Np; act = identity for X)
// as error-compensated 3xTF32 tcgen05 MMAs: with W = W_hi + W_lo and A = act(B)^T = A_hi + A_lo
// (each part rounded to tf32), D = A_lo W_hi^T + A_hi W_lo^T + A_hi W_hi^T (the lo.lo term, ~2^-22
// relative, dropped), accumulated in fp32 in tensor memory.
//
// The operands are first written as split images in core-matrix order (mca_tc_layout.h): A by
// blocks of 128 samples, W by blocks of 256 rows, both cut into K chunks of 16, each chunk the hi
// parts then the lo parts, so that one bulk copy moves one chunk. One CTA (4 warps) computes the
// transposed tile D^T[128 samples x 256 features]: thread 0 runs a two-stage ring of bulk copies
// (A chunk 16 KB + W chunk 32 KB per stage), thread 32 waits for each stage, issues its 6 MMAs
// (two K steps of 8) and releases the stage through tcgen05.commit; after the last chunk every warp
// reads its 32 tensor-memory lanes (samples) and writes the fields, 32 consecutive samples of one
// feature per store. 96 KB of shared memory and 256 tensor-memory columns per CTA, so two CTAs share
// an SM and one's epilogue overlaps the other's MMAs. Every wait is bounded (2 s); on a time-out the
// CTA records MCA_ERR_TIMEOUT, waits (bounded) for the copies it issued, frees its tensor memory
// and returns without writing.
#include "mca_device.cuh"
#include "mca_internal.h"
#include "mca_tc.cuh"
#include "mca_tc_layout.h"

namespace mca {

namespace {

constexpr int kGM = 128;                            // samples per tile (MMA M)
constexpr int kGN = 256;                            // features per tile (MMA N)
constexpr int kGK = 16;                             // K chunk of one stage
constexpr uint32_t kAHalf = kGM * kGK * 4;          // 8 KB: hi or lo of an A chunk
constexpr uint32_t kAChunk = 2 * kAHalf;
constexpr uint32_t kBHalf = kGN * kGK * 4;          // 16 KB: hi or lo of a W chunk
constexpr uint32_t kBChunk = 2 * kBHalf;
constexpr uint32_t kGStage = kAChunk + kBChunk;     // 48 KB
constexpr int kGStages = 2;
constexpr int kGThreads = 128;
constexpr int kGSmem = kGStages * kGStage;
// core-matrix strides (bytes): K-adjacent core matrices R * 16 apart, 8-row groups 128 apart
constexpr uint32_t kALBO = (kGM / 8) * 128, kASBO = 128;
constexpr uint32_t kBLBO = (kGN / 8) * 128, kBSBO = 128;
constexpr uint32_t kGIdesc = tc_idesc_tf32(kGM, kGN);

__device__ __forceinline__ void expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
               ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}

// Bulk copy whose bytes complete on `bar` (the arrival was counted by expect_tx).
__device__ __forceinline__ void bulk_copy(uint32_t dst, const void* src, uint32_t bytes,
                                          uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(dst), "l"(src), "r"(bytes), "r"(smem_u32(bar)) : "memory");
}

// A image: act(B)^T split, blocks of 128 samples. Thread: one sample n, four consecutive k.
__global__ void act_image_kernel(const float* __restrict__ B, int K, int Kp, int Np, int act,
                                 float g, float* __restrict__ img) {
  const int n = blockIdx.x * blockDim.x + threadIdx.x;
  const int k0 = blockIdx.y * 4;
  if (n >= Np) return;
  float hi[4], lo[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int k = k0 + q;
    float v = 0.0f;
    if (k < K) {
      v = B[(size_t)k * Np + n];
      if (act >= 0) v = act_rt(act, v, g);
    }
    hi[q] = tf32_rna(v);
    lo[q] = tf32_rna(v - hi[q]);
  }
  const size_t o = tc_image_index(n, k0, kGM, Kp);
  *reinterpret_cast<float4*>(img + o) = make_float4(hi[0], hi[1], hi[2], hi[3]);
  *reinterpret_cast<float4*>(img + o + tc_image_lo(kGM)) = make_float4(lo[0], lo[1], lo[2], lo[3]);
}

// W image: blocks of 256 rows. Thread: one row r, four consecutive k.
__global__ void w_image_kernel(const float* __restrict__ W, int M, int K, int Kp,
                               float* __restrict__ img) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  const int k0 = blockIdx.y * 4;
  if (r >= M) return;
  float hi[4], lo[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int k = k0 + q;
    const float v = k < K ? W[(size_t)r * K + k] : 0.0f;
    hi[q] = tf32_rna(v);
    lo[q] = tf32_rna(v - hi[q]);
  }
  const size_t o = tc_image_index(r, k0, kGN, Kp);
  *reinterpret_cast<float4*>(img + o) = make_float4(hi[0], hi[1], hi[2], hi[3]);
  *reinterpret_cast<float4*>(img + o + tc_image_lo(kGN)) = make_float4(lo[0], lo[1], lo[2], lo[3]);
}

__global__ void __launch_bounds__(kGThreads) gemm_tc_kernel(const float* __restrict__ aimg,
                                                            const float* __restrict__ bimg,
                                                            int nch, float* __restrict__ Z,
                                                            int ldz, int* err) {
  extern __shared__ __align__(1024) unsigned char gsm[];
  __shared__ __align__(8) uint64_t s_full[kGStages], s_empty[kGStages], s_done;
  __shared__ uint32_t s_tmem;
  __shared__ int s_fail;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int bs = blockIdx.x, bf = blockIdx.y;
  const unsigned char* ag =
      reinterpret_cast<const unsigned char*>(aimg) + (size_t)bs * nch * kAChunk;
  const unsigned char* bg =
      reinterpret_cast<const unsigned char*>(bimg) + (size_t)bf * nch * kBChunk;
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 256;"
                 ::"r"(smem_u32(&s_tmem)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  if (tid == 32) {
    for (int q = 0; q < kGStages; ++q) {
      mbar_init(&s_full[q], 1);
      mbar_init(&s_empty[q], 1);
    }
    mbar_init(&s_done, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    s_fail = 0;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  const uint32_t sbase = smem_u32(gsm);

  if (tid == 0) {
    // producer: chunk c into stage c % 2 once the MMAs of chunk c - 2 released it
    int issued = 0;
    for (int c = 0; c < nch; ++c) {
      const int st = c % kGStages;
      if (c >= kGStages && !mbar_wait(&s_empty[st], (uint32_t)((c / kGStages) - 1) & 1u)) {
        s_fail = 1;
        break;
      }
      expect_tx(&s_full[st], kGStage);
      bulk_copy(sbase + (uint32_t)st * kGStage, ag + (size_t)c * kAChunk, kAChunk, &s_full[st]);
      bulk_copy(sbase + (uint32_t)st * kGStage + kAChunk, bg + (size_t)c * kBChunk, kBChunk,
                &s_full[st]);
      issued = c + 1;
    }
    // copies still in flight land before the CTA can leave (the consumer waits for the rest)
    for (int c = (issued > kGStages ? issued - kGStages : 0); c < issued; ++c)
      if (!mbar_wait(&s_full[c % kGStages], (uint32_t)(c / kGStages) & 1u)) s_fail = 1;
  } else if (tid == 32) {
    // MMA issuer
    for (int c = 0; c < nch; ++c) {
      const int st = c % kGStages;
      if (!mbar_wait(&s_full[st], (uint32_t)(c / kGStages) & 1u)) {
        s_fail = 1;
        break;
      }
      tc_fence_after();
      const uint32_t sa = sbase + (uint32_t)st * kGStage, sb = sa + kAChunk;
#pragma unroll
      for (int ks = 0; ks < kGK / 8; ++ks) {
        const uint64_t ahi = umma_desc(sa + (uint32_t)ks * 2u * kALBO, kALBO, kASBO);
        const uint64_t alo = umma_desc(sa + kAHalf + (uint32_t)ks * 2u * kALBO, kALBO, kASBO);
        const uint64_t bhi = umma_desc(sb + (uint32_t)ks * 2u * kBLBO, kBLBO, kBSBO);
        const uint64_t blo = umma_desc(sb + kBHalf + (uint32_t)ks * 2u * kBLBO, kBLBO, kBSBO);
        mma_ss(tmem, alo, bhi, kGIdesc, (c > 0 || ks > 0) ? 1u : 0u);
        mma_ss(tmem, ahi, blo, kGIdesc, 1u);
        mma_ss(tmem, ahi, bhi, kGIdesc, 1u);
      }
      umma_commit(&s_empty[st]);
    }
    umma_commit(&s_done);                  // every MMA issued above has completed
  }
  __syncwarp();
  if (!mbar_wait(&s_done, 0u)) s_fail = 1;
  tc_fence_after();
  __syncthreads();
  if (!s_fail) {                           // the same value in every thread after the barrier
    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    const int n = bs * kGM + warp * 32 + lane;
    float* zc = Z + (size_t)bf * kGN * ldz + n;
    for (int c0 = 0; c0 < kGN; c0 += 16) {
      float v[16];
      tmem_ld16(tmem + lane_base + (uint32_t)c0, v);
#pragma unroll
      for (int q = 0; q < 16; ++q) zc[(size_t)(c0 + q) * ldz] = v[q];
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 256;" ::"r"(tmem));
  if (tid == 0 && s_fail) atomicCAS(err, 0, (int)MCA_ERR_TIMEOUT);
}

}  // namespace

bool gemm_tc_ok(int M, int K, int Np) { return M > 0 && M % kGN == 0 && K >= 1 && Np % kGM == 0; }

size_t gemm_tc_image_bytes(int M, int K, int Np) {
  const size_t nch = (size_t)(K + kGK - 1) / kGK;
  return nch * ((size_t)(Np / kGM) * kAChunk + (size_t)(M / kGN) * kBChunk);
}

cudaError_t launch_gemm_tc(const float* W, int M, int K, const float* B, int act, float g,
                           float* Z, int Np, float* img, int* err, cudaStream_t s) {
  if (!gemm_tc_ok(M, K, Np)) return cudaErrorInvalidValue;
  const int Kp = (K + kGK - 1) / kGK * kGK, nch = Kp / kGK;
  float* aimg = img;
  float* bimg = img + (size_t)nch * (size_t)(Np / kGM) * (kAChunk / 4);
  act_image_kernel<<<dim3((Np + 127) / 128, Kp / 4), 128, 0, s>>>(B, K, Kp, Np, act, g, aimg);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  w_image_kernel<<<dim3((M + 127) / 128, Kp / 4), 128, 0, s>>>(W, M, K, Kp, bimg);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(gemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kGSmem);
  if (e != cudaSuccess) return e;
  gemm_tc_kernel<<<dim3(Np / kGM, M / kGN), kGThreads, kGSmem, s>>>(aimg, bimg, nch, Z, Np, err);
  return cudaGetLastError();
}

}  // namespace mca
