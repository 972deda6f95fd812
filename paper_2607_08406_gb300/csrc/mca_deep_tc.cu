// Deep MLP path on the 5th-generation tensor cores: the dense part of a candidate's chain,
//   Z'_m = Z_m + W_m (f(Z'_{m-1}) - f(Z_{m-1})),   m = l+2 .. L-2   (Section 2.4),
// as error-compensated 3xTF32 tcgen05 MMAs with the accumulator in tensor memory.
//
// One CTA per (candidate, tile of kTcTS = 128 samples): 16 worker warps and one control warp. Per
// dense layer the CTA computes the transposed change D^T[samples x 256] = A[samples x 256] W_m^T,
// where A holds the previous layer's activation changes split as A = A_hi + A_lo (each rounded to
// tf32) and W_m = W_hi + W_lo (kept split in global memory, updated with every commit):
//   D = A_lo W_hi^T + A_hi W_lo^T + A_hi W_hi^T      (the A_lo W_lo^T term, ~2^-22 relative, dropped)
//
// The layers are pipelined chunk by chunk. The workers produce A in K chunks of 16 features (hi and
// lo, 16 KB) into a ring of four shared-memory slots; the control thread issues each chunk's six
// MMAs as soon as the chunk and its weight stage are there, so layer m+1's MMAs run while the
// workers are still forming layer m's later chunks. Two accumulators in tensor memory (columns
// [0, 256) and [256, 512)) alternate by layer: the workers read layer m's finished D while the
// MMAs of layer m+1 fill the other one. W streams through four 32 KB stages of 16-wide K chunks
// (hi + lo), each one bulk copy, reaching across layer boundaries. All operands are K-major without
// swizzle: 8-row x 16-byte core matrices.
//
// Worker warp w reads tensor-memory lanes 32 (w mod 4) .. + 31 (its samples) and, in every chunk,
// the four features 4 (w / 4) .. + 3: the cached field + D gives the new field, the next activation
// change f(z') - f(z) (exactly 0 where a field did not change) goes into the ring, and after the
// last dense layer the changes accumulate into the output layer instead. Every per-(candidate,
// tile) loss change depends only on that pair: the trajectory does not depend on the batch width.
// COMMIT writes the fields exactly as the evaluation computed them. Every wait is bounded (2 s); on a
// time-out the CTA records MCA_ERR_TIMEOUT, lets its issued copies and MMAs complete (bounded) and
// frees its tensor memory.
#include <cstdio>

#include "mca_deep.cuh"
#include "mca_device.cuh"
#include "mca_internal.h"
#include "mca_tc.cuh"

namespace mca {
namespace {

constexpr int kWorkWarps = 16;
constexpr int kTcThreads = (kWorkWarps + 1) * 32;   // + one control warp
constexpr int kCtl = kWorkWarps * 32;                // the control thread
constexpr int kParts = 4;                            // feature parts per lane quarter
constexpr int kTcW = 256;                            // width of the dense layers
constexpr int kTcKC = 16;                            // K chunk
constexpr int kTcChunks = kTcW / kTcKC;
constexpr int kAHalf = kTcTS * kTcKC * 4;            // 8 KB: hi or lo of one A chunk
constexpr int kASlot = 2 * kAHalf;
constexpr int kASlots = 4;
constexpr int kWHalfBytes = kTcW * kTcKC * 4;        // 16 KB: hi or lo of one W chunk
constexpr int kWStageBytes = 2 * kWHalfBytes;        // 32 KB
constexpr int kStages = 4;
constexpr int kTcSmem = kASlots * kASlot + kStages * kWStageBytes;
// core-matrix strides (bytes): A chunk: K groups 2 KB apart, sample groups 128 B apart;
// W stage: K groups 4 KB apart, row groups 128 B apart. The split weights of a layer are kept in
// global memory as kTcChunks consecutive 32 KB stage images (hi then lo), so that one bulk copy
// fills a stage.
constexpr uint32_t kALBO = (kTcTS / 8) * 128, kASBO = 128;
constexpr uint32_t kWLBO = (kTcW / 8) * 128, kWSBO = 128;
// kind::tf32, D fp32, A and B tf32 K-major, M = 128, N = 256
constexpr uint32_t kIdesc = tc_idesc_tf32(kTcTS, kTcW);

static_assert(kTcSmem + 2048 <= 227 * 1024, "shared memory of the chain kernel");
static_assert((kParts - 1) * kMaxC * kTcTS * 4 <= kStages * kWStageBytes, "output scratch");

// One thread: stage st <- the 32 KB image of one chunk, completion counted on mbarrier full.
__device__ __forceinline__ void load_stage(uint32_t dst, const void* src, uint64_t* full) {
  bulk_load(dst, src, (uint32_t)kWStageBytes, full);
}

__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

// Field rows of one layer for this tile into L2: worker thread t, row t / 2, two 128-byte lines.
__device__ __forceinline__ void prefetch_tile(const float* Zm, int Np, int n0, int t) {
  const float* r = Zm + (size_t)(t >> 1) * Np + n0 + 64 * (t & 1);
  prefetch_l2(r);
  prefetch_l2(r + 32);
}

// Four accumulator columns of this thread's lane into r, left in flight: the values may be read only
// after tmem_wait4(r).
__device__ __forceinline__ void tmem_issue4(uint32_t taddr, uint32_t (&r)[4]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(taddr) : "memory");
}

// Wait for this thread's tensor-memory loads; r is tied to the wait so that no read of it moves
// above it.
__device__ __forceinline__ void tmem_wait4(uint32_t (&r)[4]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]) :: "memory");
}

// Every lane waits for the phase; true in every lane iff no lane timed out.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity) ? 1 : 0) != 0;
}

// Worker: put four activation changes of sample s (features 4 fp .. + 3 of the chunk) into ring
// slot ga % kASlots as hi and lo tf32 parts, once the MMAs of the chunk kASlots earlier are done
// with the slot; then the warp's arrival on the slot's full barrier.
__device__ __forceinline__ bool produce_chunk(unsigned char* aring, uint64_t* afull,
                                              uint64_t* aempty, int ga, int fp, int s,
                                              const float (&d)[4]) {
  const int as = ga % kASlots;
  if (ga >= kASlots && !warp_wait(&aempty[as], (uint32_t)((ga / kASlots) - 1) & 1u)) return false;
  float hi[4], lo[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    hi[q] = tf32_rna(d[q]);
    lo[q] = tf32_rna(d[q] - hi[q]);
  }
  unsigned char* slot = aring + (size_t)as * kASlot + (size_t)fp * kALBO + (size_t)s * 16;
  *reinterpret_cast<float4*>(slot) = make_float4(hi[0], hi[1], hi[2], hi[3]);
  *reinterpret_cast<float4*>(slot + kAHalf) = make_float4(lo[0], lo[1], lo[2], lo[3]);
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  tc_fence_before();
  __syncwarp();
  if ((threadIdx.x & 31) == 0)
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&afull[as])) : "memory");
  return true;
}

// ACTH: transfer function of the hidden layers (-1: read per layer at run time).
template <bool COMMIT, int ACTH>
__global__ void __launch_bounds__(kTcThreads, 1) deep_chain_tc_kernel(DeepArgs a) {
  extern __shared__ __align__(1024) unsigned char tsm[];
  unsigned char* aring = tsm;                                 // A chunks
  unsigned char* wst = tsm + kASlots * kASlot;                // W stages
  __shared__ DeepCand s_cand;
  __shared__ float s_da[kTcTS];
  __shared__ float s_red[32];
  __shared__ __align__(8) uint64_t s_wfull[kStages], s_wempty[kStages];
  __shared__ __align__(8) uint64_t s_afull[kASlots], s_aempty[kASlots];
  __shared__ __align__(8) uint64_t s_dfull[2], s_drain;
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_fail;
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
  // this candidate's scratch slot, when it has one and a dense chain (layer <= L-3)
  float* const* sk = (!COMMIT && k < a.nscr && l <= L - 3) ? a.scr + (size_t)k * (L + 1) : nullptr;
  if (l + 1 < L - 1 && a.n_out[l + 1] == kTcW && tid < kCtl) prefetch_tile(a.Z[l + 1], Np, n0, tid);

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
        if (sk) sk[l][(size_t)j * Np + n] = zn;
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
    const int nd = dense ? (L - 2) - (l + 2) + 1 : 0;      // dense layers of the chain
    const int nchunks = nd * kTcChunks;
    const bool worker = warp < kWorkWarps;
    const int qd = warp & 3, fp = (warp >> 2) & 3;        // lane quarter, feature part
    const int s = qd * 32 + lane, n = n0 + s;
    const bool live = worker && n < N;
    const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
    uint32_t tmem = 0;
    if (dense) {
      if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;"
                     ::"r"(smem_u32(&s_tmem)));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
      }
      if (tid == kCtl) {
        for (int q = 0; q < kStages; ++q) {
          mbar_init(&s_wfull[q], 1);
          mbar_init(&s_wempty[q], 1);
        }
        for (int q = 0; q < kASlots; ++q) {
          mbar_init(&s_afull[q], kWorkWarps);
          mbar_init(&s_aempty[q], 1);
        }
        mbar_init(&s_dfull[0], 1);
        mbar_init(&s_dfull[1], 1);
        mbar_init(&s_drain, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        // the first weight chunks of the first dense layer load during the rank-1 step
        const unsigned char* w0 = reinterpret_cast<const unsigned char*>(a.whi[l + 2]);
        const uint32_t sw0 = smem_u32(wst);
        for (int q = 0; q < kStages - 1 && q < nchunks; ++q)
          load_stage(sw0 + (uint32_t)(q * kWStageBytes), w0 + (size_t)q * kWStageBytes, &s_wfull[q]);
      }
      tc_fence_before();
      __syncthreads();
      tc_fence_after();
      tmem = s_tmem;
    }
    float outp[kMaxC];
#pragma unroll
    for (int q = 0; q < kMaxC; ++q) outp[q] = 0.0f;
    const float* Wout = a.w[L - 1];
    const int Kout = a.n_in[L - 1];

    if (!worker) {
      // ---- control thread: every dense layer's MMAs, chunk by chunk as the workers produce A
      if (dense && lane == 0) {
        const uint32_t sw = smem_u32(wst), sa = smem_u32(aring);
        int issued_w = kStages - 1 < nchunks ? kStages - 1 : nchunks;   // weight chunks requested
        int landed_w = 0;                                               // ... and waited for
        bool ok = true;
        for (int gc = 0; gc < nchunks && ok; ++gc) {
          const int li = gc / kTcChunks, cc = gc % kTcChunks;
          const int as = gc % kASlots, st = gc % kStages;
          if (!mbar_wait(&s_wfull[st], (uint32_t)(gc / kStages) & 1u)) {
            ok = false;
            break;
          }
          landed_w = gc + 1;
          if (!mbar_wait(&s_afull[as], (uint32_t)(gc / kASlots) & 1u)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t dt = tmem + (uint32_t)(li & 1) * 256u;
#pragma unroll
          for (int ks = 0; ks < kTcKC / 8; ++ks) {
            const uint32_t ab = sa + (uint32_t)(as * kASlot) + (uint32_t)ks * 2u * kALBO;
            const uint32_t wb = sw + (uint32_t)(st * kWStageBytes) + (uint32_t)ks * 2u * kWLBO;
            const uint64_t dahi = umma_desc(ab, kALBO, kASBO);
            const uint64_t dalo = umma_desc(ab + kAHalf, kALBO, kASBO);
            const uint64_t dwhi = umma_desc(wb, kWLBO, kWSBO);
            const uint64_t dwlo = umma_desc(wb + kWHalfBytes, kWLBO, kWSBO);
            mma_ss(dt, dalo, dwhi, kIdesc, (cc > 0 || ks > 0) ? 1u : 0u);
            mma_ss(dt, dahi, dwlo, kIdesc, 1u);
            mma_ss(dt, dahi, dwhi, kIdesc, 1u);
          }
          umma_commit(&s_aempty[as]);
          umma_commit(&s_wempty[st]);
          if (cc == kTcChunks - 1) umma_commit(&s_dfull[li & 1]);
          // chunk gc + kStages - 1 goes to the stage chunk gc - 1 used, once its MMAs are done
          const int nc = gc + kStages - 1;
          if (nc < nchunks) {
            const int ns = nc % kStages;
            if (gc >= 1 && !mbar_wait(&s_wempty[ns], (uint32_t)((gc - 1) / kStages) & 1u)) {
              ok = false;
              break;
            }
            const int nl = l + 2 + nc / kTcChunks, nci = nc % kTcChunks;
            load_stage(sw + (uint32_t)(ns * kWStageBytes),
                       reinterpret_cast<const unsigned char*>(a.whi[nl]) +
                           (size_t)nci * kWStageBytes,
                       &s_wfull[ns]);
            issued_w = nc + 1;
          }
        }
        if (!ok) s_fail = 1;
        // drain: every MMA issued above complete, every requested weight chunk landed
        umma_commit(&s_drain);
        if (!mbar_wait(&s_drain, 0u)) s_fail = 1;
        for (int q = landed_w; q < issued_w; ++q)
          if (!mbar_wait(&s_wfull[q % kStages], (uint32_t)(q / kStages) & 1u)) s_fail = 1;
      }
    } else {
      // ---- workers
      bool ok = true;
      int ga = 0;                                         // A chunks produced
      float zo_n[4];                                      // cached fields one chunk ahead
      if (dense) prefetch_tile(a.Z[l + 2], Np, n0, tid);
      // layer l+1: rank-1 change through column j of W_{l+1}; its activation change is the first
      // A (dense) or feeds the output layer directly (l = L-3)
      {
        const int m1 = l + 1;
        const float* W1 = a.w[m1];
        const int K1 = a.n_in[m1];
        const float da = s_da[s];
        float* Zm = a.Z[m1];
        const bool moves = live && da != 0.0f;
        // loads one chunk ahead of their use (n < Np: always in the array)
        float wv[4], zo[4], wv_n[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          wv_n[q] = W1[(size_t)(fp * 4 + q) * K1 + j];
          zo_n[q] = Zm[(size_t)(fp * 4 + q) * Np + n];
        }
        for (int cc = 0; cc < kTcChunks; ++cc) {
          const int f0 = cc * kTcKC + fp * 4;
          float d[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            wv[q] = wv_n[q];
            zo[q] = zo_n[q];
          }
          if (cc + 1 < kTcChunks) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              wv_n[q] = W1[(size_t)(f0 + kTcKC + q) * K1 + j];
              zo_n[q] = Zm[(size_t)(f0 + kTcKC + q) * Np + n];
            }
          }
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float zn = fmaf(wv[q], da, zo[q]);
            const bool ch = moves && zn != zo[q];
            const float an = act<ACTH>(zn, a.g[m1], a.act[m1]);
            const float ao = act<ACTH>(zo[q], a.g[m1], a.act[m1]);
            d[q] = ch ? an - ao : 0.0f;
            if (COMMIT && ch) Zm[(size_t)(f0 + q) * Np + n] = zn;
            if (sk) sk[m1][(size_t)(f0 + q) * Np + n] = ch ? zn : zo[q];
          }
          if (dense) {
            if (!produce_chunk(aring, s_afull, s_aempty, ga, fp, s, d)) {
              ok = false;
              break;
            }
            ++ga;
          } else {
#pragma unroll
            for (int q = 0; q < 4; ++q)
#pragma unroll
              for (int o = 0; o < kMaxC; ++o)
                if (o < a.C) outp[o] = fmaf(Wout[(size_t)o * Kout + f0 + q], d[q], outp[o]);
          }
        }
      }
      // dense layers m = l+2 .. L-2: read D of layer m as its MMAs finish, form the next A
      if (dense) {
#pragma unroll
        for (int q = 0; q < 4; ++q) zo_n[q] = a.Z[l + 2][(size_t)(fp * 4 + q) * Np + n];
      }
      for (int li = 0; li < nd && ok; ++li) {
        const int m = l + 2 + li;
        const bool last = m == L - 2;
        if (!last) prefetch_tile(a.Z[m + 1], Np, n0, tid);
        if (!warp_wait(&s_dfull[li & 1], (uint32_t)(li >> 1) & 1u)) {
          ok = false;
          break;
        }
        tc_fence_after();
        float* Zm = a.Z[m];
        const uint32_t dt = tmem + lane_base + (uint32_t)(li & 1) * 256u;
        // accumulator columns one chunk ahead: chunk cc + 1's load is in flight while chunk cc is
        // processed
        uint32_t dr[4], dr_n[4];
        tmem_issue4(dt + (uint32_t)(fp * 4), dr_n);
        tmem_wait4(dr_n);
        for (int cc = 0; cc < kTcChunks; ++cc) {
          const int f0 = cc * kTcKC + fp * 4;
          float zo[4], dv[4], d[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            dr[q] = dr_n[q];
            dv[q] = __uint_as_float(dr[q]);
          }
          if (cc + 1 < kTcChunks) tmem_issue4(dt + (uint32_t)(f0 + kTcKC), dr_n);
#pragma unroll
          for (int q = 0; q < 4; ++q) zo[q] = zo_n[q];
          if (cc + 1 < kTcChunks) {            // the next chunk's cached fields, one chunk ahead
#pragma unroll
            for (int q = 0; q < 4; ++q) zo_n[q] = Zm[(size_t)(f0 + kTcKC + q) * Np + n];
          } else if (!last) {                  // the next layer's first chunk
#pragma unroll
            for (int q = 0; q < 4; ++q) zo_n[q] = a.Z[m + 1][(size_t)(fp * 4 + q) * Np + n];
          }
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float zn = zo[q] + dv[q];
            const bool ch = live && zn != zo[q];
            const float an = act<ACTH>(zn, a.g[m], a.act[m]);
            const float ao = act<ACTH>(zo[q], a.g[m], a.act[m]);
            d[q] = ch ? an - ao : 0.0f;
            if (COMMIT && ch) Zm[(size_t)(f0 + q) * Np + n] = zn;
            if (sk) sk[m][(size_t)(f0 + q) * Np + n] = ch ? zn : zo[q];
          }
          bool okc = true;
          if (!last) {
            okc = produce_chunk(aring, s_afull, s_aempty, ga, fp, s, d);
            ++ga;
          } else {
#pragma unroll
            for (int q = 0; q < 4; ++q)
#pragma unroll
              for (int o = 0; o < kMaxC; ++o)
                if (o < a.C) outp[o] = fmaf(Wout[(size_t)o * Kout + f0 + q], d[q], outp[o]);
          }
          tmem_wait4(dr_n);                    // chunk cc + 1's columns (none in flight at the end)
          if (!okc) {
            ok = false;
            break;
          }
        }
      }
      if (!ok) s_fail = 1;
    }

    // ---- output layer: the feature parts of each sample, in a fixed order
    tc_fence_before();
    __syncthreads();                                  // the control thread has drained
    float* xo = reinterpret_cast<float*>(wst);        // W stages are free now
    if (worker && fp >= 1) {
#pragma unroll
      for (int o = 0; o < kMaxC; ++o) xo[((fp - 1) * kMaxC + o) * kTcTS + s] = outp[o];
    }
    __syncthreads();
    if (worker && fp == 0) {
#pragma unroll
      for (int p = 1; p < kParts; ++p)
#pragma unroll
        for (int o = 0; o < kMaxC; ++o) outp[o] += xo[((p - 1) * kMaxC + o) * kTcTS + s];
    }
    const bool failed = s_fail != 0;                  // the same value in every thread here
    if (worker && fp == 0 && live && !failed) {
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
      if (sk) {                                       // the same output fields and loss as a commit
#pragma unroll
        for (int o = 0; o < kMaxC; ++o)
          if (o < a.C) sk[L - 1][(size_t)o * Np + n] = zz[o];
        const int Lo = L - 1;
        sk[L][n] = changed ? sample_loss<-1, -1, kMaxC>(zz, a.C, a.y[n], a.g[Lo], a.act[Lo], a.loss)
                           : a.ell[n];
      }
    } else if (sk && worker && fp == 0 && !failed) {  // padding samples keep their values
#pragma unroll
      for (int o = 0; o < kMaxC; ++o)
        if (o < a.C) sk[L - 1][(size_t)o * Np + n] = a.Z[L - 1][(size_t)o * Np + n];
      sk[L][n] = a.ell[n];
    }
    if (dense) {
      tc_fence_after();
      if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem));
      if (tid == 0 && failed) atomicCAS(&a.st->err, 0, (int)MCA_ERR_TIMEOUT);
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
