// Device building blocks of the MCA trial loop: the Philox proposal stream, transfer functions,
// per-sample losses, deterministic block reductions and a bounded grid barrier.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/mca.h"

namespace mca {

// ------------------------------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11, Section 3.2): ten rounds of two 32x32->64
// multiplies and xors over a 128-bit counter, the 64-bit key bumped by the Weyl constants between
// rounds. Counter = (tau_lo, tau_hi, 0, 0), key = (seed_lo, seed_hi).
// The proposal-stream helpers below are also compiled for the host, so that a CPU test can check
// their arithmetic against the oracle.
// ------------------------------------------------------------------------------------------------
__host__ __device__ __forceinline__ uint32_t mulhi32(uint32_t a, uint32_t b) {
#ifdef __CUDA_ARCH__
  return __umulhi(a, b);
#else
  return (uint32_t)(((uint64_t)a * b) >> 32);
#endif
}

__host__ __device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
#ifdef __CUDA_ARCH__
#pragma unroll
#endif
  for (int r = 0; r < 10; ++r) {
    if (r) {
      k.x += 0x9E3779B9u;
      k.y += 0xBB67AE85u;
    }
    const uint32_t hi0 = mulhi32(0xD2511F53u, c.x), lo0 = 0xD2511F53u * c.x;
    const uint32_t hi1 = mulhi32(0xCD9E8D57u, c.z), lo1 = 0xCD9E8D57u * c.z;
    c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
  }
  return c;
}

__host__ __device__ __forceinline__ uint4 trial_words(uint64_t seed, uint64_t tau) {
  return philox4x32_10(make_uint4((uint32_t)tau, (uint32_t)(tau >> 32), 0u, 0u),
                       make_uint2((uint32_t)seed, (uint32_t)(seed >> 32)));
}

// Threshold of the Metropolis rule (Section 3.1, Eq. 7) on the loss-sum change of trial tau. Eq. 7
// keeps a mutation with probability min{1, exp(-beta dS / N)}; with the trial's own uniform number
// u = (r3 + 1/2) 2^-32, r3 the fourth Philox word of its counter, that is u < exp(-beta dS / N),
// i.e. dS <= -(N / beta) ln u. msc = N / beta > 0. Evaluated in fp64 (once per candidate and
// batch) and rounded to the fp32 of the candidate's dS.
__host__ __device__ __forceinline__ float metropolis_theta(uint64_t seed, uint64_t tau,
                                                             double msc) {
  const uint32_t r3 = trial_words(seed, tau).w;
  const double u = ((double)r3 + 0.5) * 0x1p-32;
  return (float)(-msc * log(u));
}

// Acceptance of a candidate with loss-sum change d (Eq. 6, or Eq. 7 when metro != 0).
__host__ __device__ __forceinline__ bool accept_change(float d, int strict, int metro,
                                                       uint64_t seed, uint64_t tau, double msc) {
  const float th = metro ? metropolis_theta(seed, tau, msc) : 0.0f;
  return strict ? (d < th) : (d <= th);
}

// Layer of stretch s under the current-layer schedule (Section 2.1: a layer chosen at random, many
// mutations inside it, then the next random layer): uniform over nl layers, from the first word of
// Philox4x32-10 at counter (s_lo, s_hi, 1, 0) -- apart from every trial's counter (tau, 0, 0).
__host__ __device__ __forceinline__ int stretch_layer(uint64_t seed, uint64_t s, int nl) {
  const uint4 w = philox4x32_10(make_uint4((uint32_t)s, (uint32_t)(s >> 32), 1u, 0u),
                                make_uint2((uint32_t)seed, (uint32_t)(seed >> 32)));
  return (int)(((unsigned long long)w.x * (unsigned int)nl) >> 32);
}

// Flat index of trial tau's weight in a two-layer net (P weights, the first P1 in W1) from the
// trial's first Philox word r0 (Eq. 1): uniform over the P weights, or, under the current-layer
// schedule (stretch = M > 0), uniform inside the stretch's layer.
__host__ __device__ __forceinline__ unsigned int mlp2_trial_index(unsigned long long P,
                                                                  unsigned long long P1,
                                                                  uint64_t seed, uint64_t tau,
                                                                  uint32_t r0, int stretch) {
  if (stretch <= 0) return (unsigned int)(((unsigned long long)r0 * P) >> 32);
  const int l = stretch_layer(seed, tau / (unsigned long long)stretch, 2);
  const unsigned long long lo = l ? P1 : 0ull, n = l ? P - P1 : P1;
  return (unsigned int)(lo + (((unsigned long long)r0 * n) >> 32));
}

// Channel mutations (Section 2.3): word m of trial tau's channel stream, the m % 4-th word of
// Philox4x32-10 at counter (tau_lo, tau_hi, 2, m / 4) -- apart from the trial's own counter
// (tau, 0, 0) and the schedule's (s, 0, 1, 0); a node uniform over n from a word; a redrawn weight
// a (2u - 1) in fp32 with He's uniform amplitude a = fp32(sqrt(6 / fan_in)), u = (v >> 8) 2^-24.
__host__ __device__ __forceinline__ uint32_t channel_word(uint64_t seed, uint64_t tau, int m) {
  const uint4 w = philox4x32_10(make_uint4((uint32_t)tau, (uint32_t)(tau >> 32), 2u,
                                           (uint32_t)(m >> 2)),
                                make_uint2((uint32_t)seed, (uint32_t)(seed >> 32)));
  const int r = m & 3;
  return r == 0 ? w.x : (r == 1 ? w.y : (r == 2 ? w.z : w.w));
}

__host__ __device__ __forceinline__ int channel_node(uint32_t v, unsigned long long n) {
  return (int)(((unsigned long long)v * n) >> 32);
}

__host__ __device__ __forceinline__ float channel_he_value(uint32_t v, int fan_in) {
  const float a = (float)sqrt(6.0 / (double)fan_in);
  const float u = (float)(v >> 8) * 0x1p-24f;
  const float r = 2.0f * u;                        // exact
  return a * (r - 1.0f);
}

// u = (r >> 8) * 2^-24: exact, in [0, 1)
__device__ __forceinline__ float unit24(uint32_t r) { return __uint2float_rn(r >> 8) * 0x1p-24f; }

// ------------------------------------------------------------------------------------------------
// The new value of one weight (Eq. 1). wk: storage kind; weff / code / wfix: the layer's arrays;
// off: the weight's offset in its layer; r1: the trial's second Philox word.
//   FP32:    replace by lo + (hi - lo) u, or perturb by delta (2u - 1); u = (r1 >> 8) 2^-24; the
//            domain |w'| < bound (bound > 0) rejects without evaluation
//   TERNARY: new code floor(r1 * 3 / 2^32) - 1, effective weight scale * code
//   MASKED:  toggle the mask bit of the fixed weight
// explicit_value: take ex_new as the new effective value instead (evaluation of given candidates).
// ------------------------------------------------------------------------------------------------
struct Mutation {
  float oldw, neww;
  int new_code;
  int valid;
};

__device__ __forceinline__ Mutation draw_mutation(int wk, const float* weff,
                                                  const signed char* code, const float* wfix,
                                                  float sc, unsigned long long off, int op, float lo,
                                                  float hi, float delta, float bound, uint32_t r1,
                                                  bool explicit_value, float ex_new) {
  Mutation m;
  m.valid = 1;
  m.new_code = 0;
  m.oldw = weff[off];
  if (explicit_value) {
    m.neww = ex_new;
  } else if (wk == MCA_W_TERNARY_I8) {
    const int oc = code[off];
    const int nc = (int)(((unsigned long long)r1 * 3ull) >> 32) - 1;
    m.oldw = __fmul_rn(sc, (float)oc);
    m.neww = __fmul_rn(sc, (float)nc);
    m.new_code = nc;
  } else if (wk == MCA_W_MASKED_FP32) {
    const int om = code[off];
    const int nm = 1 - om;
    const float w = wfix[off];
    m.oldw = om ? w : 0.0f;
    m.neww = nm ? w : 0.0f;
    m.new_code = nm;
  } else {
    const float u = __uint2float_rn(r1 >> 8) * 0x1p-24f;
    if (op == MCA_OP_PERTURB) {
      const float rr = __fsub_rn(__fmul_rn(2.0f, u), 1.0f);
      m.neww = __fadd_rn(m.oldw, __fmul_rn(delta, rr));
    } else {
      m.neww = __fadd_rn(lo, __fmul_rn(__fsub_rn(hi, lo), u));
    }
    if (bound > 0.0f && !(fabsf(m.neww) < bound)) m.valid = 0;
  }
  return m;
}

// Batch width from the decayed acceptance counts (the same arithmetic wherever it is evaluated, so
// every CTA of a launch, and the host, agree).
__host__ __device__ __forceinline__ int batch_width(float acc, float trials, float c, int K) {
  const float p = (acc + 0.5f) / (trials + 1.0f);
  const float w = ceilf(c / p);
  return w >= (float)K ? K : (w < 1.0f ? 1 : (int)w);
}

// Round to tf32 (10 explicit mantissa bits, nearest, ties away), kept in an fp32 register.
__device__ __forceinline__ float tf32_rna(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return __uint_as_float(r);
}

// The same rule with one approximate division (device only; deterministic, so every CTA agrees).
__device__ __forceinline__ int batch_width_fast(float acc, float trials, float c, int K) {
  const float w = ceilf(__fdividef(c * (trials + 1.0f), acc + 0.5f));
  return w >= (float)K ? K : (w < 1.0f ? 1 : (int)w);
}

// ------------------------------------------------------------------------------------------------
// Transfer functions (Section 2) and losses (Eq. 2 with R = 0). ACT < 0 selects at run time.
//
// exp and log use the hardware base-2 units (__expf, __logf: a few ulp). tanh is its exponential
// form tanh|x| = (1 - e^{-2|x|}) / (1 + e^{-2|x|}) with the sign restored: absolute error below
// ~2e-7, far inside the 1e-5 relative tolerance on the loss sum. Exactness where it matters does not
// depend on accuracy: an unchanged field gives f(z) - f(z) = 0 exactly because both sides go through
// the same function.
// ------------------------------------------------------------------------------------------------
__device__ __forceinline__ float tanh_exp(float x) {
  const float t = __expf(-2.0f * fabsf(x));
  return copysignf(__fdividef(1.0f - t, 1.0f + t), x);
}

__device__ __forceinline__ float act_rt(int act, float z, float g) {
  switch (act) {
    case MCA_ACT_TANH: return tanh_exp(z);
    case MCA_ACT_SIGMOID: return __fdividef(1.0f, 1.0f + __expf(-z));
    case MCA_ACT_RELU: return fmaxf(z, 0.0f);
    case MCA_ACT_GAUSSIAN: return __expf(-g * z * z);
    case MCA_ACT_GELU: return 0.5f * z * (1.0f + erff(z * 0.7071067811865476f));
    default: return z;
  }
}

template <int ACT>
__device__ __forceinline__ float act(float z, float g, int act_runtime) {
  if constexpr (ACT < 0) {
    return act_rt(act_runtime, z, g);
  } else {
    return act_rt(ACT, z, g);
  }
}

// Per-sample loss of the output fields z[0..C) with label y.
template <int ACT2, int LOSS, int MAXC>
__device__ __forceinline__ float sample_loss(const float (&z)[MAXC], int C, int y, float g2,
                                             int act2_rt, int loss_rt) {
  const int loss = LOSS < 0 ? loss_rt : LOSS;
  if (loss == MCA_LOSS_MSE_ONEHOT) {
    float s = 0.0f;
#pragma unroll
    for (int k = 0; k < MAXC; ++k) {
      if (k < C) {
        const float d = act<ACT2>(z[k], g2, act2_rt) - (k == y ? 1.0f : 0.0f);
        s = fmaf(d, d, s);
      }
    }
    return s;
  }
  float a[MAXC];
  float m = -INFINITY;
#pragma unroll
  for (int k = 0; k < MAXC; ++k) {
    if (k < C) {
      a[k] = act<ACT2>(z[k], g2, act2_rt);
      m = fmaxf(m, a[k]);
    }
  }
  float s = 0.0f, ay = 0.0f;
#pragma unroll
  for (int k = 0; k < MAXC; ++k) {
    if (k < C) {
      s += __expf(a[k] - m);
      if (k == y) ay = a[k];
    }
  }
  return (__logf(s) + m) - ay;
}

// ------------------------------------------------------------------------------------------------
// Deterministic reductions (fixed shuffle tree, fixed warp order)
// ------------------------------------------------------------------------------------------------
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Sum over the block; the result is valid in every thread. red: >= 32 floats of shared memory.
__device__ __forceinline__ float block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float t = lane < nw ? red[lane] : 0.0f;
  t = warp_sum(t);
  return t;
}

__device__ __forceinline__ double block_sum_d(double v, double* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_sum_d(v);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  double t = lane < nw ? red[lane] : 0.0;
  t = warp_sum_d(t);
  return t;
}

// ------------------------------------------------------------------------------------------------
// Grid barrier for a co-resident (cooperative) grid. Every wait is bounded: after kBarrierTimeoutNs
// the waiting CTA records MCA_ERR_TIMEOUT in *err and returns false, and so does every CTA that
// sees a non-zero *err while waiting; callers then leave the kernel.
// ------------------------------------------------------------------------------------------------
struct GridBarrier {
  unsigned int count;
  unsigned int gen;
};

constexpr unsigned long long kBarrierTimeoutNs = 2000000000ull;   // 2 s

__device__ __forceinline__ unsigned long long globaltimer_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ unsigned int ld_acquire_gpu(const unsigned int* p) {
  unsigned int v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ unsigned long long ld_acquire_gpu_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_gpu(unsigned int* p, unsigned int v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// CTA-scope acquire / release on shared memory (flags between the warps of one CTA).
__device__ __forceinline__ unsigned long long ld_acquire_cta_shared_u64(
    const unsigned long long* p) {
  unsigned long long v;
  const unsigned int a = (unsigned int)__cvta_generic_to_shared(p);
  asm volatile("ld.acquire.cta.shared.u64 %0, [%1];" : "=l"(v) : "r"(a) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_cta_shared_u64(unsigned long long* p,
                                                          unsigned long long v) {
  const unsigned int a = (unsigned int)__cvta_generic_to_shared(p);
  asm volatile("st.release.cta.shared.u64 [%0], %1;" ::"r"(a), "l"(v) : "memory");
}

__device__ __forceinline__ int ld_acquire_cta_shared_s32(const int* p) {
  int v;
  const unsigned int a = (unsigned int)__cvta_generic_to_shared(p);
  asm volatile("ld.acquire.cta.shared.s32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_cta_shared_s32(int* p, int v) {
  const unsigned int a = (unsigned int)__cvta_generic_to_shared(p);
  asm volatile("st.release.cta.shared.s32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}

__device__ __forceinline__ int ld_volatile_int(const int* p) {
  return *reinterpret_cast<const volatile int*>(p);
}

// gen_local: this CTA's copy of the barrier generation (same value in every CTA between barriers).
__device__ __forceinline__ bool grid_sync(GridBarrier* bar, unsigned int nblocks,
                                          unsigned int& gen_local, int* err, int* s_flag) {
  __syncthreads();
  if (threadIdx.x == 0) {
    int ok = 1;
    const unsigned int g = gen_local;
    __threadfence();
    const unsigned int prev = atomicAdd(&bar->count, 1u);
    if (prev == nblocks - 1) {
      bar->count = 0u;
      __threadfence();
      st_release_gpu(&bar->gen, g + 1u);
    } else {
      const unsigned long long t0 = globaltimer_ns();
      unsigned int spins = 0;
      while (ld_acquire_gpu(&bar->gen) == g) {
        if (ld_volatile_int(err) != 0) {
          ok = 0;
          break;
        }
        if ((++spins & 63u) == 0u && globaltimer_ns() - t0 > kBarrierTimeoutNs) {
          atomicCAS(err, 0, (int)MCA_ERR_TIMEOUT);
          ok = 0;
          break;
        }
      }
    }
    __threadfence();
    gen_local = g + 1u;
    *s_flag = ok && ld_volatile_int(err) == 0;
  }
  __syncthreads();
  const bool ok = *s_flag != 0;
  return ok;
}

// ------------------------------------------------------------------------------------------------
// Sample records, field-major: field f of sample n at base[f * pitch + n]; fields [0, M) are the
// output fields, 14 the sample's loss, 15 its label (int bits). Field-major keeps the lanes of a warp,
// which read different samples, in different shared-memory banks.
// ------------------------------------------------------------------------------------------------
constexpr int kRecFields = 16;
constexpr int kRecLoss = 14;
constexpr int kRecLabel = 15;

template <int M>
__device__ __forceinline__ void load_srec(const float* base, int pitch, int n, float (&z)[M],
                                          float& ell, int& y) {
  static_assert(M <= kRecLoss, "at most 14 output fields per sample record");
#pragma unroll
  for (int k = 0; k < M; ++k) z[k] = base[k * pitch + n];
  ell = base[kRecLoss * pitch + n];
  y = __float_as_int(base[kRecLabel * pitch + n]);
}

template <int M>
__device__ __forceinline__ void store_srec(float* base, int pitch, int n, const float (&z)[M],
                                           float ell, int y) {
  static_assert(M <= kRecLoss, "at most 14 output fields per sample record");
#pragma unroll
  for (int k = 0; k < M; ++k) base[k * pitch + n] = z[k];
  base[kRecLoss * pitch + n] = ell;
  base[kRecLabel * pitch + n] = __int_as_float(y);
}

// ------------------------------------------------------------------------------------------------
// Compensated fp32 summation (Knuth's TwoSum): hi + lo carries the sum with the rounding error of
// every addition kept in lo. Fixed order in, fixed result out; no fp64 (which is slow on this GPU).
// ------------------------------------------------------------------------------------------------
__device__ __forceinline__ void two_sum_add(float& hi, float& lo, float x) {
  const float s = hi + x;
  const float bb = s - hi;
  const float err = (hi - (s - bb)) + (x - bb);
  hi = s;
  lo += err;
}

// Compensated sums of the rows of x (rows of n floats, n apart): out[k] for k < rows with
// take[k] != 0 (else 0), each in index order with one two_sum_add per term, the arithmetic of
// ordered_sum. Every thread of the CTA calls it: warp w takes rows w, w + nwarps, ..., loads 256
// terms of a row at a time (coalesced) into its 256 floats of buf, and its lane 0 adds them.
// Ends with a CTA barrier.
__device__ __forceinline__ void ordered_row_sums(const float* x, int n, int rows, const int* take,
                                                 float* out, float* buf) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  float* b = buf + warp * 256;
  for (int k = warp; k < rows; k += nw) {
    float hi = 0.0f, lo = 0.0f;
    if (take[k]) {
      for (int q0 = 0; q0 < n; q0 += 256) {
        const int m = min(256, n - q0);
#pragma unroll 8
        for (int i = lane; i < m; i += 32) b[i] = x[(size_t)k * n + q0 + i];
        __syncwarp();
        if (lane == 0)
          for (int i = 0; i < m; ++i) two_sum_add(hi, lo, b[i]);
        __syncwarp();
      }
    }
    if (lane == 0) out[k] = take[k] ? hi + lo : 0.0f;
  }
  __syncthreads();
}

// Compensated sum of x[0 .. n) in index order: the same additions, in the same order, as one
// two_sum_add per term, with the loads of 32 terms in flight at a time.
__device__ __forceinline__ float ordered_sum(const float* x, int n) {
  float hi = 0.0f, lo = 0.0f;
  for (int q0 = 0; q0 < n; q0 += 32) {
    float v[32];
#pragma unroll
    for (int u = 0; u < 32; ++u) v[u] = q0 + u < n ? x[q0 + u] : 0.0f;
#pragma unroll
    for (int u = 0; u < 32; ++u)
      if (q0 + u < n) two_sum_add(hi, lo, v[u]);
  }
  return hi + lo;
}

// Lane 0 receives the compensated sum of the warp's (hi, lo) pairs (fixed xor tree).
__device__ __forceinline__ float warp_sum_comp(float hi, float lo) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float h2 = __shfl_xor_sync(0xffffffffu, hi, o);
    const float l2 = __shfl_xor_sync(0xffffffffu, lo, o);
    two_sum_add(hi, lo, h2);
    lo += l2;
  }
  return hi + lo;
}

}  // namespace mca
