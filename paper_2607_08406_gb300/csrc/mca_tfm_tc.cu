// Character-level Transformer on the 5th-generation tensor cores: the trial loop's recomputation of
// a sequence from the first sub-block a mutated parameter feeds (Section 2.4's cached forward,
// applied to the pre-LN GPT network of Section 2.5), with every dense projection as
// error-compensated 3xTF32 tcgen05 MMAs and the accumulators in tensor memory. Cached per sequence:
// the stream entering each block and, after each block's attention sub-block, its mid stream; a
// parameter of a block's feed-forward sub-block (LN2, W1, b1, W2, b2) restarts there.
//
// One CTA, 512 threads, recomputes two sequences for one candidate: M = 128 token rows, rows 0-63
// the even sequence and 64-127 the odd one. Thread (warp w, lane) owns token row
// r = 32 (w mod 4) + lane (the tensor-memory lanes its warp may access) and column part
// g = w / 4: columns 32g .. 32g + 31 of a 128-wide row, attention head g, and the 16-column
// slice 16g .. 16g + 15 of a 64-wide feed-forward chunk.
//
// Per block, with the residual stream X of both sequences in shared memory (fp32):
//   LN1 -> A (tf32 hi part in tensor memory, lo part in shared memory) -> Q, K, V = A Wq^T, A Wk^T,
//   A Wv^T (tensor-memory columns 0, 128, 256; A at 384) -> K and V to shared memory -> causal
//   attention of (row, head g) on the CUDA cores with a running softmax -> its output as the next
//   A -> A Wo^T -> X += . + bo -> LN2 -> A -> per pair of 64-wide hidden chunks: U = A W1_pair^T
//   (N = 128: a tcgen05 MMA takes about as long at N = 64 as at N = 128, so pairing halves W1's
//   MMAs), then per chunk c of the pair act(U_c + b1) as A2 (hi and lo parts both in tensor
//   memory), F += A2 W2_c^T -> X += F + b2.
// After the last block: LNf -> A -> logits = A Whead^T (vocabulary padded to 128) -> next-token
// cross-entropy per row -> each sequence's loss summed over its rows in a fixed order.
//
// The weights come from split images (mca_tc_layout.h), 16 columns per chunk and one bulk copy per
// chunk, through five shared-memory stages run by one thread with full / empty mbarriers (a stage
// is refilled once the MMAs of its chunk completed, so the ring's depth sets how much of the
// copies' latency the MMAs hide); loads run ahead of the MMAs except across an attention step,
// whose K and V reuse the lo part of A and the first four stages. The
// images hold the current parameters: a candidate's changed weight W[i][j] enters as the rank-1 term
// delta * A[:, j] on output column i in that projection's epilogue, and a changed bias, LN or
// embedding parameter through a patched read. The commit kernel computes exactly what the
// evaluation computed (same images, same terms) and writes the cached residual streams and
// sequence losses; the image entry of the accepted weight is refreshed after it. In the trial loop
// the evaluation of candidate k < nscr also writes what the commit would write into scratch slot
// k, and an accepted candidate with a slot is adopted by copying it (the commit kernel returns;
// the copy kernel also refreshes the image entry).
#include <cstdio>

#include "mca_device.cuh"
#include "mca_internal.h"
#include "mca_tc.cuh"
#include "mca_tc_layout.h"
#include "mca_tfm.cuh"

namespace mca {
namespace {

constexpr int kThreads = 512;
constexpr int kRows = 128;                       // token rows per CTA: two sequences
constexpr int kD = kTcTfmD;
constexpr int kT = kTcTfmT;
constexpr int kHc = kTcTfmHc;
constexpr int kXLd = kD + 4;                     // residual row stride: conflict-free row access
constexpr int kStages = 5;
constexpr int kStageBytes = 16384;               // one chunk of 128 rows (64-row chunks use half)
constexpr int kXsBytes = kRows * kXLd * 4;       // 67,584
constexpr int kAloBytes = kRows * kD * 4;        // 65,536: lo part of A (K = 128)
constexpr int kSmem = kXsBytes + kAloBytes + kStages * kStageBytes;
constexpr uint32_t kALBO = (kRows / 8) * 128;    // A operands: K groups 2 KB apart, rows 16 B
constexpr uint32_t kIdN128 = tc_idesc_tf32(kRows, 128);
// tensor-memory columns
constexpr uint32_t kColQ = 0, kColK = 128, kColV = 256, kColA = 384;
constexpr uint32_t kColU = 0, kColF = 128, kColA2 = 256;   // Wo and the head also use kColU
constexpr uint32_t kColA2lo = 320;                         // lo part of A2 (K = 64)
// weight chunks of one block: Wq Wk Wv (24), Wo (8), then per pair p of hidden chunks W1 of the pair
// (8, N = 128) and W2 of its two chunks (4 + 4)
constexpr int kQkvChunks = 24, kWoChunk0 = 24, kFfnChunk0 = 32, kFfnPerPair = 16;
constexpr int kHp = kTcTfmHp;                    // hidden columns per W1 product
constexpr int kHeadChunks = 8;

static_assert(kSmem + 8 * 1024 <= 227 * 1024, "shared memory of the Transformer tensor-core kernel");
// K and V (2 x 64 KB) overlay the lo part of A and the first four stages
static_assert(2 * kRows * kD * 4 <= kAloBytes + 4 * kStageBytes, "K and V overlay");

__device__ __forceinline__ float prm(const TfmArgs& a, unsigned long long i,
                                     unsigned long long midx, float mval) {
  return i == midx ? mval : a.params[i];
}

// The weight matrix entry a parameter is (kTcMatNone for biases, LN parameters, embeddings).
struct Target {
  int mat, row, col;
};

__device__ __forceinline__ Target tc_target(const TfmArgs& a, unsigned long long idx, int stage) {
  Target t;
  t.mat = kTcMatNone;
  t.row = 0;
  t.col = 0;
  if (stage >= 0 && stage < a.nL) {
    const unsigned long long off = idx - a.o_blk0 - (unsigned long long)stage * a.blk_size;
    const unsigned long long dd = (unsigned long long)a.d * a.d, fd = (unsigned long long)a.F * a.d;
    const unsigned int rq[4] = {a.r_wq, a.r_wk, a.r_wv, a.r_wo};
#pragma unroll
    for (int m = 0; m < 4; ++m)
      if (off >= rq[m] && off < rq[m] + dd) {
        t.mat = m;
        t.row = (int)((off - rq[m]) / a.d);
        t.col = (int)((off - rq[m]) % a.d);
      }
    if (off >= a.r_w1 && off < a.r_w1 + fd) {
      t.mat = kTcW1;
      t.row = (int)((off - a.r_w1) / a.d);
      t.col = (int)((off - a.r_w1) % a.d);
    }
    if (off >= a.r_w2 && off < a.r_w2 + fd) {
      t.mat = kTcW2;
      t.row = (int)((off - a.r_w2) / a.F);
      t.col = (int)((off - a.r_w2) % a.F);
    }
  } else if (stage == a.nL && idx >= a.o_wh && idx < a.o_wh + (unsigned long long)a.V * a.d) {
    t.mat = kTcHead;
    t.row = (int)((idx - a.o_wh) / a.d);
    t.col = (int)((idx - a.o_wh) % a.d);
  }
  return t;
}

// Where candidate k's recomputation starts, from its proposal alone, as a key that orders the
// recomputations by length: 4 stage, plus 2 for a block's feed-forward sub-block, plus 3 for one of
// its hidden units (then block stage + 1, key 4 stage + 4, follows a short rank-1 step).
__device__ __forceinline__ int candidate_stage(const TfmArgs& a, int k) {
  unsigned int idx;
  if (a.n_explicit > 0) {
    idx = a.ex_idx[k];
  } else {
    const uint4 w = trial_words(a.seed, tfm_batch_tau(a) + (unsigned long long)k);
    idx = (unsigned int)(((unsigned long long)w.x * a.P) >> 32);
  }
  const int st = tfm_stage(a, idx);
  const int rs = tfm_restart(a, idx, st);
  return 4 * st + (rs == kRestartFfn ? 2 : rs == kRestartUnit ? 3 : 0);
}

struct Ctx {
  float* xs;                 // residual stream [128][kXLd]
  unsigned char* alo;        // lo part of A, core-matrix order (element (r, k) at (k/4) kALBO + 16 r)
  unsigned char* wst;        // weight stages
  float* ks;                 // K [128][128], 16-byte slots of a row swizzled by (row mod 8)
  float* vs;                 // V, same
  uint32_t tmem;             // tensor-memory base address
  uint32_t trow;             // this warp's lane quarter in a tensor-memory address
  int r, g, sl, t;           // token row, column part, sequence of the pair, position
  int b0s, nb, cpb, total;   // first block run, blocks run, chunks per block, chunks in all
  int q0, nbc;               // the first block's first chunk (its FFN's when ffn0), block chunks run
  bool ffn0;                 // the first block starts at its feed-forward sub-block
  bool unit0;                // a hidden unit of block cstage: rank-1 step, then block cstage + 1
  unsigned long long midx;   // patched parameter (~0: none)
  float mval, dlt;           // its value, and the change of a weight-matrix entry
  int cstage;                // the stage the candidate feeds (-1 embeddings)
  Target tg;
};

// State of the weight ring, in shared memory: nload belongs to the loading thread, nwait and
// ncommit to the MMA thread, limit is set before the CTA barrier that starts an MMA phase.
struct Issuer {
  int nload;                 // next chunk to load
  int limit;                 // chunks at or past this one may not be loaded yet
  int nwait;                 // chunks whose data arrived
  int ncommit;               // chunks whose MMAs were issued and committed
};

__device__ __forceinline__ void chunk_src(const TfmArgs& a, const Ctx& c, int x, const float*& src,
                                          uint32_t& bytes) {
  if (x < c.nbc) {
    const int xx = x + c.q0, jb = xx / c.cpb, q = xx - jb * c.cpb;
    const float* base = a.wimg + (size_t)(c.b0s + jb) * tfm_tc_block_floats(a.F);
    if (q < kFfnChunk0) {
      src = base + (size_t)q * 4096;
      bytes = 16384;
      return;
    }
    const int f = q - kFfnChunk0, p = f / kFfnPerPair, u = f - p * kFfnPerPair;
    if (u < 8) {                                 // W1 of pair p
      src = base + 131072 + (size_t)(p * 8 + u) * 4096;
    } else {                                     // W2 of hidden chunk 2p + (u - 8) / 4
      src = base + 131072 + (size_t)256 * a.F + (size_t)(p * 8 + u - 8) * 4096;
    }
    bytes = 16384;
  } else {
    src = a.wimg + (size_t)a.nL * tfm_tc_block_floats(a.F) + (size_t)(x - c.nbc) * 4096;
    bytes = 16384;
  }
}

// Load chunks up to (not including) `upto`, within the limit; a stage is reused once the MMAs of the
// chunk that held it completed.
__device__ bool topup(const TfmArgs& a, const Ctx& c, Issuer& is, int upto, uint64_t* full,
                      uint64_t* empty) {
  const int end = min(upto, is.limit);
  while (is.nload < end) {
    const int x = is.nload, st = x % kStages;
    if (x >= kStages && !mbar_wait(&empty[st], (uint32_t)((x - kStages) / kStages) & 1u))
      return false;
    const float* src;
    uint32_t bytes;
    chunk_src(a, c, x, src, bytes);
    bulk_load(smem_u32(c.wst + st * kStageBytes), src, bytes, &full[st]);
    ++is.nload;
  }
  return true;
}

// One thread: the MMAs of chunks x0 .. x0 + n - 1, each released to its stage's empty barrier. It
// waits only for each chunk's data; the stages are refilled by another thread (produce).
__device__ bool issue(const TfmArgs& a, const Ctx& c, Issuer& is, int x0, int n, uint64_t* full,
                      uint64_t* empty) {
  tc_fence_after();
  const uint32_t salo = smem_u32(c.alo), sw = smem_u32(c.wst);
  for (int x = x0; x < x0 + n; ++x) {
    const int st = x % kStages;
    if (!mbar_wait(&full[st], (uint32_t)(x / kStages) & 1u)) return false;
    is.nwait = x + 1;
    uint32_t dcol = kColU, idesc = kIdN128, alo = salo, acol = kColA, R = 128;
    bool lo_tm = false;                          // A's lo part in tensor memory (A2)
    int kc;
    bool first;
    if (x < c.nbc) {
      const int q = (x + c.q0) % c.cpb;
      if (q < kWoChunk0) {                       // Wq, Wk, Wv
        dcol = kColQ + 128u * (uint32_t)(q >> 3);
        kc = q & 7;
        first = kc == 0;
      } else if (q < kFfnChunk0) {               // Wo
        kc = q - kWoChunk0;
        first = kc == 0;
      } else {
        const int f = q - kFfnChunk0, p = f / kFfnPerPair, u = f - p * kFfnPerPair;
        if (u < 8) {                             // W1 of hidden pair p (N = 128)
          kc = u;
          first = kc == 0;
        } else {                                 // W2 of hidden chunk 2p + (u-8)/4, accumulated
          dcol = kColF;
          lo_tm = true;
          acol = kColA2;
          kc = (u - 8) & 3;
          first = p == 0 && u == 8;
        }
      }
    } else {                                     // head
      kc = x - c.nbc;
      first = kc == 0;
    }
    const uint32_t lbo = R * 16u;
#pragma unroll
    for (int ks = 0; ks < 2; ++ks) {
      const int gk = kc * 2 + ks;                // K step of 8 within the product
      const uint64_t da = umma_desc(alo + (uint32_t)gk * 2u * kALBO, kALBO, 128u);
      const uint32_t wb = sw + (uint32_t)(st * kStageBytes) + (uint32_t)ks * 2u * lbo;
      const uint64_t dwhi = umma_desc(wb, lbo, 128u);
      const uint64_t dwlo = umma_desc(wb + 4u * lbo, lbo, 128u);
      const uint32_t d = c.tmem + dcol, ta = c.tmem + acol + (uint32_t)gk * 8u;
      if (lo_tm)
        mma_ts(d, c.tmem + kColA2lo + (uint32_t)gk * 8u, dwhi, idesc, (first && ks == 0) ? 0u : 1u);
      else
        mma_ss(d, da, dwhi, idesc, (first && ks == 0) ? 0u : 1u);
      mma_ts(d, ta, dwlo, idesc, 1u);
      mma_ts(d, ta, dwhi, idesc, 1u);
    }
    umma_commit(&empty[st]);
    is.ncommit = x + 1;
  }
  return true;
}

// An MMA phase of chunks x0 .. x0 + n - 1: thread 0 issues the MMAs while thread 32 refills each
// stage as soon as the MMAs of its previous chunk complete, up to kStages - 1 chunks past the
// phase (within the limit), so that the MMA thread never waits for a refill. Both waits end by
// the time the phase's MMAs complete.
__device__ __forceinline__ void mma_phase(const TfmArgs& a, const Ctx& c, Issuer& is, int x0, int n,
                                          uint64_t* full, uint64_t* empty, volatile int* fail) {
  if (threadIdx.x == 0) {
    if (!issue(a, c, is, x0, n, full, empty)) *fail = 1;
  } else if (threadIdx.x == 32) {
    if (!topup(a, c, is, x0 + n - 1 + kStages, full, empty)) *fail = 1;
  }
}

// Every thread: wait for the MMAs of chunk `last` (and so of every earlier chunk); false, the same
// in every thread, if any wait of the CTA gave up.
__device__ __forceinline__ bool group_done(uint64_t* empty, int last, volatile int* s_fail) {
  if (!mbar_wait(&empty[last % kStages], (uint32_t)(last / kStages) & 1u)) *s_fail = 1;
  tc_fence_after();
  __syncthreads();
  return *s_fail == 0;
}

__device__ __forceinline__ void ld32(const Ctx& c, uint32_t col, float (&v)[32]) {
  float a0[16], a1[16];
  tmem_ld16(c.tmem + c.trow + col, a0);
  tmem_ld16(c.tmem + c.trow + col + 16u, a1);
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    v[i] = a0[i];
    v[16 + i] = a1[i];
  }
}

// v[i] += val for the one i == at (none if at is outside the array).
template <int N>
__device__ __forceinline__ void add_at(float (&v)[N], int at, float val) {
#pragma unroll
  for (int i = 0; i < N; ++i)
    if (i == at) v[i] += val;
}

// The A operand of row r, columns k0 .. k0 + 16 h - 1 (h = 1 or 2 halves): tf32 hi part into
// tensor-memory columns col .., lo part into the shared-memory operand lo_base.
template <int N>
__device__ __forceinline__ void store_a(const Ctx& c, const float (&v)[N], uint32_t col,
                                        unsigned char* lo_base, int k0) {
#pragma unroll
  for (int h = 0; h < N / 16; ++h) {
    float hi[16], lo[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      hi[q] = tf32_rna(v[16 * h + q]);
      lo[q] = tf32_rna(v[16 * h + q] - hi[q]);
    }
    tmem_st16(c.tmem + c.trow + col + 16u * (uint32_t)h, hi);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int k = k0 + 16 * h + 4 * q;
      *reinterpret_cast<float4*>(lo_base + (size_t)(k >> 2) * kALBO + (size_t)c.r * 16) =
          make_float4(lo[4 * q], lo[4 * q + 1], lo[4 * q + 2], lo[4 * q + 3]);
    }
  }
}

// The A2 operand of row r, columns k0 .. k0 + 15: tf32 hi and lo parts into tensor-memory columns
// col .. and lo_col .. .
__device__ __forceinline__ void store_a2(const Ctx& c, const float (&v)[16], uint32_t col,
                                         uint32_t lo_col) {
  float hi[16], lo[16];
#pragma unroll
  for (int q = 0; q < 16; ++q) {
    hi[q] = tf32_rna(v[q]);
    lo[q] = tf32_rna(v[q] - hi[q]);
  }
  tmem_st16(c.tmem + c.trow + col, hi);
  tmem_st16(c.tmem + c.trow + lo_col, lo);
}

// Layer norm of row r (its 32 columns here, statistics over all four parts) written as the A
// operand; the normalised value of column `stash` (if it is one of this thread's) to s_acol[r].
__device__ void ln_to_a(const TfmArgs& a, const Ctx& c, unsigned long long og,
                        unsigned long long ob, int stash, float* s_part, float* s_acol) {
  float x[32];
  const float* xr = c.xs + c.r * kXLd + 32 * c.g;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float4 v = *reinterpret_cast<const float4*>(xr + 4 * i);
    x[4 * i] = v.x;
    x[4 * i + 1] = v.y;
    x[4 * i + 2] = v.z;
    x[4 * i + 3] = v.w;
  }
  float s = 0.0f;
#pragma unroll
  for (int i = 0; i < 32; ++i) s += x[i];
  s_part[c.g * kRows + c.r] = s;
  __syncthreads();
  const float mean = (((s_part[c.r] + s_part[kRows + c.r]) + s_part[2 * kRows + c.r]) +
                      s_part[3 * kRows + c.r]) / (float)kD;
  float v = 0.0f;
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const float e = x[i] - mean;
    v = fmaf(e, e, v);
  }
  s_part[(4 + c.g) * kRows + c.r] = v;
  __syncthreads();
  const float var = (((s_part[4 * kRows + c.r] + s_part[5 * kRows + c.r]) +
                      s_part[6 * kRows + c.r]) + s_part[7 * kRows + c.r]) / (float)kD;
  const float rstd = rsqrtf(var + a.eps);
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const unsigned long long col = (unsigned long long)(32 * c.g + i);
    x[i] = (x[i] - mean) * rstd * prm(a, og + col, c.midx, c.mval) + prm(a, ob + col, c.midx, c.mval);
  }
#pragma unroll
  for (int i = 0; i < 32; ++i)
    if (32 * c.g + i == stash) s_acol[c.r] = x[i];
  store_a<32>(c, x, kColA + 32u * (uint32_t)c.g, c.alo, 32 * c.g);
}

// A candidate in W1, b1, W2 or b2 of block b changes one hidden unit j of the block's feed-forward
// network, so the block's output stream (cached) moves by a rank-1 term: by W2[:, j] (f(u'_j) -
// f(u_j)) for W1[j][k] and b1[j], by delta f(u_j) on column i for W2[i][j], by delta on column i
// for b2[i], with u_j = LN2(mid stream) . W1[j, :] + b1[j] recomputed here on the CUDA cores (the
// candidate's own entry at its old value: in a commit the parameter already holds the new one).
// The new output stream of this thread's row part goes to xr.
__device__ void ffn_unit(const TfmArgs& a, const Ctx& c, const DeepCand& cd, int s0, float* xr,
                         float* s_part, float* s_acol) {
  const int b = cd.layer;
  const unsigned long long base = a.o_blk0 + (unsigned long long)b * a.blk_size;
  const unsigned long long off = (unsigned long long)cd.idx - base;
  const size_t seq_floats = (size_t)kT * kD;
  int kind, j = 0, i0 = -1, kcol = -1;       // kind: 0 W1[j][kcol], 1 b1[j], 2 W2[i0][j], 3 b2[i0]
  if (off < a.r_b1) {
    kind = 0;
    j = (int)((off - a.r_w1) / kD);
    kcol = (int)((off - a.r_w1) % kD);
  } else if (off < a.r_w2) {
    kind = 1;
    j = (int)(off - a.r_b1);
  } else if (off < a.r_b2) {
    kind = 2;
    i0 = (int)((off - a.r_w2) / (unsigned long long)a.F);
    j = (int)((off - a.r_w2) % (unsigned long long)a.F);
  } else {
    kind = 3;
    i0 = (int)(off - a.r_b2);
  }
  const size_t row = ((size_t)(s0 + c.sl)) * seq_floats + (size_t)c.t * kD + 32 * c.g;
  float xn[32];
  const float* xo = a.X + (size_t)(b + 1) * a.B * seq_floats + row;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float4 v = reinterpret_cast<const float4*>(xo)[i];
    xn[4 * i] = v.x;
    xn[4 * i + 1] = v.y;
    xn[4 * i + 2] = v.z;
    xn[4 * i + 3] = v.w;
  }
  if (kind == 3) {
    add_at(xn, i0 - 32 * c.g, cd.delta);
  } else {
    float x[32];
    const float* xm = a.Xmid + (size_t)b * a.B * seq_floats + row;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float4 v = reinterpret_cast<const float4*>(xm)[i];
      x[4 * i] = v.x;
      x[4 * i + 1] = v.y;
      x[4 * i + 2] = v.z;
      x[4 * i + 3] = v.w;
    }
    float sm = 0.0f;
#pragma unroll
    for (int i = 0; i < 32; ++i) sm += x[i];
    s_part[c.g * kRows + c.r] = sm;
    __syncthreads();
    const float mean = (((s_part[c.r] + s_part[kRows + c.r]) + s_part[2 * kRows + c.r]) +
                        s_part[3 * kRows + c.r]) / (float)kD;
    float v = 0.0f;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const float e = x[i] - mean;
      v = fmaf(e, e, v);
    }
    s_part[(4 + c.g) * kRows + c.r] = v;
    __syncthreads();
    const float var = (((s_part[4 * kRows + c.r] + s_part[5 * kRows + c.r]) +
                        s_part[6 * kRows + c.r]) + s_part[7 * kRows + c.r]) / (float)kD;
    const float rstd = rsqrtf(var + a.eps);
    const unsigned long long w1 = base + a.r_w1 + (unsigned long long)j * kD;
    float p = 0.0f;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const int col = 32 * c.g + i;
      const float ln = (x[i] - mean) * rstd * a.params[base + a.r_ln2g + col] +
                       a.params[base + a.r_ln2b + col];
      if (col == kcol) s_acol[c.r] = ln;
      const float w = w1 + col == cd.idx ? cd.oldw : a.params[w1 + col];
      p = fmaf(ln, w, p);
    }
    s_part[c.g * kRows + c.r] = p;           // every thread has read the means (barrier above)
    __syncthreads();
    const float bj = kind == 1 ? cd.oldw : a.params[base + a.r_b1 + j];
    const float u = ((((s_part[c.r] + s_part[kRows + c.r]) + s_part[2 * kRows + c.r]) +
                      s_part[3 * kRows + c.r])) + bj;
    if (kind == 2) {
      add_at(xn, i0 - 32 * c.g, cd.delta * act_rt(a.act, u, a.g));
    } else {
      const float un = kind == 0 ? fmaf(cd.delta, s_acol[c.r], u) : u + cd.delta;
      const float da = act_rt(a.act, un, a.g) - act_rt(a.act, u, a.g);
      const unsigned long long w2 = base + a.r_w2 + (unsigned long long)j;
#pragma unroll
      for (int i = 0; i < 32; ++i)
        xn[i] = fmaf(a.params[w2 + (unsigned long long)(32 * c.g + i) * a.F], da, xn[i]);
    }
  }
#pragma unroll
  for (int i = 0; i < 8; ++i)
    *reinterpret_cast<float4*>(xr + 4 * i) =
        make_float4(xn[4 * i], xn[4 * i + 1], xn[4 * i + 2], xn[4 * i + 3]);
}

// Causal attention of query row r with head g over the keys of its sequence (K and V in shared
// memory), with a running maximum and sum over blocks of 8 keys.
__device__ __forceinline__ void attention(const Ctx& c, const float (&q)[32], float (&o)[32]) {
  const float scale = rsqrtf(32.0f);
  const float* kb = c.ks + (size_t)(c.sl * kT) * kD + 32 * c.g;
  const float* vb = c.vs + (size_t)(c.sl * kT) * kD + 32 * c.g;
  float m = -INFINITY, l = 0.0f;
#pragma unroll
  for (int i = 0; i < 32; ++i) o[i] = 0.0f;
  const int jend = (c.t | 31) + 1;               // the same for every lane of the warp
  for (int j0 = 0; j0 < jend; j0 += 8) {
    float sc[8];
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
      const float* kr = kb + (size_t)(j0 + jj) * kD;
      float s = 0.0f;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float4 kv = *reinterpret_cast<const float4*>(kr + 4 * (i ^ jj));
        s = fmaf(q[4 * i], kv.x, s);
        s = fmaf(q[4 * i + 1], kv.y, s);
        s = fmaf(q[4 * i + 2], kv.z, s);
        s = fmaf(q[4 * i + 3], kv.w, s);
      }
      sc[jj] = j0 + jj <= c.t ? s * scale : -INFINITY;
    }
    float bm = sc[0];
#pragma unroll
    for (int jj = 1; jj < 8; ++jj) bm = fmaxf(bm, sc[jj]);
    const float mn = fmaxf(m, bm);               // finite: key 0 is in the first block
    const float corr = __expf(m - mn);
    l *= corr;
#pragma unroll
    for (int i = 0; i < 32; ++i) o[i] *= corr;
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
      const float p = __expf(sc[jj] - mn);
      l += p;
      const float* vr = vb + (size_t)(j0 + jj) * kD;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float4 vv = *reinterpret_cast<const float4*>(vr + 4 * (i ^ jj));
        o[4 * i] = fmaf(p, vv.x, o[4 * i]);
        o[4 * i + 1] = fmaf(p, vv.y, o[4 * i + 1]);
        o[4 * i + 2] = fmaf(p, vv.z, o[4 * i + 2]);
        o[4 * i + 3] = fmaf(p, vv.w, o[4 * i + 3]);
      }
    }
    m = mn;
  }
  const float inv = 1.0f / l;
#pragma unroll
  for (int i = 0; i < 32; ++i) o[i] *= inv;
}

template <int MODE>
__global__ void __launch_bounds__(kThreads, 1) tfm_tc_kernel(TfmArgs a) {
  extern __shared__ __align__(1024) unsigned char tsm[];
  __shared__ DeepCand s_c;
  __shared__ int s_tok[2][kT + 1];
  __shared__ float s_part[8 * kRows];
  __shared__ float s_acol[kRows];
  __shared__ float s_zy[kRows];
  __shared__ float s_rowv[kRows];
  __shared__ int s_stage[kKmax];
  __shared__ __align__(8) uint64_t s_full[kStages], s_empty[kStages];
  __shared__ uint32_t s_tmem;
  __shared__ int s_fail, s_k;
  __shared__ int s_skip[2];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  Ctx c;
  c.g = warp >> 2;
  c.r = (warp & 3) * 32 + lane;
  c.sl = c.r / kT;
  c.t = c.r % kT;
  c.trow = (uint32_t)((warp & 3) * 32) << 16;
  c.xs = reinterpret_cast<float*>(tsm);
  c.alo = tsm + kXsBytes;
  c.wst = c.alo + kAloBytes;
  c.ks = reinterpret_cast<float*>(c.alo);
  c.vs = c.ks + kRows * kD;
  // the commit recomputes an accepted candidate that has no scratch slot (kstar >= nscr); one with
  // a slot is adopted from it by tfm_tc_adopt_kernel
  if (MODE == kTfmCommit && a.ctl->kstar < a.nscr) return;
  int k = 0, pair = blockIdx.x;
  if (MODE == kTfmEval) {
    // Longest recomputations first: CTAs start in linear block order, so the linear index is
    // mapped to (candidate rank, sequence pair) with the candidates ranked by the stage they feed
    // (earlier = longer), ties by index.
    const int Kb = gridDim.x, npair = gridDim.y;
    const int lid = blockIdx.x + blockIdx.y * gridDim.x;
    const int rank = lid / npair;
    pair = lid - rank * npair;
    if (tid < Kb) s_stage[tid] = candidate_stage(a, tid);
    __syncthreads();
    if (tid < Kb) {
      const int my = s_stage[tid];
      int rk = 0;
      for (int q = 0; q < Kb; ++q) rk += (s_stage[q] < my || (s_stage[q] == my && q < tid)) ? 1 : 0;
      if (rk == rank) s_k = tid;
    }
    __syncthreads();
    k = s_k;
  }
  const int s0 = 2 * pair;
  if (tid == 0) {
    if (MODE == kTfmEval) {
      s_c = tfm_candidate(a, k);
    } else if (MODE == kTfmCommit) {
      s_c = a.ctl->acc;
    } else {
      DeepCand d;
      d.idx = 0xffffffffu;
      d.layer = -1;
      d.row = -1;
      d.col = 0;
      d.oldw = d.neww = 0.0f;
      d.delta = 1.0f;
      d.new_code = 0;
      d.valid = 1;
      s_c = d;
    }
    s_fail = 0;
  }
  for (int e = tid; e < 2 * (kT + 1); e += kThreads)
    s_tok[e / (kT + 1)][e % (kT + 1)] = a.tokens[(size_t)s0 * (kT + 1) + e];
  __syncthreads();
  const DeepCand cd = s_c;
  float* part = a.partial + (size_t)k * a.B + s0;
  if (MODE == kTfmEval && k >= tfm_batch_width(a, tfm_batch_tau(a))) {   // past the run's end
    if (tid < 2) part[tid] = 0.0f;
    return;
  }
  // where the recomputed residual streams and sequence losses go: the handle's (commit, forward)
  // or, in an evaluation, the candidate's scratch slot when it has one
  const size_t seq_floats = (size_t)kT * kD;
  const bool slot = MODE == kTfmEval && k < a.nscr;
  float* const xout = MODE != kTfmEval ? a.X
                      : slot ? a.scrX + (size_t)k * (size_t)(2 * a.nL + 1) * a.B * seq_floats
                             : nullptr;
  float* const xmout = MODE != kTfmEval ? a.Xmid
                       : slot ? xout + (size_t)(a.nL + 1) * a.B * seq_floats : nullptr;
  float* const lout = MODE != kTfmEval ? a.ell : slot ? a.scr_ell + (size_t)k * a.B : nullptr;
  if (!cd.valid || cd.delta == 0.0f) {
    if (MODE == kTfmEval && tid < 2) part[tid] = 0.0f;
    return;
  }
  if (tid < 2) {                 // a tok_emb entry: a sequence without that token is unchanged
    int skip = 0;
    if (MODE != kTfmForward && cd.row >= 0) {
      skip = 1;
      for (int t = 0; t < kT; ++t) skip &= s_tok[tid][t] != cd.row;
    }
    s_skip[tid] = skip;
  }
  __syncthreads();
  if (s_skip[0] && s_skip[1]) {
    if (MODE == kTfmEval && tid < 2) part[tid] = 0.0f;
    return;
  }
  const bool fwd = MODE == kTfmForward;
  c.midx = fwd ? ~0ull : (unsigned long long)cd.idx;
  c.mval = cd.neww;
  c.dlt = fwd ? 0.0f : cd.delta;
  c.cstage = fwd ? -1 : cd.layer;
  if (fwd) {
    c.tg.mat = kTcMatNone;
    c.tg.row = c.tg.col = 0;
  } else {
    c.tg = tc_target(a, cd.idx, cd.layer);
  }
  const int b0 = (fwd || cd.layer < 0) ? -1 : cd.layer;
  const int rs = fwd ? kRestartBlock : tfm_restart(a, cd.idx, cd.layer);
  c.unit0 = rs == kRestartUnit;
  c.b0s = b0 < 0 ? 0 : b0 + (c.unit0 ? 1 : 0);
  c.nb = a.nL - c.b0s;
  c.cpb = kFfnChunk0 + kFfnPerPair * (a.F / kHp);
  c.ffn0 = rs == kRestartFfn;
  c.q0 = c.ffn0 ? kFfnChunk0 : 0;
  c.nbc = c.nb * c.cpb - c.q0;
  c.total = c.nbc + kHeadChunks;

  // tensor memory, the stage ring, the first chunks
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;"
                 ::"r"(smem_u32(&s_tmem)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  __shared__ Issuer s_is;
  Issuer& is = s_is;
  if (tid == 0) {
    is.nload = is.nwait = is.ncommit = 0;
    // loads stop at the first output projection after an attention step (K and V take the stages)
    is.limit = c.nb == 0 ? kHeadChunks
               : !c.ffn0 ? kWoChunk0
               : c.nb > 1 ? c.cpb - c.q0 + kWoChunk0 : c.total;
  }
  if (tid == 0) {
    for (int q = 0; q < kStages; ++q) {
      mbar_init(&s_full[q], 1);
      mbar_init(&s_empty[q], 1);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    topup(a, c, is, kStages, s_full, s_empty);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  c.tmem = s_tmem;

  // residual stream entering the first stage run
  float* xr = c.xs + c.r * kXLd + 32 * c.g;
  if (b0 < 0) {
    const int tok = s_tok[c.sl][c.t];
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const unsigned long long col = (unsigned long long)(32 * c.g + i);
      xr[i] = prm(a, a.o_tok + (unsigned long long)tok * kD + col, c.midx, c.mval) +
              prm(a, a.o_pos + (unsigned long long)c.t * kD + col, c.midx, c.mval);
    }
    if (xout && !s_skip[c.sl]) {
      float* dst = xout + (size_t)(s0 + c.sl) * seq_floats + (size_t)c.t * kD + 32 * c.g;
#pragma unroll
      for (int i = 0; i < 8; ++i)
        reinterpret_cast<float4*>(dst)[i] = *reinterpret_cast<const float4*>(xr + 4 * i);
    }
  } else if (c.unit0) {
    ffn_unit(a, c, cd, s0, xr, s_part, s_acol);
    if (xout) {                  // block b0's new output stream
      float* dst = xout + ((size_t)(b0 + 1) * a.B + s0 + c.sl) * seq_floats + (size_t)c.t * kD + 32 * c.g;
#pragma unroll
      for (int i = 0; i < 8; ++i)
        reinterpret_cast<float4*>(dst)[i] = *reinterpret_cast<const float4*>(xr + 4 * i);
    }
  } else {
    const float* src = (c.ffn0 ? a.Xmid : a.X) + ((size_t)b0 * a.B + s0 + c.sl) * seq_floats +
                       (size_t)c.t * kD + 32 * c.g;
#pragma unroll
    for (int i = 0; i < 8; ++i)
      *reinterpret_cast<float4*>(xr + 4 * i) = reinterpret_cast<const float4*>(src)[i];
  }

  volatile int* fail = &s_fail;
  int gc = 0;                    // next chunk whose MMAs are issued (the same in every thread)
  bool ok = true;
  const int nP = a.F / kHp;
  for (int b = c.b0s; ok && b < a.nL; ++b) {
    const bool here = b == c.cstage;
    const unsigned long long base = a.o_blk0 + (unsigned long long)b * a.blk_size;
    if (!(c.ffn0 && b == c.b0s)) {   // (a feed-forward candidate's block starts at its mid stream)
      // ---- attention: LN1, Q K V, attention, output projection
      ln_to_a(a, c, base + a.r_ln1g, base + a.r_ln1b,
              (here && c.tg.mat >= kTcQ && c.tg.mat <= kTcV) ? c.tg.col : -1, s_part, s_acol);
      tc_publish_operands();
      __syncthreads();
      mma_phase(a, c, is, gc, kQkvChunks, s_full, s_empty, fail);
      gc += kQkvChunks;
      if (!(ok = group_done(s_empty, gc - 1, fail))) break;
      float q[32];
      {
        float v[32];
#pragma unroll
        for (int p = 0; p < 2; ++p) {
          ld32(c, (p ? kColV : kColK) + 32u * (uint32_t)c.g, v);
          const unsigned long long bb = base + (p ? a.r_bv : a.r_bk) + 32 * c.g;
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] += prm(a, bb + i, c.midx, c.mval);
          if (here && c.tg.mat == (p ? kTcV : kTcK)) add_at(v, c.tg.row - 32 * c.g, c.dlt * s_acol[c.r]);
          float* dst = (p ? c.vs : c.ks) + (size_t)c.r * kD + 32 * c.g;
#pragma unroll
          for (int i = 0; i < 8; ++i)
            *reinterpret_cast<float4*>(dst + 4 * (i ^ (c.r & 7))) =
                make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
        }
        ld32(c, kColQ + 32u * (uint32_t)c.g, q);
        const unsigned long long bq = base + a.r_bq + 32 * c.g;
#pragma unroll
        for (int i = 0; i < 32; ++i) q[i] += prm(a, bq + i, c.midx, c.mval);
        if (here && c.tg.mat == kTcQ) add_at(q, c.tg.row - 32 * c.g, c.dlt * s_acol[c.r]);
      }
      __syncthreads();             // K and V complete
      {
        float o[32];
        attention(c, q, o);
        __syncthreads();           // every row done with K and V: their memory takes the next A
        if (here && c.tg.mat == kTcO) {
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (32 * c.g + i == c.tg.col) s_acol[c.r] = o[i];
        }
        store_a<32>(c, o, kColA + 32u * (uint32_t)c.g, c.alo, 32 * c.g);
      }
      if (tid == 0) {              // loads may now run into the next block's Q, K, V chunks
        const int jb = b - c.b0s;
        is.limit = jb + 1 < c.nb ? (jb + 1) * c.cpb - c.q0 + kWoChunk0 : c.total;
      }
      tc_publish_operands();
      __syncthreads();
      mma_phase(a, c, is, gc, kFfnChunk0 - kWoChunk0, s_full, s_empty, fail);
      gc += kFfnChunk0 - kWoChunk0;
      if (!(ok = group_done(s_empty, gc - 1, fail))) break;
      {
        float v[32];
        ld32(c, kColU + 32u * (uint32_t)c.g, v);
        if (here && c.tg.mat == kTcO) add_at(v, c.tg.row - 32 * c.g, c.dlt * s_acol[c.r]);
        const unsigned long long bo = base + a.r_bo + 32 * c.g;
#pragma unroll
        for (int i = 0; i < 32; ++i) xr[i] += v[i] + prm(a, bo + i, c.midx, c.mval);
      }
      if (xmout && !s_skip[c.sl]) {    // the mid stream: block b after its attention sub-block
        float* dst = xmout + ((size_t)b * a.B + s0 + c.sl) * seq_floats + (size_t)c.t * kD + 32 * c.g;
#pragma unroll
        for (int i = 0; i < 8; ++i)
          reinterpret_cast<float4*>(dst)[i] = *reinterpret_cast<const float4*>(xr + 4 * i);
      }
    }
    // ---- feed-forward network: W1 for two 64-wide hidden chunks at a time (N = 128), then per
    // chunk the activation as A2 and its W2 product
    ln_to_a(a, c, base + a.r_ln2g, base + a.r_ln2b, (here && c.tg.mat == kTcW1) ? c.tg.col : -1,
            s_part, s_acol);
    tc_publish_operands();
    __syncthreads();
    mma_phase(a, c, is, gc, 8, s_full, s_empty, fail);
    gc += 8;
    for (int h = 0; h < 2 * nP; ++h) {
      if (!(ok = group_done(s_empty, gc - 1, fail))) break;
      // this thread's 16 hidden units of chunk h, from the pair's U (columns 0-63 or 64-127)
      float u[16];
      tmem_ld16(c.tmem + c.trow + kColU + (uint32_t)((h & 1) * kHc) + 16u * (uint32_t)c.g, u);
      const int f0 = h * kHc + 16 * c.g;
      if (here && c.tg.mat == kTcW1) add_at(u, c.tg.row - f0, c.dlt * s_acol[c.r]);
#pragma unroll
      for (int i = 0; i < 16; ++i)
        u[i] = act_rt(a.act, u[i] + prm(a, base + a.r_b1 + f0 + i, c.midx, c.mval), a.g);
      if (here && c.tg.mat == kTcW2) {
#pragma unroll
        for (int i = 0; i < 16; ++i)
          if (f0 + i == c.tg.col) s_acol[c.r] = u[i];
      }
      store_a2(c, u, kColA2 + 16u * (uint32_t)c.g, kColA2lo + 16u * (uint32_t)c.g);
      tc_publish_operands();
      __syncthreads();
      // W2 of chunk h; after a pair's second chunk (its U fully read) also W1 of the next pair
      const int n = (h & 1) && h + 1 < 2 * nP ? 12 : 4;
      mma_phase(a, c, is, gc, n, s_full, s_empty, fail);
      gc += n;
    }
    if (!ok || !(ok = group_done(s_empty, gc - 1, fail))) break;
    {
      float v[32];
      ld32(c, kColF + 32u * (uint32_t)c.g, v);
      if (here && c.tg.mat == kTcW2) add_at(v, c.tg.row - 32 * c.g, c.dlt * s_acol[c.r]);
      const unsigned long long b2 = base + a.r_b2 + 32 * c.g;
#pragma unroll
      for (int i = 0; i < 32; ++i) xr[i] += v[i] + prm(a, b2 + i, c.midx, c.mval);
    }
    if (xout && !s_skip[c.sl]) {
      float* dst = xout + ((size_t)(b + 1) * a.B + s0 + c.sl) * seq_floats + (size_t)c.t * kD + 32 * c.g;
#pragma unroll
      for (int i = 0; i < 8; ++i)
        reinterpret_cast<float4*>(dst)[i] = *reinterpret_cast<const float4*>(xr + 4 * i);
    }
  }

  // ---- final layer norm, head, next-token cross-entropy
  if (ok) {
    const bool here = c.cstage == a.nL;
    ln_to_a(a, c, a.o_lnf_g, a.o_lnf_b, (here && c.tg.mat == kTcHead) ? c.tg.col : -1, s_part,
            s_acol);
    tc_publish_operands();
    __syncthreads();
    mma_phase(a, c, is, gc, kHeadChunks, s_full, s_empty, fail);
    gc += kHeadChunks;
    ok = group_done(s_empty, gc - 1, fail);
  }
  if (ok) {
    const bool here = c.cstage == a.nL;
    float z[32];
    ld32(c, kColU + 32u * (uint32_t)c.g, z);
    if (here && c.tg.mat == kTcHead) add_at(z, c.tg.row - 32 * c.g, c.dlt * s_acol[c.r]);
    float zmax = -INFINITY;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const int col = 32 * c.g + i;
      z[i] = col < a.V ? z[i] + prm(a, a.o_bh + (unsigned long long)col, c.midx, c.mval) : -INFINITY;
      zmax = fmaxf(zmax, z[i]);
    }
    s_part[c.g * kRows + c.r] = zmax;
    __syncthreads();
    const float m = fmaxf(fmaxf(fmaxf(s_part[c.r], s_part[kRows + c.r]), s_part[2 * kRows + c.r]),
                          s_part[3 * kRows + c.r]);
    float se = 0.0f;
    const int y = s_tok[c.sl][c.t + 1];
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      if (32 * c.g + i < a.V) se += __expf(z[i] - m);
      if (32 * c.g + i == y) s_zy[c.r] = z[i];
    }
    s_part[(4 + c.g) * kRows + c.r] = se;
    __syncthreads();
    if (c.g == 0) {
      const float sum = ((s_part[4 * kRows + c.r] + s_part[5 * kRows + c.r]) +
                         s_part[6 * kRows + c.r]) + s_part[7 * kRows + c.r];
      s_rowv[c.r] = (__logf(sum) + m) - s_zy[c.r];
    }
    __syncthreads();
    if (tid < 2) {
      float l = 0.0f;
      for (int t = 0; t < kT; ++t) l += s_rowv[tid * kT + t];
      if (MODE == kTfmEval) part[tid] = s_skip[tid] ? 0.0f : l - a.ell[s0 + tid];
      if (lout && !s_skip[tid]) lout[s0 + tid] = l;
    }
  }

  if (!ok && tid == 0) {
    // copies still in flight land before the CTA ends, and issued MMAs finish before the
    // tensor memory is released (both bounded)
    for (int x = is.nwait; x < is.nload; ++x) mbar_wait(&s_full[x % kStages], (uint32_t)(x / kStages) & 1u);
    if (is.ncommit > 0) {
      const int x = is.ncommit - 1;
      mbar_wait(&s_empty[x % kStages], (uint32_t)(x / kStages) & 1u);
    }
    atomicCAS(&a.st->err, 0, (int)MCA_ERR_TIMEOUT);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(c.tmem));
}

// Split images of every weight matrix (hi = tf32(W), lo = tf32(W - hi)); head rows past the
// vocabulary are zero. blockIdx.y = 6 b + matrix (Wq, Wk, Wv, Wo, W1, W2) or 6 nL for the head.
__global__ void tfm_tc_split_kernel(TfmArgs a) {
  const int slot = blockIdx.y;
  int mat, b = 0, rows = kD, cols = kD;
  unsigned long long src;
  if (slot == 6 * a.nL) {
    mat = kTcHead;
    src = a.o_wh;
  } else {
    b = slot / 6;
    mat = slot % 6;
    const unsigned long long base = a.o_blk0 + (unsigned long long)b * a.blk_size;
    const unsigned int off[6] = {a.r_wq, a.r_wk, a.r_wv, a.r_wo, a.r_w1, a.r_w2};
    src = base + off[mat];
    if (mat == kTcW1) rows = a.F;
    if (mat == kTcW2) cols = a.F;
  }
  const size_t lo = tc_image_lo(tfm_tc_rows(mat));
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < rows * cols; e += gridDim.x * blockDim.x) {
    const int r = e / cols, kk = e - r * cols;
    const float w = (mat == kTcHead && r >= a.V) ? 0.0f : a.params[src + (unsigned long long)e];
    const float hi = tf32_rna(w);
    const size_t o = tfm_tc_image_offset(mat, b, r, kk, a.F, a.nL);
    a.wimg[o] = hi;
    a.wimg[o + lo] = tf32_rna(w - hi);
  }
}

// The image entry of the accepted weight-matrix parameter (after the commit kernel, which reads the
// old one).
__device__ void image_update(const TfmArgs& a, const DeepCand& c) {
  const Target tg = tc_target(a, c.idx, c.layer);
  if (tg.mat == kTcMatNone) return;
  const float w = a.params[c.idx];
  const float hi = tf32_rna(w);
  const size_t o = tfm_tc_image_offset(tg.mat, c.layer, tg.row, tg.col, a.F, a.nL);
  a.wimg[o] = hi;
  a.wimg[o + tc_image_lo(tfm_tc_rows(tg.mat))] = tf32_rna(w - hi);
}

// After the decision and the commit kernel: the image entry of the accepted weight (CTA (0, 0)),
// and, for an accepted candidate with a scratch slot, its residual streams (those its evaluation
// recomputed: X[0 ..] and Xmid[0 ..] for an embedding; X[b + 1 ..] and Xmid[b ..] for block b,
// Xmid[b + 1 ..] for its feed-forward sub-block; none for the final LN and head) and sequence
// losses, copied from the slot. CTA (s, x) copies sequence s of stream x (X for x <= nL, then
// Xmid); sequences the evaluation skipped (a token embedding whose token they do not contain) keep
// theirs.
__global__ void tfm_tc_adopt_kernel(TfmArgs a) {
  const int ks = a.ctl->kstar;
  if (ks < 0) return;
  const DeepCand cd = a.ctl->acc;
  if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0) image_update(a, cd);
  if (ks >= a.nscr || !cd.valid || cd.delta == 0.0f) return;
  const int s = blockIdx.x, x = blockIdx.y;
  __shared__ int s_skip;
  if (threadIdx.x == 0) {
    int skip = 0;
    if (cd.row >= 0) {
      skip = 1;
      for (int t = 0; t < kT; ++t) skip &= a.tokens[(size_t)s * (kT + 1) + t] != cd.row;
    }
    s_skip = skip;
  }
  __syncthreads();
  if (s_skip) return;
  if (x == 0 && threadIdx.x == 0) a.ell[s] = a.scr_ell[(size_t)ks * a.B + s];
  const bool mid = x > a.nL;
  const int xs = mid ? x - a.nL - 1 : x;                // stream within X or Xmid
  const int first = cd.layer < 0 ? 0
                    : mid && !tfm_ffn_param(a, cd.idx, cd.layer) ? cd.layer : cd.layer + 1;
  if (xs < first) return;
  const size_t seq_floats = (size_t)kT * kD;
  const size_t at = ((size_t)xs * a.B + s) * seq_floats;
  const float* sb = a.scrX + (size_t)ks * (size_t)(2 * a.nL + 1) * a.B * seq_floats +
                    (mid ? (size_t)(a.nL + 1) * a.B * seq_floats : 0);
  const float4* src = reinterpret_cast<const float4*>(sb + at);
  float4* dst = reinterpret_cast<float4*>((mid ? a.Xmid : a.X) + at);
  for (int q = threadIdx.x; q < (int)(seq_floats / 4); q += blockDim.x) dst[q] = src[q];
}

template <int MODE>
cudaError_t launch_tc(const TfmArgs& a, dim3 grid, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute((const void*)tfm_tc_kernel<MODE>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  if (e != cudaSuccess) return e;
  tfm_tc_kernel<MODE><<<grid, kThreads, kSmem, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_tfm_tc_split(const TfmArgs& a, cudaStream_t s) {
  tfm_tc_split_kernel<<<dim3(32, 6 * a.nL + 1), 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_tfm_tc_eval(const TfmArgs& a, cudaStream_t s) {
  const int Kb = a.n_explicit > 0 ? a.n_explicit : a.Kb;
  return launch_tc<kTfmEval>(a, dim3(Kb, a.B / 2), s);
}

cudaError_t launch_tfm_tc_commit(const TfmArgs& a, cudaStream_t s) {
  return launch_tc<kTfmCommit>(a, dim3(a.B / 2), s);
}

cudaError_t launch_tfm_tc_forward(const TfmArgs& a, cudaStream_t s) {
  return launch_tc<kTfmForward>(a, dim3(a.B / 2), s);
}

cudaError_t launch_tfm_tc_adopt(const TfmArgs& a, cudaStream_t s) {
  tfm_tc_adopt_kernel<<<dim3(a.B, 2 * a.nL + 1), 256, 0, s>>>(a);
  return cudaGetLastError();
}


}  // namespace mca
