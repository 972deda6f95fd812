// Internal declarations shared by the C-ABI layer (mca_api.cu) and the kernels.
#pragma once

#include <cstdint>
#include <string>
#include <vector>

#include <cuda_runtime.h>

#include "../../include/mca.h"

namespace mca {

struct GridBarrier;

constexpr int kKmax = 128;        // speculative candidates per batch
constexpr int kMaxC = 14;         // output fields a sample record holds
constexpr int kSR = 16;           // fields per sample record: outputs [0, C), loss 14, label 15
constexpr int kMaxClasses = kSR - 2;
constexpr int kLoopThreads = 512; // threads per CTA of the trial-loop kernel
constexpr int kLoopWarps = kLoopThreads / 32;
constexpr int kMaxSubs = 8;       // sub-chunks of one candidate inside one sample range
constexpr int kRangeTarget = 64;
// Batch width of the single-hidden-layer loop: ceil(c / p) candidates, p = (A + 0.5) / (T + 1) from
// counts decayed per batch.
constexpr float kRateDecay = 0.95f;
constexpr float kWidthMlp2 = 2.0f;
// Host-driven batches (deep nets, the Transformer): a batch of K candidates consumes
// (1 - (1 - p)^K) / p trials on average and costs about r + K candidate evaluations, r being its
// fixed part (decision, adoption or commit, launch gaps, the last partial wave of CTAs). The width
// maximises trials per cost. r was fitted to fixed-width runs on GB300 (batch time against K):
// about 1.9 candidate-times for the 24 x 256 chain at N = 10000, 0.5 for the d_model 128
// Transformer on 256 sequences.
constexpr float kBatchCostDeep = 1.9f;
constexpr float kBatchCostTfm = 0.5f;

inline int batch_width_cost(float acc, float trials, float r, int K) {
  const double p = ((double)acc + 0.5) / ((double)trials + 1.0);
  double qk = 1.0, best = -1.0;
  int kb = 1;
  for (int k = 1; k <= K; ++k) {
    qk *= 1.0 - p;
    const double v = (1.0 - qk) / ((double)r + (double)k);
    if (v > best) {
      best = v;
      kb = k;
    }
  }
  return kb;
}
constexpr int kSmemRecordBytes = 160 * 1024;  // larger ranges keep their records in global memory
// Window of the trial loop: kWS candidate slots per CTA, each caching up to kCap entries of the
// candidate's segment (range-local sample, activation change, new hidden field), prepared ahead of
// the batches. Batches are at most kWinBatch wide.
constexpr int kWS = 96;
constexpr int kCap = 160;
constexpr int kWinBatch = 64;
// Per-batch accumulator buffer of the windowed loop: one packed word per candidate (arrival count
// in bits 56..63, count of out-of-range shares in 48..55, fixed-point sum below), padding. Three
// buffers rotate. One warp reads a batch's words, two per lane; the count fields cap the ranges at
// 255.
constexpr int kAccStride = 2 * kKmax + 32;
constexpr int kArrivalWord = 64;   // count-only word of a batch without a live candidate
constexpr int kWindowMaxRanges = 255;
static_assert(kWinBatch <= 64 && kWinBatch < kWS, "a windowed batch is read by one warp, two per lane");

// Device-resident run state (one per handle).
struct DevState {
  double S;                  // loss sum of the cached state
  unsigned long long trials, accepts, candidates, batches, wasted, forced, trace_written;
  unsigned long long alg_bytes;  // compulsory DRAM bytes of the evaluated candidates and commits
  unsigned long long phase_ns[8];  // CTA 0: set-up, evaluate, arrive, wait, reduce+decide, commit;
                                   // [6] wait averaged over all CTAs
  unsigned long long alg_flops;    // deep path: FLOPs of the evaluated candidates' chains
  float rate_acc, rate_trials;     // decayed counts of accepts and trials (batch-width choice)
  int err;                   // first device-side error (mca_status), 0 = none
  int pad;
};

// Arguments of the two-layer trial loop (input -> hidden -> output). The samples are split into NR
// contiguous ranges of RS samples (RS a multiple of 8); CTA r owns range r.
struct Mlp2Args {
  int N, D, H, C, Np;
  int NR, RS, SUB;           // ranges, samples per range, entries per sub-chunk (multiple of 32)
  int smem_records;          // 1: each CTA keeps its range's sample records in shared memory
  int window;                // 1: run the windowed trial loop (records and window in shared memory)
  unsigned long long P, P1;
  const int* xs_off;         // [D + 1] CSR of X by feature: entries of feature i in [off[i], off[i+1])
  const int* xs_n;           // [nnz] sample index of each entry (ascending inside a feature)
  const float* xs_v;         // [nnz] value x[n, i] != 0
  const int* xs_sect;        // [D] 32-byte sectors of a z1 row that feature i's entries touch
  const int* xs_roff;        // [D x (NR + 1)] first entry of feature i in range r
  float* z1;                 // [H x Np] hidden fields, feature-major
  float* srec;               // [kSR x Np] field-major: output fields, loss, label
  float* w1;                 // [H x D] effective weights
  float* w2;                 // [C x H]
  signed char* code1;        // ternary codes / mask bits (nullable for fp32 layers)
  signed char* code2;
  const float* wfix1;        // masked layers: fixed weights
  const float* wfix2;
  int wk1, wk2;
  float sc1, sc2;
  int act1, act2;
  float g1, g2;
  int loss;
  int op;
  float lo, hi, delta, bound;
  int strict;
  int metro;                 // 1: Metropolis rule (Eq. 7) with msc = N / beta; 0: greedy (Eq. 6)
  double msc;
  int stretch;               // > 0: current-layer schedule, trials per stretch; 0: uniform index
  unsigned long long seed, tau0, n_trials;
  int K;
  int fixed_K;
  float* partial;            // [2 x kKmax x NR] per-candidate, per-range loss changes
  unsigned long long* accum; // [3 x kAccStride] windowed loop: fixed-point sums, counts, arrivals
  GridBarrier* bar;
  DevState* st;
  mca_trace_rec* trace;
  int trace_cap;
  const unsigned long long* ftau;
  const unsigned char* facc;
  int nforce;
  int n_explicit;            // > 0: evaluate these candidates once, no decision, no commit
  const unsigned int* ex_idx;
  const float* ex_new;
  double* ex_out;
};

// ------------------------------------------------------------------------------------------------
// Deep MLP path (three or more weight layers): every layer's fields are cached; a candidate in layer
// l updates row j of layer l, then layer l+1 by one weight column (rank-1), then recomputes the layers
// from l+2 on as  Z'_m = Z_m + W_m (f(Z'_{m-1}) - f(Z_{m-1}))  over tiles of kDeepTS samples.
// ------------------------------------------------------------------------------------------------
constexpr int kMaxLayers = 32;
constexpr int kDeepTS = 64;        // samples per tile
constexpr int kTcTS = 128;         // samples per tile of the tensor-core chain (one MMA M)
constexpr int kDeepThreads = 256;
constexpr int kDeepMaxWidth = 256; // widths of the layers inside the dense chain
constexpr int kDeepKC = 16;        // weight-tile depth of the chain GEMM
constexpr int kDeepScrSlots = 16;  // candidates whose fields the tensor-core evaluation keeps
constexpr int kTfmScrSlots = 16;   // candidates whose residual streams the evaluation keeps

struct DeepCand {
  unsigned int idx;
  int layer, row, col;
  float oldw, neww, delta;
  int new_code, valid;
};

// Decision of the last batch, written by the decide kernel and read by the commit kernel and host.
struct DeepCtl {
  int kstar;                 // accepted candidate, -1 none, -2 non-finite loss change
  int consumed;              // trials consumed by the batch
  DeepCand acc;              // the accepted candidate
};

struct DeepArgs {
  int L, N, Np, D, C, ntiles;
  int n_in[kMaxLayers], n_out[kMaxLayers], act[kMaxLayers], wk[kMaxLayers];
  float g[kMaxLayers], sc[kMaxLayers];
  unsigned long long off[kMaxLayers + 1];
  float* w[kMaxLayers];
  signed char* code[kMaxLayers];
  const float* wfix[kMaxLayers];
  float* Z[kMaxLayers];      // [n_out[l] x Np] fields of layer l; Z[L-1] are the output fields
  float* whi[kMaxLayers];    // tensor-core chain: tf32(W_m) and tf32(W_m - tf32(W_m)) of the
                             //   256 x 256 layers 1 .. L-2 as stage images (null otherwise)
  int tc;                    // 1: dense chain on the tensor cores, tiles of kTcTS samples
  const float* XT;           // [D x Np]
  float* ell;                // [Np] per-sample loss
  const int* y;
  int loss;
  int op;
  float lo, hi, delta, bound;
  int strict;
  int metro;                 // 1: Metropolis rule (Eq. 7) with msc = N / beta; 0: greedy (Eq. 6)
  double msc;
  int stretch;               // > 0: current-layer schedule, trials per stretch; 0: uniform index
  unsigned long long seed, tau;
  int Kb;
  float* partial;            // [kKmax x ntiles]
  DevState* st;
  DeepCtl* ctl;
  mca_trace_rec* trace;
  int trace_cap;
  const unsigned long long* ftau;
  const unsigned char* facc;
  int nforce;
  int n_explicit;
  const unsigned int* ex_idx;
  const float* ex_new;
  double* ex_out;
  // tensor-core evaluation of candidate k < nscr with a dense chain (layer <= L-3): every field it
  // computes goes to scr[k * (L + 1) + m] (layer m: row j of the mutated layer, the full layers
  // after it; m = L: the per-sample losses), so that an accepted candidate's fields are adopted
  // by swapping pointers instead of recomputing them
  float* const* scr;
  int nscr;
};

cudaError_t launch_deep_eval(const DeepArgs& a, cudaStream_t s);    // grid (Kb, ntiles)
cudaError_t launch_deep_decide(const DeepArgs& a, cudaStream_t s);  // one CTA
cudaError_t launch_deep_commit(const DeepArgs& a, cudaStream_t s);  // grid ntiles
cudaError_t launch_deep_forward_layer(const DeepArgs& a, int l, cudaStream_t s);
cudaError_t launch_deep_losses(const DeepArgs& a, cudaStream_t s);
cudaError_t launch_deep_split(const DeepArgs& a, cudaStream_t s);     // W_hi / W_lo of all layers
cudaError_t launch_deep_eval_tc(const DeepArgs& a, cudaStream_t s);   // grid (Kb, ntiles)
cudaError_t launch_deep_commit_tc(const DeepArgs& a, cudaStream_t s); // grid ntiles

// ------------------------------------------------------------------------------------------------
// Character-level Transformer path: pre-LN GPT blocks over B sequences of T tokens. All parameters
// live in one flat fp32 array; a candidate recomputes each sequence from the first stage its
// parameter feeds (embeddings, block b, or the final LN and head), reading the parameters through
// a one-element patch (index midx reads mval), on the cached residual stream at that stage.
// ------------------------------------------------------------------------------------------------
constexpr int kTfmMaxBlocks = 8;
constexpr int kTfmThreads = 512;
constexpr int kTfmMaxT = 64;
constexpr int kTfmMaxD = 128;
constexpr int kTfmMaxV = 128;
constexpr int kTfmFC = 128;        // FFN hidden columns per chunk

enum TfmMode { kTfmEval = 0, kTfmCommit = 1, kTfmForward = 2 };

struct TfmArgs {
  int V, T, d, H, dh, F, nL, B;
  float eps;
  int act;
  float g;
  // flat offsets: embeddings, the first block, the block stride, the final LN and the head; and the
  // offsets inside a block
  unsigned long long o_tok, o_pos, o_blk0, blk_size, o_lnf_g, o_lnf_b, o_wh, o_bh, P;
  unsigned int r_ln1g, r_ln1b, r_wq, r_bq, r_wk, r_bk, r_wv, r_bv, r_wo, r_bo, r_ln2g, r_ln2b,
      r_w1, r_b1, r_w2, r_b2;
  float* params;             // [P]
  const int* tokens;         // [B x (T + 1)]
  float* X;                  // [(nL + 1) x B x T x d] residual stream entering block b (b = nL: final)
  float* Xmid;               // [nL x B x T x d] block b's stream after its attention sub-block (tc)
  float* ell;                // [B] per-sequence loss sums
  int loss_unused;
  int op;
  float lo, hi, delta, bound;
  int strict;
  int metro;                 // 1: Metropolis rule (Eq. 7) with msc = N / beta; 0: greedy (Eq. 6)
  double msc;
  int stretch;               // > 0: current-layer schedule, trials per stretch; 0: uniform index
  unsigned long long seed, tau;
  int Kb;
  int mode;
  size_t smem;               // dynamic shared memory of the sequence kernel
  float* partial;            // [kKmax x B]
  DevState* st;
  DeepCtl* ctl;
  mca_trace_rec* trace;
  int trace_cap;
  const unsigned long long* ftau;
  const unsigned char* facc;
  int nforce;
  int n_explicit;
  const unsigned int* ex_idx;
  const float* ex_new;
  double* ex_out;
  int tc;                    // 1: the tensor-core kernels (mca_tfm_tc.cu) run the sequences
  float* wimg;               // their split-weight images (mca_tc_layout.h), tc = 1 only
  // scratch slots (tc = 1, trial loop only): candidate k < nscr of a batch writes the residual
  // streams it recomputes to slot k of scrX ([nscr][(2 nL + 1) x B x T x d]: X, then Xmid) and its
  // sequence losses to scr_ell ([nscr][B]); an accepted candidate with a slot is adopted from it
  float* scrX;
  float* scr_ell;
  int nscr;
  // batches run ahead of the host (tc = 1, trial loop): the batch's first trial is read from
  // tau_dev, which the decision advances by the trials it consumed; trials at or past tau_end do not
  // exist (a batch that starts there does nothing). nullptr: the batch starts at tau.
  unsigned long long* tau_dev;
  unsigned long long tau_end;
};

size_t tfm_smem_bytes(int T, int d, int dh, int V);
cudaError_t launch_tfm_eval(const TfmArgs& a, cudaStream_t s);      // grid (Kb, B)
cudaError_t launch_tfm_decide(const TfmArgs& a, cudaStream_t s);    // one CTA
cudaError_t launch_tfm_commit(const TfmArgs& a, cudaStream_t s);    // grid B
cudaError_t launch_tfm_forward(const TfmArgs& a, cudaStream_t s);   // grid B, writes every stage
// Tensor-core Transformer kernels (two sequences per CTA): the split-weight images from the
// parameters, the three sequence modes, and the image entry of the accepted parameter after a commit.
cudaError_t launch_tfm_tc_split(const TfmArgs& a, cudaStream_t s);
cudaError_t launch_tfm_tc_eval(const TfmArgs& a, cudaStream_t s);      // grid (Kb, B / 2)
cudaError_t launch_tfm_tc_commit(const TfmArgs& a, cudaStream_t s);    // grid B / 2
cudaError_t launch_tfm_tc_forward(const TfmArgs& a, cudaStream_t s);   // grid B / 2
// After the commit kernel: the accepted weight's image entry and, with a scratch slot, adoption.
cudaError_t launch_tfm_tc_adopt(const TfmArgs& a, cudaStream_t s);     // grid (B, 2 nL + 1)

// Launchers (mca_mlp2.cu). All enqueue on `stream` and return the CUDA error of the launch.
cudaError_t launch_transpose_pad(const float* X, int N, int D, float* XT, int Np, cudaStream_t s);
cudaError_t launch_csr_count(const float* XT, int Np, int N, int D, int* cnt, cudaStream_t s);
cudaError_t launch_csr_fill(const float* XT, int Np, int N, int D, const int* off, int* xs_n,
                            float* xs_v, cudaStream_t s);
cudaError_t launch_csr_sectors(const int* off, const int* xs_n, int D, int* sect, cudaStream_t s);
cudaError_t launch_csr_range_offsets(const int* off, const int* xs_n, int D, int NR, int RS,
                                     int* roff, cudaStream_t s);
cudaError_t launch_count_nonfinite(const float* p, size_t n, int* out, cudaStream_t s);
cudaError_t launch_init_layer(int wkind, float scale, const float* src, const signed char* mask,
                              size_t n, float* w_eff, signed char* code, float* wfix,
                              cudaStream_t s);
cudaError_t launch_sgemm_nn(int M, int Ncol, int K, const float* A, int lda, const float* B,
                            int ldb, float* C, int ldc, cudaStream_t s);
cudaError_t launch_mlp2_outputs(const Mlp2Args& a, const int* y, cudaStream_t s);
// S = sum of ell[0 .. N) in fp64 (fixed order) into st->S.
cudaError_t launch_sum_loss(const float* ell, int N, DevState* st, cudaStream_t s);
// Cooperative persistent trial loop, one CTA per sample range (grid = NR).
cudaError_t launch_mlp2_loop(const Mlp2Args& a, cudaStream_t s);
size_t mlp2_window_smem_bytes(int RS);
int mlp2_loop_max_grid(const Mlp2Args& a, int num_sms);
size_t mlp2_loop_smem_bytes(const Mlp2Args& a);

// Proposals of trials tau0 .. tau0 + n - 1 as explicit candidates (mca_propose.cu): the trial's
// record (index, effective weights before and after, validity) and the candidate arrays of the
// explicit evaluation (a rejected proposal is evaluated as the no-op).
struct ProposeArgs {
  int L, n;
  unsigned long long off[kMaxLayers + 1];   // flat offset of each layer; off[L] = P
  int wk[kMaxLayers];
  float sc[kMaxLayers];
  const float* w[kMaxLayers];
  const signed char* code[kMaxLayers];
  const float* wfix[kMaxLayers];
  int op;
  float lo, hi, delta, bound;
  int stretch;
  unsigned long long seed, tau0;
  mca_trace_rec* rec;        // [n]
  unsigned int* ex_idx;      // [n]
  float* ex_new;             // [n]
};
cudaError_t launch_propose(const ProposeArgs& a, cudaStream_t s);

// Fields of a layer on the tensor cores (mca_gemm_tc.cu): Z[M x Np] = W[M x K] act(B)[K x Np]
// (act < 0: B as it is), 3xTF32. img: scratch of gemm_tc_image_bytes(M, K, Np) bytes, 256-byte
// aligned; err: device status word (MCA_ERR_TIMEOUT when a bounded wait ran out).
bool gemm_tc_ok(int M, int K, int Np);
size_t gemm_tc_image_bytes(int M, int K, int Np);
cudaError_t launch_gemm_tc(const float* W, int M, int K, const float* B, int act, float g,
                           float* Z, int Np, float* img, int* err, cudaStream_t s);

}  // namespace mca

struct mca_handle;

namespace mca {
// Kernel arguments of a handle's trial loop (its state and workspace scratch).
Mlp2Args handle_mlp2_args(mca_handle* h);

}  // namespace mca

struct mca_handle {
  std::string err;
  std::vector<mca_layer> layers;
  int loss = 0;
  mca_domain dom{};
  mca_options opt{};
  long long N = 0;
  int D = 0, C = 0, Np = 0;
  unsigned long long P = 0;
  std::vector<unsigned long long> off;   // flat offset of each layer
  cudaStream_t stream = nullptr;
  int device = 0, num_sms = 0;
  // memory
  void* ws = nullptr;
  size_t ws_bytes = 0;
  bool ws_owned = false;
  float* XT = nullptr;                   // [D x Np]
  int* y = nullptr;
  int* xs_off = nullptr;
  int* xs_n = nullptr;
  float* xs_v = nullptr;
  int* xs_sect = nullptr;
  int* xs_roff = nullptr;
  long long nnz = 0;
  int max_nnz = 0;
  std::vector<float*> w_eff;
  std::vector<signed char*> code;
  std::vector<float*> wfix;
  float* z1 = nullptr;
  float* srec = nullptr;
  // deep path
  bool deep = false;
  bool tc = false;                   // deep: dense chain on the tensor cores; Transformer: the
                                     // tensor-core sequence kernels
  std::vector<float*> Z;
  std::vector<float*> whi;           // split-weight images of layers 1 .. L-2 (tensor-core chain)
  float* ell = nullptr;
  mca::DeepCtl* ctl = nullptr;
  int ntiles = 0;
  float* partial = nullptr;
  unsigned long long* accum = nullptr;
  int NR = 0, RS = 0, SUB = 0, smem_records = 0, window = 0;
  mca::GridBarrier* bar = nullptr;
  mca::DevState* st = nullptr;
  mca_trace_rec* trace = nullptr;
  int trace_cap = 0;
  unsigned int* ex_idx = nullptr;
  float* ex_new = nullptr;
  double* ex_out = nullptr;
  mca_trace_rec* prop = nullptr;         // [kKmax] proposals of mca_eval_trials
  float* gimg = nullptr;                 // operand images of the tensor-core forward pass
  int nscr = 0;                          // tensor-core paths: candidate scratch slots
  std::vector<float*> scr;               // [nscr x (L + 1)] layer m of slot k (m = L: losses)
  float** scr_dev = nullptr;             // the same table in device memory
  cudaEvent_t ev_c[2] = {nullptr, nullptr};   // around the adoption / commit after a decision
  bool ev_c_pending = false;
  // test hook
  unsigned long long* ftau = nullptr;
  unsigned char* facc = nullptr;
  int nforce = 0;
  // host-side counters
  unsigned long long tau = 0;
  unsigned long long launches = 0, resyncs = 0;
  cudaEvent_t ev[3] = {nullptr, nullptr, nullptr};   // per-batch kernel timing (deep, Transformer)
  // Transformer tensor-core path, batches run ahead of the host: two decision buffers (device),
  // the batch's first trial (device), their pinned host mirror, and per-buffer events
  mca::DeepCtl* ctl2 = nullptr;
  unsigned long long* tau_dev = nullptr;
  struct PipeHost {
    mca::DeepCtl ctl[2];
    unsigned long long tau;
  }* pipe_host = nullptr;
  cudaEvent_t ev_p[2][3] = {{nullptr, nullptr, nullptr}, {nullptr, nullptr, nullptr}};
  unsigned long long eval_ns = 0, rest_ns = 0;
  bool broken = false;                   // a sticky CUDA error or device timeout was seen
  float rate_acc = 0.0f, rate_trials = 0.0f;   // deep path: acceptance counts (batch width)
  // transformer path
  bool tfm = false;
  mca_tfm_spec tspec{};
  float* params = nullptr;               // [P] flat parameters
  int* tokens = nullptr;                 // [B x (ctx + 1)]
  float* X = nullptr;                    // cached residual stream at every stage
  float* tfm_img = nullptr;
  float* tfm_Xmid = nullptr;             // its mid streams (after each block's attention)
  float* tfm_scrX = nullptr;             // Transformer tensor-core path: candidate scratch slots
  float* tfm_scr_ell = nullptr;          // (h->nscr of them)              // split-weight images of the tensor-core kernels (tc)
};
