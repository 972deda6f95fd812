/*
 * mca.h -- C ABI of the GB300 (sm_103a) Monte Carlo mutation-selection (MCA) trial loop.
 *
 * The method (paper "Beyond Backpropagation: Monte Carlo Method Can Train Deep Neural Networks"):
 * pick one parameter at random, give it a new random value (Section 2, Eq. 1), re-evaluate the
 * full-batch training loss (Eq. 2 with R = 0) and keep the change iff the loss does not rise
 * (greedy rule, Section 3.1 Eq. 6; or Eq. 7's Metropolis rule, mca_domain.temperature);
 * otherwise restore the old value and try again. The loss is re-evaluated from cached per-layer
 * local fields (Section 2.4): a mutation of weight (j, i) of
 * layer l changes only row j of that layer's fields (a rank-1 update over all samples) and, through
 * neuron j's activation change, the next layer's fields by one weight column. Also: the
 * current-layer proposal schedule (Section 2.1, mca_domain.layer_stretch) and multi-parameter
 * channel mutations (Section 2.3, mca_run_channels).
 *
 * Conventions shared by every call:
 *  - Every call returns an mca_status; no C++ exception crosses this boundary. A failed call
 *    leaves a message readable with mca_last_error().
 *  - Pointers documented "host or device" may point to either (the library asks the CUDA driver
 *    which); all others are host pointers.
 *  - All GPU work of a handle is queued on the stream given at creation (mca_options.stream; NULL
 *    = the legacy default stream). A handle is not thread-safe.
 *  - Flat parameter order: layers in forward order; inside a layer the weight matrix
 *    [n_out x n_in] row-major (weight (j, i) at offset j * n_in + i). There are no biases.
 *  - Sizes: N < 2^31 samples, total parameter count P < 2^32.
 */
#ifndef MCA_H
#define MCA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MCA_OK = 0,
  MCA_ERR_INVALID = 1,     /* bad argument, size or spec */
  MCA_ERR_CUDA = 2,        /* a CUDA call failed; the handle must be destroyed */
  MCA_ERR_OOM = 3,         /* device memory exhausted, or the caller's workspace is too small */
  MCA_ERR_TIMEOUT = 4,     /* a bounded device-side wait ran out; the handle must be destroyed */
  MCA_ERR_NUMERIC = 5,     /* NaN or Inf in the data, the parameters or the loss */
  MCA_ERR_UNSUPPORTED = 6  /* a valid spec this build does not implement */
} mca_status;

/* Transfer functions (Section 2: ReLU and the Gaussian exp(-gamma x^2); tanh, sigmoid and the
 * exact-erf GELU of the Transformer section). */
typedef enum {
  MCA_ACT_IDENTITY = 0,
  MCA_ACT_TANH = 1,
  MCA_ACT_SIGMOID = 2,
  MCA_ACT_RELU = 3,
  MCA_ACT_GAUSSIAN = 4,    /* exp(-act_param * x^2) */
  MCA_ACT_GELU = 5
} mca_act;

/* Per-sample loss on the last layer's activations a (Section 2; Eq. 2 with R = 0):
 *   MSE_ONEHOT:  sum_k (a_k - [k == y])^2
 *   SOFTMAX_CE:  log(sum_k exp(a_k)) - a_y   (natural log)
 * Decisions use the loss sum S over all samples; mca_loss() reports S / N. */
typedef enum { MCA_LOSS_MSE_ONEHOT = 0, MCA_LOSS_SOFTMAX_CE = 1 } mca_loss_kind;

/* Weight storage of a layer (Section 2: discrete weights and pruning; Section 3.4 Eq. 12).
 *   FP32:        the weight is an fp32 value; mutations draw a new value (mca_domain.op).
 *   TERNARY_I8:  an int8 code t in {-1, 0, +1}; the effective weight is scale * t. A mutation
 *                sets a uniformly drawn code (which may equal the old one: a no-op trial).
 *   MASKED_FP32: a fixed fp32 weight w and a mask bit m (initially 1); the effective weight is
 *                m ? w : 0. A mutation toggles m (pruning, and regrowth of a pruned weight). */
typedef enum { MCA_W_FP32 = 0, MCA_W_TERNARY_I8 = 1, MCA_W_MASKED_FP32 = 2 } mca_wkind;

/* Mutation operator of FP32 layers (Section 2, Eq. 1).
 *   REPLACE: w' = lo + (hi - lo) * u,  u = (r1 >> 8) * 2^-24 (two fp32 roundings; exact for
 *            [lo, hi) = [-1, 1)).
 *   PERTURB: w' = w + delta * (2u - 1) in fp32 (Eq. 1's w + delta * rand). */
typedef enum { MCA_OP_REPLACE = 0, MCA_OP_PERTURB = 1 } mca_op;

typedef struct {
  int32_t n_in, n_out;     /* fan-in and fan-out */
  int32_t act;             /* mca_act applied to this layer's fields */
  float act_param;         /* gamma of MCA_ACT_GAUSSIAN; ignored otherwise */
  int32_t wkind;           /* mca_wkind */
  float scale;             /* TERNARY_I8: effective weight = scale * code; ignored otherwise */
} mca_layer;

/* Weight domain and acceptance rule (Eq. 1; Eq. 6, or Eq. 7 with temperature > 0). */
typedef struct {
  int32_t op;              /* mca_op */
  float lo, hi;            /* REPLACE range [lo, hi) */
  float delta;             /* PERTURB amplitude */
  float bound;             /* > 0: a proposal with !(|w'| < bound) is rejected unevaluated */
  int32_t strict;          /* 0: accept iff dS <= theta; 1: accept iff dS < theta */
  float temperature;       /* 1 / beta of the Metropolis rule (Section 3.1, Eq. 7), finite, >= 0.
                              0: the greedy rule (Eq. 6), theta = 0. > 0: Eq. 7's acceptance
                              probability min{1, exp(-beta dS / N)} as a per-trial threshold
                              theta = -(N / beta) ln u on the loss-sum change, with the trial's
                              own uniform number u = (r3 + 1/2) 2^-32, r3 the fourth word of
                              Philox4x32-10(key = seed, counter = tau); N = samples (MLP) or
                              n_seq * ctx predicted tokens (Transformer). theta depends only on
                              the trial, so speculative batches keep the sequential chain */
  int32_t layer_stretch;   /* 0: each trial's parameter is uniform over all P parameters (Eq. 1).
                              M > 0 (MLPs; the current-layer schedule of Section 2.1): trials come
                              in stretches of M, stretch s = tau / M mutating only layer l_s,
                              l_s = floor(q * n_layers / 2^32) with q the first word of
                              Philox4x32-10(key = seed, counter = (s_lo, s_hi, 1, 0)); the index
                              is uniform inside that layer: first index of l_s +
                              floor(r0 * (size of l_s) / 2^32). The Transformer takes 0 only
                              (MCA_ERR_UNSUPPORTED otherwise) */
} mca_domain;

/* Training set. x: [n x d] fp32, sample-major (sample n's features at x + n * d); y: [n] int32
 * labels in [0, n_classes). Host or device; copied at creation, not retained. */
typedef struct {
  const float* x;
  const int32_t* y;
  int64_t n;
  int32_t d;
} mca_dataset;

typedef struct {
  int32_t K;               /* speculative candidates per batch, 1..128 (the trajectory does not
                              depend on K: the lowest-index improving candidate is accepted) */
  int32_t resync_period;   /* > 0: recompute every cached field from scratch each time tau
                              crosses a multiple of this; 0: only at creation and set_params */
  void* stream;            /* cudaStream_t; NULL = legacy default stream */
  int32_t trace_cap;       /* > 0: keep the last trace_cap trial records (mca_get_trace) */
  int32_t grid;            /* > 0: target number of sample ranges = CTAs of the trial-loop
                              kernel (capped at what is co-resident); 0: automatic. The ranges
                              fix the summation order of dS, so runs with different grids agree
                              only to rounding */
  void* workspace;         /* NULL: the library allocates its device memory itself; otherwise a
                              caller-owned device buffer of >= mca_workspace_size() bytes,
                              256-byte aligned, that must outlive the handle */
  size_t workspace_bytes;
  int32_t fixed_K;         /* 0: the batch width follows p, the recently observed acceptance rate
                              per trial, at most K (fewer discarded candidates while many are
                              accepted; the trajectory is the same): ceil(2 / p) candidates for
                              single-hidden-layer networks; for deep nets and Transformers the K
                              that maximises the expected trials consumed, (1 - (1-p)^K) / p, per
                              batch cost r + K (r about 2 candidate evaluations);
                              1: every batch evaluates K candidates */
} mca_options;

typedef struct {
  uint64_t trials;         /* trials consumed (sequential trials; discarded speculation excluded) */
  uint64_t accepts;
  uint64_t candidates;     /* candidates evaluated on the GPU */
  uint64_t batches;
  uint64_t wasted;         /* candidates evaluated after the accepted one in their batch */
  uint64_t forced;         /* decisions taken from mca_force_decisions */
  uint64_t resyncs;
  uint64_t launches;       /* kernels this handle launched */
  uint64_t tau;            /* next trial counter */
  double S;                /* current loss sum */
  uint64_t alg_bytes;      /* compulsory DRAM bytes of the distinct candidates evaluated (each
                              trial counted once, the first time it is evaluated) and commits:
                              per first-layer candidate 32 B per hidden-field sector its input
                              feature's non-zeros touch + 8 B per non-zero; per output-layer
                              candidate 4 B per sample (one hidden-field row); per accepted
                              first-layer candidate the sectors written back */
  uint64_t phase_ns[8];    /* two-layer nets, device time per phase of the trial loop. Windowed
                              loop (used when its shared-memory window fits), mean over CTAs, [0]
                              to [6] only in a build with MCA_PHASE_TIMERS=1: [0] batch set-up
                              together with the previous batch's commit (overlapped), [1]
                              evaluation, [2] the waiting warp's wait for every CTA's shares +
                              decision, [3] the whole CTA's wait (including bringing later slots up
                              to date), [4] adding the CTA's shares, [5] 0, [6] the consumer warps'
                              wait for slots still being prepared (summed over warps); [7] (a count,
                              always) slots prepared again after a commit invalidated them. Other
                              loop, first CTA:
                              [0] proposal + evaluation, [1] grid barrier, [2] reduction +
                              decision, [3] commit. Deep nets and the Transformer (CUDA
                              events around each batch's launches): [0] candidate evaluation
                              kernel, [1] decision + commit kernels. Rest 0 */
  uint64_t alg_flops;      /* deep nets: FLOPs of the evaluated candidates' recomputation (2 per
                              multiply-add: the row update, the rank-1 layer, the dense layers) */
  uint32_t tensor_cores;   /* 1: this handle's dense recomputation runs on the tcgen05 tensor-core
                              kernels (3xTF32): a deep net whose hidden layers are all 256 x 256,
                              or a Transformer with ctx 64, d_model 128, 4 heads, d_ff a multiple
                              of 128 up to 1024, vocab <= 128 and an even number of sequences
                              (unless the process sets MCA_TFM_TENSOR_CORES=0 before creating
                              the handle); 0: the SIMT fp32 kernels */
  uint32_t reserved;       /* 0 */
} mca_run_stats;

typedef struct {
  uint64_t tau;            /* trial counter */
  uint32_t idx;            /* flat parameter index */
  int32_t accept;          /* 1 accepted, 0 rejected */
  float old_w, new_w;      /* effective weights before / after the proposal */
  int32_t valid;           /* 0: outside the weight domain, rejected unevaluated */
  int32_t forced;          /* 1: decision taken from mca_force_decisions */
  double dS;               /* S' - S of the candidate (NaN when not evaluated) */
  double S;                /* loss sum before the trial */
} mca_trace_rec;

/* Character-level Transformer (Section 2.5): token + learned position embeddings, n_layer pre-LN
 * blocks (causal multi-head self-attention; feed-forward d_model -> d_ff -> d_model with act =
 * MCA_ACT_GELU or MCA_ACT_GAUSSIAN), a final LN and an untied head; loss = sum over positions of the
 * next-token softmax cross-entropy. Limits of this build: ctx <= 64, d_model <= 128,
 * d_model / n_head <= 64, vocab <= 128, n_layer <= 8.
 * Flat parameter order (matrices [out x in] row-major): tok_emb [vocab x d], pos_emb [ctx x d];
 * per block: ln1.g [d], ln1.b [d], wq [d x d], bq [d], wk, bk, wv, bv, wo, bo, ln2.g, ln2.b,
 * w1 [d_ff x d], b1 [d_ff], w2 [d x d_ff], b2 [d]; then lnf.g, lnf.b, w_head [vocab x d], b_head. */
typedef struct {
  int32_t vocab, ctx, d_model, n_layer, n_head, d_ff;
  int32_t act;
  float act_param;
  float ln_eps;
} mca_tfm_spec;

typedef struct mca_handle mca_handle;

/* Bytes of device workspace mca_create needs for this spec and dataset (counts the non-zeros of
 * the dataset, so data must be valid). Same argument rules as mca_create. */
mca_status mca_workspace_size(const mca_layer* layers, int32_t n_layers, int32_t loss,
                              const mca_dataset* data, const mca_options* opt, size_t* bytes);

/* Build a trial loop for the MLP `layers` (Section 2, Fig. 1a) on `data`.
 *  init_params: [P] fp32, host or device, flat order; FP32 and MASKED layers hold the weight,
 *               TERNARY layers hold the code (-1, 0 or 1) as a float.
 *  Requirements: n_layers >= 2, layers[0].n_in == data->d, layers[l].n_out == layers[l+1].n_in,
 *  the last layer's n_out <= 16 (the number of classes), labels in range.
 *  Computes every cached field with a full forward pass (the trial counter tau starts at 0).
 *  On success *out owns a handle to release with mca_destroy. Errors: INVALID (spec/sizes),
 *  NUMERIC (non-finite x or init, or a non-finite initial loss), OOM, CUDA, UNSUPPORTED.
 *  Deep nets whose inner layers are all 256 x 256 run their dense chain on the tensor cores; the
 *  evaluation of candidates k < min(K, 16) then keeps every field it computes in per-candidate
 *  scratch slots of the workspace, from which an accepted candidate is adopted (MCA_ADOPT=0 in the
 *  environment, read by this call and mca_workspace_size, leaves the slots out). */
mca_status mca_create(const mca_layer* layers, int32_t n_layers, int32_t loss,
                      const mca_domain* dom, const mca_dataset* data, const float* init_params,
                      const mca_options* opt, mca_handle** out);

/* Bytes of device workspace mca_create_transformer needs. */
mca_status mca_tfm_workspace_size(const mca_tfm_spec* spec, int64_t n_seq, const mca_options* opt,
                                  size_t* bytes);

/* Build a trial loop for the Transformer `spec` on n_seq fixed sequences. tokens: [n_seq x (ctx+1)]
 * int32, host or device (inputs tokens[:, :ctx], targets tokens[:, 1:]); init_params: [P] fp32,
 * host or device, in the flat order above. Every parameter is an fp32 weight (Eq. 1 replacement or
 * perturbation). mca_loss reports S / (n_seq * ctx). Errors as for mca_create.
 * Kernels: with ctx 64, d_model 128, 4 heads, d_ff a multiple of 128 up to 1024, vocab <= 128 and an
 * even n_seq the sequences run on the tensor-core kernels (3xTF32 tcgen05, two sequences per CTA);
 * for other shapes, or when the process environment has MCA_TFM_TENSOR_CORES=0, on the SIMT fp32
 * kernels. The variable is read by this call and by mca_tfm_workspace_size (the tensor-core kernels'
 * weight images are part of the workspace), so it must not change between the two. mca_run_stats
 * .tensor_cores reports the choice. On the tensor-core kernels a candidate's recomputation starts at
 * the first sub-block its parameter feeds (a block's input, its cached stream after the attention
 * sub-block for LN2, a rank-1 step for one hidden unit of the feed-forward network), the evaluation
 * of candidates k < min(K, 16) keeps what it recomputed in per-candidate scratch slots of the
 * workspace (at most 8 GiB) from which an accepted candidate is adopted, and mca_run enqueues each
 * batch before it reads the previous decision unless resync_period > 0. MCA_ADOPT=0 in the
 * environment (read like MCA_TFM_TENSOR_CORES; it applies to deep MLPs on the tensor cores too)
 * leaves out the slots: every accepted candidate is then recomputed by the commit kernels. */
mca_status mca_create_transformer(const mca_tfm_spec* spec, const mca_domain* dom,
                                  const int32_t* tokens, int64_t n_seq, const float* init_params,
                                  const mca_options* opt, mca_handle** out);

/* Run n_trials sequential trials tau, tau+1, ... (Eq. 1 proposals drawn from Philox4x32-10 with
 * key = seed and counter = tau; Eq. 6 selection). Returns when they are done. stats: nullable.
 * Errors: TIMEOUT (a device-side wait ran out), NUMERIC (the loss became non-finite), CUDA. */
mca_status mca_run(mca_handle* h, uint64_t n_trials, uint64_t seed, mca_run_stats* stats);

/* Current mean loss L = S / N (Eq. 2 with R = 0) from the cached fields. */
mca_status mca_loss(mca_handle* h, double* L);

/* Effective weights (fp32, flat order) into dst[0 .. n) (host or device); n must equal P. */
mca_status mca_get_params(mca_handle* h, float* dst, size_t n);

/* Per-parameter int8 codes into dst[0 .. n): ternary code, mask bit, or 0 for FP32 layers. */
mca_status mca_get_codes(mca_handle* h, int8_t* dst, size_t n);

/* Resume: load parameters in mca_create's init format (ternary codes; for MASKED layers the
 * mask is taken from `codes`, nullable = all ones), set the trial counter to tau and recompute
 * every cached field. Host or device pointers. */
mca_status mca_set_params(mca_handle* h, const float* params, const int8_t* codes, size_t n,
                          uint64_t tau);

/* Recompute every cached field and S from the parameters with a full forward pass. */
mca_status mca_resync(mca_handle* h);

/* Copy up to cap of the most recent trial records, oldest first, into dst (host); *n gets the
 * count. Requires trace_cap > 0 at creation. */
mca_status mca_get_trace(mca_handle* h, mca_trace_rec* dst, size_t cap, size_t* n);

/* Test hook: decide trial tau[m] by accept[m] instead of by its loss change (tau strictly
 * increasing, host arrays). Used to replay a reference trajectory through trials whose loss change
 * is within rounding of zero. n = 0 clears the list. */
mca_status mca_force_decisions(mca_handle* h, const uint64_t* tau, const uint8_t* accept,
                               size_t n);

/* Statistics accumulated over the handle's lifetime. */
mca_status mca_get_stats(mca_handle* h, mca_run_stats* stats);

/* Loss changes dS of n hypothetical single-weight changes, all against the current state, with
 * no commit: weight flat_idx[m] set to the effective value new_w[m] (host arrays, n <= 128).
 * Same kernels as mca_run's evaluation step. dS: [n] doubles (host). */
mca_status mca_eval_candidates(mca_handle* h, const uint32_t* flat_idx, const float* new_w,
                               size_t n, double* dS);

/* The proposals of trials tau .. tau+n-1 (n <= 128) as mca_run would draw them with Philox key
 * `seed` (Eq. 1: index rule, current-layer schedule, mutation of the layer's storage kind, domain
 * check), each evaluated against the current state with no commit (the kernels of
 * mca_eval_candidates). out[k] (host): tau, idx, old_w, new_w (effective weights), valid, dS (NaN
 * for a proposal outside the weight domain), S (the handle's current loss sum), accept = forced =
 * 0. The handle's trial counter and state do not change. This is one shard's step of a chain whose
 * samples are split over several handles (the loss is a sum over samples, Eq. 2): every shard
 * evaluates the same trials on its own samples, the shards' dS are added, one decision
 * (mca_decide_batch) is taken for all, and every shard commits it (mca_force_decisions for the
 * batch's consumed trials, then mca_run over them). */
mca_status mca_eval_trials(mca_handle* h, uint64_t seed, uint64_t tau, size_t n,
                           mca_trace_rec* out);

/* The decision of a batch of trials tau .. tau+n-1 with loss changes dS[k] (host arrays; valid[k]
 * = 0 skips trial k, as for a proposal outside the weight domain): *kstar = the lowest k with
 * dS[k] <= theta_{tau+k} (< when the domain is strict), theta = 0 under the greedy rule (Eq. 6)
 * and -(N / beta) ln u_{tau+k} under Eq. 7's Metropolis rule (mca_domain.temperature), evaluated
 * exactly as the kernels do (dS rounded to fp32); -1 if none. N = n_samples, the chain's whole
 * sample count (a sharded chain's sum over all shards), or the handle's own when n_samples = 0.
 * Host only, no device work. Errors: INVALID, NUMERIC (a non-finite dS of a valid trial before
 * the accepted one). */
mca_status mca_decide_batch(mca_handle* h, uint64_t seed, uint64_t tau, size_t n,
                            const uint8_t* valid, const double* dS, int64_t n_samples,
                            int32_t* kstar);

/* The same evaluation as mca_eval_candidates, for callers that cannot allocate device memory:
 * a caller whose device memory is entirely reserved by another allocator (a framework's caching
 * allocator, a fixed arena), or a latency-critical loop that cannot afford the device-wide
 * synchronisation a cudaMalloc or cudaFree may cause. The paper has no counterpart; this is an
 * interface convenience. Single-hidden-layer handles only: a deep or Transformer handle gives
 * MCA_ERR_UNSUPPORTED before any device work and stays usable. The handle's device must be the
 * current device (else MCA_ERR_INVALID, handle unchanged). flat_idx [n] (uint32), new_w [n]
 * (fp32) and dS [n] (fp64) are DEVICE arrays owned by the caller; the call copies flat_idx and
 * new_w back to the host (on the stack) to check them against P and for finiteness, and
 * synchronises the handle's stream twice (after that read and after the evaluation), so it
 * returns with the results in dS. The evaluation's scratch (one partial per candidate and sample
 * range, plus a grid barrier) lives in a fixed 128 KB + 256 B device array inside the library,
 * which every GPU that loads the library holds until the process exits; nothing is allocated per
 * call. Limits: n <= 128 candidates and a handle of at most 256 sample ranges, else
 * MCA_ERR_INVALID with a message. The first call on a device looks up the array's device address
 * (once per device), so make that first call before any stream capture. All calls share the
 * array: calls whose work overlaps on the GPU (two handles on different streams, or two threads)
 * race and must be serialised by the caller. */
mca_status mca_eval_candidates_noalloc(mca_handle* h, const uint32_t* flat_idx,
                                       const float* new_w, size_t n, double* dS);

/* Multi-parameter channel mutations (Section 2.3) on an MLP handle whose layers are all
 * MCA_W_FP32. Trial tau draws a channel -- one node of every layer, input c_0, hidden c_1 ..
 * c_{L-1}, output c_L, each uniform: c_m = floor(v_m * n_m / 2^32) -- and changes the L weights
 * W_m[c_{m+1}][c_m] at once: scheme MCA_CHANNEL_HE redraws weight m as a_m * (2u - 1) in fp32,
 * a_m = fp32(sqrt(6 / n_in of layer m)) (He's uniform amplitude), u = (v_{L+1+m} >> 8) * 2^-24;
 * MCA_CHANNEL_ZERO sets them to 0 (the Dropout-like scheme). The words v_0, v_1, ... are those of
 * Philox4x32-10(key = seed, counter = (tau_lo, tau_hi, 2, q)), q = 0, 1, ..., four per counter.
 * Every layer changes, so each trial recomputes every cached field with the full forward pass
 * (the kernels of creation and mca_resync), then keeps the channel iff dS <= theta (Eq. 6, or Eq.
 * 7 with the domain's temperature; forced decisions apply); a rejected channel is restored and
 * the fields recomputed again. Trials run one at a time (no speculation) from the handle's trial
 * counter tau, which advances by n_trials; mca_run_stats and the trace count single-weight trials
 * only. accepted [n_trials] (uint8, 1 kept) and dS [n_trials] (S' - S) are nullable HOST arrays.
 * Errors: INVALID (NULL handle, unknown scheme), UNSUPPORTED (a Transformer handle or a ternary /
 * masked layer), NUMERIC (a non-finite loss change), CUDA. */
typedef enum { MCA_CHANNEL_HE = 0, MCA_CHANNEL_ZERO = 1 } mca_channel_scheme;
mca_status mca_run_channels(mca_handle* h, uint64_t n_trials, uint64_t seed, int32_t scheme,
                            uint8_t* accepted, double* dS);

/* Failure-detection self-test (the library's own check; the paper has no counterpart). Runs the
 * bounded grid barrier of the trial loop in one CTA that waits for a second CTA which is never
 * launched: a peer that never arrives. The wait must give up after its 2 s limit, record
 * MCA_ERR_TIMEOUT and let the kernel return, leaving the CUDA context usable. *status receives the
 * status the kernel recorded (MCA_ERR_TIMEOUT when the limit works); *waited_ms (nullable) the
 * host wall time of the kernel. Runs on the legacy default stream and allocates 256 bytes of
 * device memory for its barrier. Returns MCA_OK when the kernel ran and returned, MCA_ERR_CUDA
 * otherwise. */
mca_status mca_selftest_wait_timeout(int32_t* status, double* waited_ms);

void mca_destroy(mca_handle* h);

/* Message of the last failed call on h (h may be NULL: then the last failed mca_create or
 * mca_workspace_size of this thread). Never NULL. */
const char* mca_last_error(mca_handle* h);

#ifdef __cplusplus
}
#endif

#endif /* MCA_H */
