// C ABI of the MCA trial loop (include/mca.h): argument checks, device memory layout, the
// creation-time full forward pass, and the host side of mca_run.
#include <algorithm>
#include <chrono>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <string>
#include <thread>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "mca_device.cuh"
#include "mca_internal.h"
#include "mca_tc_layout.h"

using mca::DevState;
using mca::GridBarrier;

namespace {

// NVTX range for profilers (nsys, ncu --nvtx): creation, each mca_run call, each host-driven batch
// of the deep and Transformer paths, each persistent trial-loop segment, each resync. Without an
// attached tool a push / pop is a check of one function pointer.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

thread_local std::string g_create_err;

mca_status fail(mca_handle* h, mca_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  if (h)
    h->err = buf;
  else
    g_create_err = buf;
  return st;
}

void mark_broken(mca_handle* h, cudaError_t e) {
  // An allocation failure leaves the context usable; any other CUDA error may be sticky.
  if (h && e != cudaErrorMemoryAllocation) h->broken = true;
}

#define CUDA_TRY(h, expr)                                                                    \
  do {                                                                                       \
    cudaError_t e_ = (expr);                                                                 \
    if (e_ != cudaSuccess) {                                                                 \
      mark_broken((h), e_);                                                                  \
      return fail((h), e_ == cudaErrorMemoryAllocation ? MCA_ERR_OOM : MCA_ERR_CUDA,         \
                  "%s: %s (%s:%d)", #expr, cudaGetErrorString(e_), __FILE__, __LINE__);      \
    }                                                                                        \
  } while (0)

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

bool is_device_ptr(const void* p) {
  if (!p) return false;
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

struct Layout {
  size_t XT, y, xs_off, xs_n, xs_v, xs_sect, xs_roff, z1, srec, partial, accum, bar, st, trace,
      ex_idx, ex_new, ex_out, prop, scratch, ell, ctl, gimg, scr_tab, total;
  std::vector<size_t> w_eff, code, wfix, Z, whi, scr;
};

bool is_deep(const std::vector<mca_layer>& layers) { return layers.size() > 2; }
int deep_tiles(long long N) { return (int)((N + mca::kDeepTS - 1) / mca::kDeepTS); }

// The dense chain runs on the tensor cores when every layer between the first and the output layer
// is 256 x 256 (the kernel's fixed width).
bool deep_tc_ok(const std::vector<mca_layer>& layers) {
  if (layers.size() < 3) return false;
  for (size_t l = 1; l + 1 < layers.size(); ++l)
    if (layers[l].n_in != 256 || layers[l].n_out != 256) return false;
  return true;
}
int deep_tc_tiles(long long N) { return (int)((N + mca::kTcTS - 1) / mca::kTcTS); }

// Accepted candidates are adopted from scratch slots written by their evaluation (deep and
// Transformer tensor-core paths) unless the process sets MCA_ADOPT=0: then the commit kernels
// recompute them. Read by the workspace-size calls and creation, so it must not change between them.
bool adopt_enabled() {
  const char* e = std::getenv("MCA_ADOPT");
  return !(e && std::strcmp(e, "0") == 0);
}

// Candidate scratch slots of the deep tensor-core path (min(K, kDeepScrSlots)); none elsewhere.
int deep_scratch_slots(const std::vector<mca_layer>& layers, int K) {
  return deep_tc_ok(layers) && adopt_enabled() ? std::min(K, mca::kDeepScrSlots) : 0;
}

int pad_n(long long N) { return (int)((N + 127) / 128 * 128); }

// The forward pass (creation, resync) computes the fields of a layer on the tensor cores
// (mca_gemm_tc.cu) when its shape allows, unless the process sets MCA_FORWARD_TENSOR_CORES=0 (then
// with the SIMT SGEMM). Read by mca_workspace_size and mca_create (the operand images are part of
// the workspace), so it must not change between the two.
bool forward_tc_enabled() {
  const char* e = std::getenv("MCA_FORWARD_TENSOR_CORES");
  return !(e && std::strcmp(e, "0") == 0);
}

// Layers whose fields the forward pass computes with a GEMM: the first layer of a two-layer net
// (its output fields have their own kernel), every layer of a deep net.
bool forward_tc_layer(const std::vector<mca_layer>& layers, size_t l, int Np) {
  if (!forward_tc_enabled()) return false;
  if (!is_deep(layers) && l != 0) return false;
  return mca::gemm_tc_ok(layers[l].n_out, layers[l].n_in, Np);
}

size_t forward_tc_image_bytes(const std::vector<mca_layer>& layers, int Np) {
  size_t b = 0;
  for (size_t l = 0; l < layers.size(); ++l)
    if (forward_tc_layer(layers, l, Np))
      b = std::max(b, mca::gemm_tc_image_bytes(layers[l].n_out, layers[l].n_in, Np));
  return b;
}

// Device memory of a handle. Single hidden layer: feature CSR of X, z1, sample records, per-range
// partials. Deep: the fields of every layer, per-sample losses, per-tile partials.
Layout plan(const std::vector<mca_layer>& layers, long long N, int D, long long nnz, int trace_cap,
            int NR, int nscr) {
  const bool deep = is_deep(layers);
  Layout L;
  size_t o = 0;
  auto take = [&](size_t bytes) {
    size_t at = o;
    o = align256(o + bytes);
    return at;
  };
  const int Np = pad_n(N);
  const int H = layers[0].n_out;
  L.XT = take(sizeof(float) * (size_t)D * Np);
  L.y = take(sizeof(int) * (size_t)N);
  if (deep) nnz = 0;
  L.xs_off = take(sizeof(int) * (size_t)(D + 1));
  L.xs_n = take(sizeof(int) * (size_t)std::max<long long>(nnz, 1));
  L.xs_v = take(sizeof(float) * (size_t)std::max<long long>(nnz, 1));
  L.xs_sect = take(sizeof(int) * (size_t)D);
  L.xs_roff = take(sizeof(int) * (size_t)D * (NR + 1));
  for (const auto& ly : layers) {
    const size_t n = (size_t)ly.n_in * ly.n_out;
    L.w_eff.push_back(take(sizeof(float) * n));
    L.code.push_back(ly.wkind != MCA_W_FP32 ? take(n) : SIZE_MAX);
    L.wfix.push_back(ly.wkind == MCA_W_MASKED_FP32 ? take(sizeof(float) * n) : SIZE_MAX);
  }
  if (deep) {
    for (const auto& ly : layers) L.Z.push_back(take(sizeof(float) * (size_t)ly.n_out * Np));
    if (deep_tc_ok(layers)) {
      for (size_t l = 1; l + 1 < layers.size(); ++l)
        L.whi.push_back(take(sizeof(float) * 2 * 256 * 256));   // hi and lo stage images
    }
    L.ell = take(sizeof(float) * (size_t)Np);
    L.ctl = take(sizeof(mca::DeepCtl));
    L.z1 = L.srec = SIZE_MAX;
    L.partial = take(sizeof(float) * (size_t)mca::kKmax * deep_tiles(N));
  } else {
    L.ell = L.ctl = SIZE_MAX;
    L.z1 = take(sizeof(float) * (size_t)H * Np);
    L.srec = take(sizeof(float) * (size_t)mca::kSR * Np);
    L.partial = take(sizeof(float) * 2 * (size_t)mca::kKmax * NR);
  }
  L.accum = take(sizeof(unsigned long long) * 3 * mca::kAccStride);
  L.bar = take(sizeof(GridBarrier));
  L.st = take(sizeof(DevState));
  L.trace = take(sizeof(mca_trace_rec) * (size_t)std::max(trace_cap, 0));
  L.ex_idx = take(sizeof(unsigned int) * mca::kKmax);
  L.ex_new = take(sizeof(float) * mca::kKmax);
  L.ex_out = take(sizeof(double) * mca::kKmax);
  L.prop = take(sizeof(mca_trace_rec) * mca::kKmax);
  L.scratch = take(sizeof(int) * (size_t)(D + 8));
  const size_t gb = forward_tc_image_bytes(layers, Np);
  L.gimg = gb ? take(gb) : SIZE_MAX;
  L.scr_tab = SIZE_MAX;
  if (deep && nscr > 0) {
    L.scr_tab = take(sizeof(float*) * (size_t)nscr * (layers.size() + 1));
    for (int k = 0; k < nscr; ++k) {
      for (const auto& ly : layers) L.scr.push_back(take(sizeof(float) * (size_t)ly.n_out * Np));
      L.scr.push_back(take(sizeof(float) * (size_t)Np));
    }
  }
  L.total = o;
  return L;
}

mca_status check_spec(const mca_layer* layers, int n_layers, int loss, const mca_dataset* data,
                      std::vector<mca_layer>* out) {
  if (!layers || n_layers < 2) return fail(nullptr, MCA_ERR_INVALID, "need n_layers >= 2");
  if (!data || !data->x || !data->y || data->n <= 0 || data->d <= 0)
    return fail(nullptr, MCA_ERR_INVALID, "empty or missing dataset");
  if (data->n >= (1ll << 31) - 1024) return fail(nullptr, MCA_ERR_INVALID, "N too large");
  if (loss != MCA_LOSS_MSE_ONEHOT && loss != MCA_LOSS_SOFTMAX_CE)
    return fail(nullptr, MCA_ERR_INVALID, "unknown loss %d", loss);
  unsigned long long P = 0;
  for (int l = 0; l < n_layers; ++l) {
    const mca_layer& L = layers[l];
    if (L.n_in <= 0 || L.n_out <= 0) return fail(nullptr, MCA_ERR_INVALID, "layer %d: bad size", l);
    if (l == 0 && L.n_in != data->d)
      return fail(nullptr, MCA_ERR_INVALID, "layer 0 n_in %d != data d %d", L.n_in, data->d);
    if (l > 0 && L.n_in != layers[l - 1].n_out)
      return fail(nullptr, MCA_ERR_INVALID, "layer %d n_in != layer %d n_out", l, l - 1);
    if (L.act < MCA_ACT_IDENTITY || L.act > MCA_ACT_GELU)
      return fail(nullptr, MCA_ERR_INVALID, "layer %d: unknown act %d", l, L.act);
    if (L.wkind < MCA_W_FP32 || L.wkind > MCA_W_MASKED_FP32)
      return fail(nullptr, MCA_ERR_INVALID, "layer %d: unknown wkind %d", l, L.wkind);
    if (!std::isfinite(L.act_param) || !std::isfinite(L.scale))
      return fail(nullptr, MCA_ERR_INVALID, "layer %d: non-finite parameter", l);
    P += (unsigned long long)L.n_in * (unsigned long long)L.n_out;
  }
  if (P >= (1ull << 32)) return fail(nullptr, MCA_ERR_INVALID, "P = %llu >= 2^32", P);
  const int C = layers[n_layers - 1].n_out;
  if (C > mca::kMaxClasses)
    return fail(nullptr, MCA_ERR_UNSUPPORTED, "%d outputs > %d", C, mca::kMaxClasses);
  if (n_layers > mca::kMaxLayers)
    return fail(nullptr, MCA_ERR_UNSUPPORTED, "%d layers > %d", n_layers, mca::kMaxLayers);
  if (n_layers > 2)
    for (int l = 0; l + 1 < n_layers; ++l)
      if (layers[l].n_out > mca::kDeepMaxWidth)
        return fail(nullptr, MCA_ERR_UNSUPPORTED, "deep nets: hidden width %d > %d",
                    layers[l].n_out, mca::kDeepMaxWidth);
  out->assign(layers, layers + n_layers);
  return MCA_OK;
}

mca_options default_options() {
  mca_options o;
  std::memset(&o, 0, sizeof(o));
  o.K = 32;
  return o;
}

mca_domain default_domain() {
  mca_domain d;
  std::memset(&d, 0, sizeof(d));
  d.op = MCA_OP_REPLACE;
  d.lo = -1.0f;
  d.hi = 1.0f;
  d.delta = 0.01f;
  return d;
}

// Non-zeros of a host array, counted by up to 16 threads (the counts add up in any order).
long long host_nnz(const float* x, size_t n) {
  auto count = [x](size_t b, size_t e) {
    long long c = 0;
    for (size_t i = b; i < e; ++i) c += x[i] != 0.0f;
    return c;
  };
  const unsigned hw = std::thread::hardware_concurrency();
  const unsigned nt = n < (size_t)(1u << 22) ? 1u : std::max(1u, std::min(16u, hw));
  if (nt == 1) return count(0, n);
  const size_t per = (n + nt - 1) / nt;
  std::vector<long long> part(nt, 0);
  std::vector<std::thread> th;
  th.reserve(nt);
  for (unsigned t = 0; t < nt; ++t)
    th.emplace_back([&, t] { part[t] = count(std::min(n, t * per), std::min(n, (t + 1) * per)); });
  for (auto& q : th) q.join();
  long long c = 0;
  for (long long v : part) c += v;
  return c;
}

// One CTA waits in the trial loop's grid barrier for a second CTA that is never launched
// (mca_selftest_wait_timeout): the bounded wait must give up and record MCA_ERR_TIMEOUT in *err.
__global__ void wait_selftest_kernel(GridBarrier* bar, int* err) {
  __shared__ int s_flag;
  unsigned int gen = 0u;
  mca::grid_sync(bar, 2u, gen, err, &s_flag);
}

__global__ void count_nonzero_kernel(const float* __restrict__ p, size_t n,
                                     unsigned long long* out) {
  unsigned int c = 0;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x)
    c += p[i] != 0.0f;
  c = __reduce_add_sync(0xffffffffu, c);
  if ((threadIdx.x & 31) == 0) atomicAdd(out, (unsigned long long)c);
}

mca_status count_nnz(const mca_dataset* d, cudaStream_t s, long long* nnz) {
  const size_t n = (size_t)d->n * (size_t)d->d;
  if (!is_device_ptr(d->x)) {
    *nnz = host_nnz(d->x, n);
    return MCA_OK;
  }
  unsigned long long* dc = nullptr;
  CUDA_TRY(nullptr, cudaMalloc(&dc, sizeof(unsigned long long)));
  unsigned long long hc = 0;
  cudaError_t e = cudaMemsetAsync(dc, 0, sizeof(unsigned long long), s);
  if (e == cudaSuccess) {
    const int grid = (int)std::min<size_t>(4096, (n + 255) / 256);
    count_nonzero_kernel<<<grid, 256, 0, s>>>(d->x, n, dc);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaMemcpyAsync(&hc, dc, sizeof(hc), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  cudaFree(dc);
  CUDA_TRY(nullptr, e);
  *nnz = (long long)hc;
  return MCA_OK;
}

// Sample ranges of the trial loop: one CTA per range, all CTAs co-resident. Ranges hold a multiple
// of 8 samples (whole 32-byte sectors of a hidden-field row) and at least about kRangeTarget.
struct Ranges {
  int NR, RS, SUB, smem_records, window;
};

mca_status choose_ranges(const std::vector<mca_layer>& layers, int loss, long long N, int grid_opt,
                         Ranges* out) {
  int dev = 0, sms = 0;
  CUDA_TRY(nullptr, cudaGetDevice(&dev));
  CUDA_TRY(nullptr, cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  mca::Mlp2Args probe;
  std::memset(&probe, 0, sizeof(probe));
  probe.act1 = layers[0].act;
  probe.act2 = layers[1].act;
  probe.loss = loss;
  for (int smem_records = 1; smem_records >= 0; --smem_records) {
    probe.smem_records = 0;
    const int maxgrid0 = mca::mlp2_loop_max_grid(probe, sms);
    if (maxgrid0 <= 0) return fail(nullptr, MCA_ERR_CUDA, "trial-loop kernel cannot be resident");
    long long target = grid_opt > 0 ? grid_opt : (N + mca::kRangeTarget - 1) / mca::kRangeTarget;
    target = std::max<long long>(1, std::min<long long>(target, maxgrid0));
    int RS = (int)((N + target - 1) / target);
    RS = (RS + 7) / 8 * 8;
    const int NR = (int)((N + RS - 1) / RS);
    int SUB = (RS + mca::kMaxSubs - 1) / mca::kMaxSubs;
    SUB = std::max(128, (SUB + 31) / 32 * 32);
    Ranges R{NR, RS, SUB, 0, 0};
    if (smem_records && (size_t)RS * mca::kSR * sizeof(float) <= (size_t)mca::kSmemRecordBytes) {
      probe.smem_records = 1;
      probe.RS = RS;
      if (mca::mlp2_loop_max_grid(probe, sms) < NR) continue;
      R.smem_records = 1;
      // the windowed loop when its records and candidate window fit next to the static state
      if (NR <= mca::kWindowMaxRanges &&
          mca::mlp2_window_smem_bytes(RS) + 24 * 1024 <= 227 * 1024) {
        probe.window = 1;
        if (mca::mlp2_loop_max_grid(probe, sms) >= NR) R.window = 1;
        probe.window = 0;
      }
    } else if (smem_records) {
      continue;
    }
    *out = R;
    return MCA_OK;
  }
  return fail(nullptr, MCA_ERR_CUDA, "no co-resident launch shape for the trial loop");
}

mca::Mlp2Args mlp2_args(mca_handle* h) {
  mca::Mlp2Args a;
  std::memset(&a, 0, sizeof(a));
  const mca_layer& L1 = h->layers[0];
  const mca_layer& L2 = h->layers[1];
  a.N = (int)h->N;
  a.D = h->D;
  a.H = L1.n_out;
  a.C = h->C;
  a.Np = h->Np;
  a.NR = h->NR;
  a.RS = h->RS;
  a.SUB = h->SUB;
  a.smem_records = h->smem_records;
  a.window = h->window;
  a.P = h->P;
  a.P1 = (unsigned long long)L1.n_in * L1.n_out;
  a.xs_off = h->xs_off;
  a.xs_n = h->xs_n;
  a.xs_v = h->xs_v;
  a.xs_sect = h->xs_sect;
  a.xs_roff = h->xs_roff;
  a.z1 = h->z1;
  a.srec = h->srec;
  a.w1 = h->w_eff[0];
  a.w2 = h->w_eff[1];
  a.code1 = h->code[0];
  a.code2 = h->code[1];
  a.wfix1 = h->wfix[0];
  a.wfix2 = h->wfix[1];
  a.wk1 = L1.wkind;
  a.wk2 = L2.wkind;
  a.sc1 = L1.scale;
  a.sc2 = L2.scale;
  a.act1 = L1.act;
  a.act2 = L2.act;
  a.g1 = L1.act_param;
  a.g2 = L2.act_param;
  a.loss = h->loss;
  a.op = h->dom.op;
  a.lo = h->dom.lo;
  a.hi = h->dom.hi;
  a.delta = h->dom.delta;
  a.bound = h->dom.bound;
  a.strict = h->dom.strict;
  a.metro = h->dom.temperature > 0.0f ? 1 : 0;
  a.msc = (double)h->N * (double)h->dom.temperature;
  a.stretch = h->dom.layer_stretch;
  a.K = h->opt.K;
  a.fixed_K = h->opt.fixed_K;
  a.partial = h->partial;
  a.accum = h->accum;
  a.bar = h->bar;
  a.st = h->st;
  a.trace = h->trace;
  a.trace_cap = h->trace_cap;
  a.ftau = h->ftau;
  a.facc = h->facc;
  a.nforce = h->nforce;
  return a;
}

mca::DeepArgs deep_args(mca_handle* h) {
  mca::DeepArgs a;
  std::memset(&a, 0, sizeof(a));
  a.L = (int)h->layers.size();
  a.N = (int)h->N;
  a.Np = h->Np;
  a.D = h->D;
  a.C = h->C;
  a.ntiles = h->ntiles;
  for (int l = 0; l < a.L; ++l) {
    const mca_layer& L = h->layers[l];
    a.n_in[l] = L.n_in;
    a.n_out[l] = L.n_out;
    a.act[l] = L.act;
    a.g[l] = L.act_param;
    a.wk[l] = L.wkind;
    a.sc[l] = L.scale;
    a.off[l] = h->off[l];
    a.w[l] = h->w_eff[l];
    a.code[l] = h->code[l];
    a.wfix[l] = h->wfix[l];
    a.Z[l] = h->Z[l];
    a.whi[l] = h->tc && l >= 1 && l + 1 < a.L ? h->whi[l - 1] : nullptr;
  }
  a.tc = h->tc ? 1 : 0;
  a.off[a.L] = h->P;
  a.XT = h->XT;
  a.ell = h->ell;
  a.y = h->y;
  a.loss = h->loss;
  a.op = h->dom.op;
  a.lo = h->dom.lo;
  a.hi = h->dom.hi;
  a.delta = h->dom.delta;
  a.bound = h->dom.bound;
  a.strict = h->dom.strict;
  a.metro = h->dom.temperature > 0.0f ? 1 : 0;
  a.msc = (double)h->N * (double)h->dom.temperature;
  a.stretch = h->dom.layer_stretch;
  a.partial = h->partial;
  a.st = h->st;
  a.ctl = h->ctl;
  a.trace = h->trace;
  a.trace_cap = h->trace_cap;
  a.ftau = h->ftau;
  a.facc = h->facc;
  a.nforce = h->nforce;
  return a;
}

// Full forward pass: every cached field, every sample's loss, and S (Section 2.4's cache).
mca::TfmArgs tfm_args(mca_handle* h);

mca_status resync(mca_handle* h) {
  NvtxRange nv("mca resync");
  if (h->tfm) {
    const mca::TfmArgs a = tfm_args(h);
    if (a.tc) {
      CUDA_TRY(h, mca::launch_tfm_tc_split(a, h->stream));
      h->launches += 1;
    }
    CUDA_TRY(h, mca::launch_tfm_forward(a, h->stream));
    CUDA_TRY(h, mca::launch_sum_loss(h->ell, a.B, h->st, h->stream));
    h->launches += 2;
    return MCA_OK;
  }
  if (h->deep) {
    const mca::DeepArgs a = deep_args(h);
    if (a.tc) {
      CUDA_TRY(h, mca::launch_deep_split(a, h->stream));
      h->launches += 1;
    }
    for (int l = 0; l < a.L; ++l) {
      if (h->gimg && forward_tc_layer(h->layers, (size_t)l, h->Np)) {
        CUDA_TRY(h, mca::launch_gemm_tc(a.w[l], a.n_out[l], a.n_in[l], l == 0 ? a.XT : a.Z[l - 1],
                                        l == 0 ? -1 : a.act[l - 1], l == 0 ? 0.0f : a.g[l - 1],
                                        a.Z[l], h->Np, h->gimg, &h->st->err, h->stream));
        h->launches += 2;                      // its two operand-image kernels
      } else {
        CUDA_TRY(h, mca::launch_deep_forward_layer(a, l, h->stream));
      }
    }
    CUDA_TRY(h, mca::launch_deep_losses(a, h->stream));
    CUDA_TRY(h, mca::launch_sum_loss(h->ell, (int)h->N, h->st, h->stream));
    h->launches += a.L + 2;
    return MCA_OK;
  }
  mca::Mlp2Args a = mlp2_args(h);
  if (h->gimg && forward_tc_layer(h->layers, 0, h->Np)) {
    CUDA_TRY(h, mca::launch_gemm_tc(h->w_eff[0], a.H, h->D, h->XT, -1, 0.0f, h->z1, h->Np, h->gimg,
                                    &h->st->err, h->stream));
    h->launches += 2;                          // the two operand-image kernels
  } else {
    CUDA_TRY(h, mca::launch_sgemm_nn(a.H, h->Np, h->D, h->w_eff[0], h->D, h->XT, h->Np, h->z1,
                                     h->Np, h->stream));
  }
  CUDA_TRY(h, mca::launch_mlp2_outputs(a, h->y, h->stream));
  CUDA_TRY(h, mca::launch_sum_loss(h->srec + (size_t)mca::kRecLoss * h->Np, (int)h->N, h->st,
                                    h->stream));
  h->launches += 3;
  return MCA_OK;
}

// Load parameters in the init format into the per-layer weight arrays.
mca_status load_params(mca_handle* h, const float* params, const signed char* codes) {
  const bool pdev = is_device_ptr(params);
  const bool cdev = codes && is_device_ptr(codes);
  float* tmp = nullptr;
  signed char* ctmp = nullptr;
  const size_t P = h->P;
  if (!pdev) {
    CUDA_TRY(h, cudaMalloc(&tmp, sizeof(float) * P));
    CUDA_TRY(h, cudaMemcpyAsync(tmp, params, sizeof(float) * P, cudaMemcpyHostToDevice, h->stream));
  }
  if (codes && !cdev) {
    CUDA_TRY(h, cudaMalloc(&ctmp, P));
    CUDA_TRY(h, cudaMemcpyAsync(ctmp, codes, P, cudaMemcpyHostToDevice, h->stream));
  }
  const float* src = pdev ? params : tmp;
  const signed char* csrc = codes ? (cdev ? codes : ctmp) : nullptr;
  mca_status rc = MCA_OK;
  int* dflag = nullptr;
  cudaError_t e = cudaMalloc(&dflag, sizeof(int));
  if (e == cudaSuccess) e = cudaMemsetAsync(dflag, 0, sizeof(int), h->stream);
  if (e == cudaSuccess) e = mca::launch_count_nonfinite(src, P, dflag, h->stream);
  for (size_t l = 0; e == cudaSuccess && l < h->layers.size(); ++l) {
    const mca_layer& L = h->layers[l];
    const size_t n = (size_t)L.n_in * L.n_out;
    e = mca::launch_init_layer(L.wkind, L.scale, src + h->off[l], csrc ? csrc + h->off[l] : nullptr,
                               n, h->w_eff[l], h->code[l], h->wfix[l], h->stream);
    h->launches++;
  }
  int hflag = 0;
  if (e == cudaSuccess) e = cudaMemcpyAsync(&hflag, dflag, sizeof(int), cudaMemcpyDeviceToHost,
                                            h->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
  cudaFree(dflag);
  if (tmp) cudaFree(tmp);
  if (ctmp) cudaFree(ctmp);
  CUDA_TRY(h, e);
  if (hflag) rc = fail(h, MCA_ERR_NUMERIC, "non-finite parameter value");
  return rc;
}

mca_status read_state(mca_handle* h, DevState* out) {
  CUDA_TRY(h, cudaMemcpyAsync(out, h->st, sizeof(DevState), cudaMemcpyDeviceToHost, h->stream));
  CUDA_TRY(h, cudaStreamSynchronize(h->stream));
  return MCA_OK;
}

void fill_stats(mca_handle* h, const DevState& d, mca_run_stats* s) {
  s->trials = d.trials;
  s->accepts = d.accepts;
  s->candidates = d.candidates;
  s->batches = d.batches;
  s->wasted = d.wasted;
  s->forced = d.forced;
  s->resyncs = h->resyncs;
  s->launches = h->launches;
  s->tau = h->tau;
  s->S = d.S;
  s->alg_bytes = d.alg_bytes;
  for (int q = 0; q < 8; ++q) s->phase_ns[q] = d.phase_ns[q];
  if (h->deep || h->tfm) {           // host-timed kernels of the per-batch loop (CUDA events)
    s->phase_ns[0] = h->eval_ns;
    s->phase_ns[1] = h->rest_ns;
  }
  s->alg_flops = d.alg_flops;
  s->tensor_cores = h->tc ? 1u : 0u;
  s->reserved = 0u;
}

// ---------------------------------------------------------------- Transformer handles

struct TfmLayout {
  unsigned long long o_tok, o_pos, o_blk0, blk, o_lnf_g, o_lnf_b, o_wh, o_bh, P;
  unsigned int r[16];        // ln1g ln1b wq bq wk bk wv bv wo bo ln2g ln2b w1 b1 w2 b2
};

TfmLayout tfm_offsets(const mca_tfm_spec& t) {
  TfmLayout L;
  const unsigned long long d = t.d_model, f = t.d_ff, v = t.vocab, c = t.ctx;
  L.o_tok = 0;
  L.o_pos = v * d;
  L.o_blk0 = L.o_pos + c * d;
  const unsigned long long sizes[16] = {d, d, d * d, d, d * d, d, d * d, d, d * d, d, d, d,
                                        f * d, f, d * f, d};
  unsigned long long o = 0;
  for (int q = 0; q < 16; ++q) {
    L.r[q] = (unsigned int)o;
    o += sizes[q];
  }
  L.blk = o;
  L.o_lnf_g = L.o_blk0 + (unsigned long long)t.n_layer * L.blk;
  L.o_lnf_b = L.o_lnf_g + d;
  L.o_wh = L.o_lnf_b + d;
  L.o_bh = L.o_wh + v * d;
  L.P = L.o_bh + v;
  return L;
}

mca_status tfm_check(const mca_tfm_spec* t, int64_t n_seq) {
  if (!t) return fail(nullptr, MCA_ERR_INVALID, "spec is NULL");
  if (n_seq <= 0 || n_seq > 65535) return fail(nullptr, MCA_ERR_INVALID, "n_seq outside 1..65535");
  if (t->vocab < 2 || t->ctx < 1 || t->d_model < 1 || t->n_layer < 1 || t->n_head < 1 ||
      t->d_ff < 1)
    return fail(nullptr, MCA_ERR_INVALID, "bad transformer sizes");
  if (t->d_model % t->n_head != 0) return fail(nullptr, MCA_ERR_INVALID, "d_model % n_head != 0");
  if (t->act != MCA_ACT_GELU && t->act != MCA_ACT_GAUSSIAN)
    return fail(nullptr, MCA_ERR_INVALID, "feed-forward act must be GELU or Gaussian");
  if (!std::isfinite(t->act_param) || !(t->ln_eps > 0.0f))
    return fail(nullptr, MCA_ERR_INVALID, "bad act_param or ln_eps");
  if (t->ctx > mca::kTfmMaxT || t->d_model > mca::kTfmMaxD || t->vocab > mca::kTfmMaxV ||
      t->d_model / t->n_head > 64 || t->n_layer > mca::kTfmMaxBlocks)
    return fail(nullptr, MCA_ERR_UNSUPPORTED, "transformer larger than this build supports");
  if (mca::tfm_smem_bytes(t->ctx, t->d_model, t->d_model / t->n_head, t->vocab) > 227 * 1024)
    return fail(nullptr, MCA_ERR_UNSUPPORTED, "transformer tile exceeds shared memory");
  if (tfm_offsets(*t).P >= (1ull << 32)) return fail(nullptr, MCA_ERR_INVALID, "P >= 2^32");
  return MCA_OK;
}

struct TfmMem {
  size_t params, tokens, X, ell, partial, st, ctl, trace, ex_idx, ex_new, ex_out, prop, scratch,
      wimg, Xmid, scrX, scr_ell, ctl2, tau_dev, total;
  int nscr;
};

// The tensor-core Transformer kernels (mca_tfm_tc.cu) run a handle's sequences when the shape is
// one they handle, unless the process sets MCA_TFM_TENSOR_CORES=0 (then, and for every other shape,
// the SIMT kernels do). Read once per mca_create_transformer / mca_tfm_workspace_size call.
bool tfm_use_tc(const mca_tfm_spec& t, long long B) {
  const char* e = std::getenv("MCA_TFM_TENSOR_CORES");
  if (e && std::strcmp(e, "0") == 0) return false;
  return mca::tfm_tc_shape_ok(t.ctx, t.d_model, t.n_head, t.d_ff, t.vocab, B);
}

// Scratch slots of the tensor-core Transformer kernels: candidate k < nscr of a batch writes its
// residual streams (X and the mid streams) and sequence losses to slot k, min(K, kTfmScrSlots)
// slots within 8 GiB.
int tfm_scratch_slots(const mca_tfm_spec& t, long long B, int K, bool tc) {
  if (!tc || !adopt_enabled()) return 0;
  const size_t slot = sizeof(float) * ((size_t)(2 * t.n_layer + 1) * B * t.ctx * t.d_model + B);
  const size_t cap = (size_t)8 << 30;
  return (int)std::min<size_t>((size_t)std::min(K, mca::kTfmScrSlots), cap / slot);
}

TfmMem tfm_plan(const mca_tfm_spec& t, long long B, int trace_cap, bool tc, int K) {
  TfmMem M;
  size_t o = 0;
  auto take = [&](size_t bytes) {
    size_t at = o;
    o = align256(o + bytes);
    return at;
  };
  const TfmLayout L = tfm_offsets(t);
  M.params = take(sizeof(float) * L.P);
  M.tokens = take(sizeof(int) * (size_t)B * (t.ctx + 1));
  M.X = take(sizeof(float) * (size_t)(t.n_layer + 1) * B * t.ctx * t.d_model);
  M.ell = take(sizeof(float) * (size_t)B);
  M.partial = take(sizeof(float) * (size_t)mca::kKmax * B);
  M.st = take(sizeof(DevState));
  M.ctl = take(sizeof(mca::DeepCtl));
  M.trace = take(sizeof(mca_trace_rec) * (size_t)std::max(trace_cap, 0));
  M.ex_idx = take(sizeof(unsigned int) * mca::kKmax);
  M.ex_new = take(sizeof(float) * mca::kKmax);
  M.ex_out = take(sizeof(double) * mca::kKmax);
  M.prop = take(sizeof(mca_trace_rec) * mca::kKmax);
  M.scratch = take(sizeof(int) * 8);
  M.wimg = tc ? take(sizeof(float) * mca::tfm_tc_image_floats(t.d_ff, t.n_layer)) : 0;
  M.Xmid = take(tc ? sizeof(float) * (size_t)t.n_layer * B * t.ctx * t.d_model : 0);
  M.nscr = tfm_scratch_slots(t, B, K, tc);
  M.scrX = take(sizeof(float) * (size_t)M.nscr * (2 * t.n_layer + 1) * B * t.ctx * t.d_model);
  M.scr_ell = take(sizeof(float) * (size_t)M.nscr * B);
  M.ctl2 = take(2 * sizeof(mca::DeepCtl));
  M.tau_dev = take(sizeof(unsigned long long));
  M.total = o;
  return M;
}

mca::TfmArgs tfm_args(mca_handle* h) {
  mca::TfmArgs a;
  std::memset(&a, 0, sizeof(a));
  const mca_tfm_spec& t = h->tspec;
  const TfmLayout L = tfm_offsets(t);
  a.V = t.vocab;
  a.T = t.ctx;
  a.d = t.d_model;
  a.H = t.n_head;
  a.dh = t.d_model / t.n_head;
  a.F = t.d_ff;
  a.nL = t.n_layer;
  a.B = (int)(h->N / t.ctx);
  a.eps = t.ln_eps;
  a.act = t.act;
  a.g = t.act_param;
  a.o_tok = L.o_tok;
  a.o_pos = L.o_pos;
  a.o_blk0 = L.o_blk0;
  a.blk_size = L.blk;
  a.o_lnf_g = L.o_lnf_g;
  a.o_lnf_b = L.o_lnf_b;
  a.o_wh = L.o_wh;
  a.o_bh = L.o_bh;
  a.P = L.P;
  unsigned int* r[16] = {&a.r_ln1g, &a.r_ln1b, &a.r_wq, &a.r_bq, &a.r_wk, &a.r_bk, &a.r_wv,
                         &a.r_bv, &a.r_wo, &a.r_bo, &a.r_ln2g, &a.r_ln2b, &a.r_w1, &a.r_b1,
                         &a.r_w2, &a.r_b2};
  for (int q = 0; q < 16; ++q) *r[q] = L.r[q];
  a.params = h->params;
  a.tokens = h->tokens;
  a.X = h->X;
  a.Xmid = h->tfm_Xmid;
  a.ell = h->ell;
  a.op = h->dom.op;
  a.lo = h->dom.lo;
  a.hi = h->dom.hi;
  a.delta = h->dom.delta;
  a.bound = h->dom.bound;
  a.strict = h->dom.strict;
  a.metro = h->dom.temperature > 0.0f ? 1 : 0;
  a.msc = (double)h->N * (double)h->dom.temperature;
  a.stretch = h->dom.layer_stretch;
  a.smem = mca::tfm_smem_bytes(a.T, a.d, a.dh, a.V);
  a.partial = h->partial;
  a.st = h->st;
  a.ctl = h->ctl;
  a.trace = h->trace;
  a.trace_cap = h->trace_cap;
  a.ftau = h->ftau;
  a.facc = h->facc;
  a.nforce = h->nforce;
  a.tc = h->tc ? 1 : 0;
  a.wimg = h->tfm_img;
  return a;
}

// Transformer tensor-core batches with the host one batch ahead of the decisions: the kernels of
// batch i + 1 are enqueued before the host reads batch i's decision. The batch's first trial lives
// on the device (the decision advances it by the trials it consumed), so the GPU does not wait for
// the host between batches; a batch enqueued past the end of the run does nothing. A batch's width
// comes from the acceptance counts up to the batch before the previous one. Every batch has one of
// two decision buffers, read by the host from pinned memory.
mca_status run_tfm_pipelined(mca_handle* h, mca::TfmArgs ta, uint64_t n_trials) {
  if (!h->pipe_host) {
    CUDA_TRY(h, cudaMallocHost(reinterpret_cast<void**>(&h->pipe_host), sizeof(*h->pipe_host)));
    for (auto& b : h->ev_p)
      for (auto& e : b) CUDA_TRY(h, cudaEventCreate(&e));
  }
  auto* ph = h->pipe_host;
  ph->tau = h->tau;
  CUDA_TRY(h, cudaMemcpyAsync(h->tau_dev, &ph->tau, sizeof(ph->tau), cudaMemcpyHostToDevice,
                              h->stream));
  ta.tau_dev = h->tau_dev;
  ta.tau_end = h->tau + n_trials;
  ta.nscr = h->nscr;
  ta.scrX = h->tfm_scrX;
  ta.scr_ell = h->tfm_scr_ell;
  auto launch = [&](int i) -> mca_status {
    const int p = i & 1;
    const int Kw = h->opt.fixed_K ? h->opt.K
                                  : mca::batch_width_cost(h->rate_acc, h->rate_trials,
                                                          mca::kBatchCostTfm, h->opt.K);
    ta.Kb = (int)std::min<uint64_t>(n_trials, (uint64_t)Kw);
    ta.ctl = h->ctl2 + p;
    CUDA_TRY(h, cudaEventRecord(h->ev_p[p][0], h->stream));
    CUDA_TRY(h, mca::launch_tfm_eval(ta, h->stream));
    CUDA_TRY(h, cudaEventRecord(h->ev_p[p][1], h->stream));
    CUDA_TRY(h, mca::launch_tfm_decide(ta, h->stream));
    CUDA_TRY(h, mca::launch_tfm_commit(ta, h->stream));
    CUDA_TRY(h, mca::launch_tfm_tc_adopt(ta, h->stream));
    CUDA_TRY(h, cudaMemcpyAsync(&ph->ctl[p], h->ctl2 + p, sizeof(mca::DeepCtl),
                                cudaMemcpyDeviceToHost, h->stream));
    CUDA_TRY(h, cudaEventRecord(h->ev_p[p][2], h->stream));
    h->launches += 4;
    return MCA_OK;
  };
  uint64_t done = 0;
  mca_status rc = launch(0);
  if (rc != MCA_OK) return rc;
  for (int i = 0;; ++i) {
    NvtxRange nv_batch("mca batch (transformer, one ahead)");
    rc = launch(i + 1);
    if (rc != MCA_OK) return rc;
    const int p = i & 1;
    CUDA_TRY(h, cudaEventSynchronize(h->ev_p[p][2]));
    float ms_eval = 0.0f, ms_rest = 0.0f;
    CUDA_TRY(h, cudaEventElapsedTime(&ms_eval, h->ev_p[p][0], h->ev_p[p][1]));
    CUDA_TRY(h, cudaEventElapsedTime(&ms_rest, h->ev_p[p][1], h->ev_p[p][2]));
    h->eval_ns += (uint64_t)(ms_eval * 1e6f);
    h->rest_ns += (uint64_t)(ms_rest * 1e6f);
    const mca::DeepCtl ctl = ph->ctl[p];
    if (ctl.kstar == -2 || ctl.consumed <= 0) {
      cudaStreamSynchronize(h->stream);
      h->broken = true;
      return fail(h, MCA_ERR_NUMERIC, "non-finite loss change");
    }
    done += (uint64_t)ctl.consumed;
    h->rate_acc = h->rate_acc * mca::kRateDecay + (ctl.kstar >= 0 ? 1.0f : 0.0f);
    h->rate_trials = h->rate_trials * mca::kRateDecay + (float)ctl.consumed;
    if (done >= n_trials) break;
  }
  // the batch enqueued last starts at the run's end and does nothing; let it finish
  CUDA_TRY(h, cudaStreamSynchronize(h->stream));
  h->tau += done;
  return MCA_OK;
}

}  // namespace

namespace mca {
Mlp2Args handle_mlp2_args(mca_handle* h) { return mlp2_args(h); }
}  // namespace mca

extern "C" {

const char* mca_last_error(mca_handle* h) {
  return h ? h->err.c_str() : g_create_err.c_str();
}

mca_status mca_workspace_size(const mca_layer* layers, int32_t n_layers, int32_t loss,
                              const mca_dataset* data, const mca_options* opt, size_t* bytes) {
  std::vector<mca_layer> ls;
  mca_status rc = check_spec(layers, n_layers, loss, data, &ls);
  if (rc != MCA_OK) return rc;
  if (!bytes) return fail(nullptr, MCA_ERR_INVALID, "bytes is NULL");
  const mca_options o = opt ? *opt : default_options();
  if (is_deep(ls)) {
    *bytes = plan(ls, data->n, data->d, 0, o.trace_cap, 0, deep_scratch_slots(ls, o.K)).total;
    return MCA_OK;
  }
  long long nnz = 0;
  rc = count_nnz(data, (cudaStream_t)o.stream, &nnz);
  if (rc != MCA_OK) return rc;
  Ranges R;
  rc = choose_ranges(ls, loss, data->n, o.grid, &R);
  if (rc != MCA_OK) return rc;
  *bytes = plan(ls, data->n, data->d, nnz, o.trace_cap, R.NR, deep_scratch_slots(ls, o.K)).total;
  return MCA_OK;
}

mca_status mca_create(const mca_layer* layers, int32_t n_layers, int32_t loss,
                      const mca_domain* dom, const mca_dataset* data, const float* init_params,
                      const mca_options* opt, mca_handle** out) {
  NvtxRange nv("mca_create");
  if (!out) return fail(nullptr, MCA_ERR_INVALID, "out is NULL");
  *out = nullptr;
  std::vector<mca_layer> ls;
  mca_status rc = check_spec(layers, n_layers, loss, data, &ls);
  if (rc != MCA_OK) return rc;
  if (!init_params) return fail(nullptr, MCA_ERR_INVALID, "init_params is NULL");
  const mca_options o = opt ? *opt : default_options();
  if (o.K < 1 || o.K > mca::kKmax)
    return fail(nullptr, MCA_ERR_INVALID, "K = %d outside 1..%d", o.K, mca::kKmax);
  if (o.resync_period < 0 || o.trace_cap < 0 || o.grid < 0)
    return fail(nullptr, MCA_ERR_INVALID, "negative option");
  const mca_domain d = dom ? *dom : default_domain();
  if (d.op != MCA_OP_REPLACE && d.op != MCA_OP_PERTURB)
    return fail(nullptr, MCA_ERR_INVALID, "unknown op %d", d.op);
  if (!std::isfinite(d.lo) || !std::isfinite(d.hi) || !std::isfinite(d.delta) || !(d.hi > d.lo))
    return fail(nullptr, MCA_ERR_INVALID, "bad domain");
  if (!std::isfinite(d.temperature) || d.temperature < 0.0f)
    return fail(nullptr, MCA_ERR_INVALID, "temperature %g: must be finite and >= 0", d.temperature);
  if (d.layer_stretch < 0)
    return fail(nullptr, MCA_ERR_INVALID, "layer_stretch = %d < 0", d.layer_stretch);

  mca_handle* h = new (std::nothrow) mca_handle();
  if (!h) return fail(nullptr, MCA_ERR_OOM, "host allocation failed");
  h->layers = ls;
  h->loss = loss;
  h->dom = d;
  h->opt = o;
  h->N = data->n;
  h->D = data->d;
  h->C = ls.back().n_out;
  h->Np = pad_n(h->N);
  h->stream = (cudaStream_t)o.stream;
  unsigned long long P = 0;
  for (const auto& L : ls) {
    h->off.push_back(P);
    P += (unsigned long long)L.n_in * L.n_out;
  }
  h->P = P;
  h->trace_cap = o.trace_cap;

  auto bail = [&](mca_status st) {
    g_create_err = h->err;
    mca_destroy(h);
    return st;
  };
#define TRY(expr)                                   \
  do {                                              \
    mca_status s_ = (expr);                         \
    if (s_ != MCA_OK) return bail(s_);              \
  } while (0)
#define CTRY(expr)                                                                             \
  do {                                                                                         \
    cudaError_t e_ = (expr);                                                                   \
    if (e_ != cudaSuccess)                                                                     \
      return bail(fail(h, e_ == cudaErrorMemoryAllocation ? MCA_ERR_OOM : MCA_ERR_CUDA,        \
                       "%s: %s", #expr, cudaGetErrorString(e_)));                              \
  } while (0)

  CTRY(cudaGetDevice(&h->device));
  CTRY(cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device));
  h->deep = is_deep(ls);
  h->tc = h->deep && deep_tc_ok(ls);
  h->ntiles = h->tc ? deep_tc_tiles(h->N) : deep_tiles(h->N);
  if (!h->deep) {
    long long nnz = 0;
    mca_status s = count_nnz(data, h->stream, &nnz);
    if (s != MCA_OK) {
      h->err = g_create_err;
      return bail(s);
    }
    h->nnz = nnz;
  }
  if (!h->deep) {
    Ranges R;
    mca_status s = choose_ranges(ls, loss, h->N, o.grid, &R);
    if (s != MCA_OK) {
      h->err = g_create_err;
      return bail(s);
    }
    h->NR = R.NR;
    h->RS = R.RS;
    h->SUB = R.SUB;
    h->smem_records = R.smem_records;
    h->window = R.window;
  }
  h->nscr = h->deep ? deep_scratch_slots(ls, o.K) : 0;
  const Layout L = plan(ls, h->N, h->D, h->nnz, o.trace_cap, h->NR, h->nscr);
  if (o.workspace) {
    if (o.workspace_bytes < L.total)
      return bail(fail(h, MCA_ERR_OOM, "workspace of %zu bytes < %zu needed", o.workspace_bytes,
                       L.total));
    if (reinterpret_cast<uintptr_t>(o.workspace) % 256 != 0)
      return bail(fail(h, MCA_ERR_INVALID, "workspace not 256-byte aligned"));
    h->ws = o.workspace;
    h->ws_bytes = o.workspace_bytes;
  } else {
    CTRY(cudaMalloc(&h->ws, L.total));
    h->ws_owned = true;
    h->ws_bytes = L.total;
  }
  char* base = static_cast<char*>(h->ws);
  h->XT = reinterpret_cast<float*>(base + L.XT);
  h->y = reinterpret_cast<int*>(base + L.y);
  h->xs_off = reinterpret_cast<int*>(base + L.xs_off);
  h->xs_n = reinterpret_cast<int*>(base + L.xs_n);
  h->xs_v = reinterpret_cast<float*>(base + L.xs_v);
  h->xs_sect = reinterpret_cast<int*>(base + L.xs_sect);
  h->xs_roff = reinterpret_cast<int*>(base + L.xs_roff);
  for (size_t l = 0; l < ls.size(); ++l) {
    h->w_eff.push_back(reinterpret_cast<float*>(base + L.w_eff[l]));
    h->code.push_back(L.code[l] == SIZE_MAX ? nullptr
                                            : reinterpret_cast<signed char*>(base + L.code[l]));
    h->wfix.push_back(L.wfix[l] == SIZE_MAX ? nullptr : reinterpret_cast<float*>(base + L.wfix[l]));
  }
  if (h->deep) {
    for (size_t l = 0; l < ls.size(); ++l) h->Z.push_back(reinterpret_cast<float*>(base + L.Z[l]));
    for (size_t q = 0; q < L.whi.size(); ++q)
      h->whi.push_back(reinterpret_cast<float*>(base + L.whi[q]));
    h->ell = reinterpret_cast<float*>(base + L.ell);
    h->ctl = reinterpret_cast<mca::DeepCtl*>(base + L.ctl);
    CTRY(cudaMemsetAsync(h->ctl, 0, sizeof(mca::DeepCtl), h->stream));
    if (h->nscr > 0) {
      for (size_t q = 0; q < L.scr.size(); ++q)
        h->scr.push_back(reinterpret_cast<float*>(base + L.scr[q]));
      h->scr_dev = reinterpret_cast<float**>(base + L.scr_tab);
      CTRY(cudaMemcpyAsync(h->scr_dev, h->scr.data(), sizeof(float*) * h->scr.size(),
                           cudaMemcpyHostToDevice, h->stream));
    }
  } else {
    h->z1 = reinterpret_cast<float*>(base + L.z1);
    h->srec = reinterpret_cast<float*>(base + L.srec);
  }
  h->partial = reinterpret_cast<float*>(base + L.partial);
  h->accum = reinterpret_cast<unsigned long long*>(base + L.accum);
  h->bar = reinterpret_cast<GridBarrier*>(base + L.bar);
  h->st = reinterpret_cast<DevState*>(base + L.st);
  h->trace = o.trace_cap > 0 ? reinterpret_cast<mca_trace_rec*>(base + L.trace) : nullptr;
  h->ex_idx = reinterpret_cast<unsigned int*>(base + L.ex_idx);
  h->ex_new = reinterpret_cast<float*>(base + L.ex_new);
  h->ex_out = reinterpret_cast<double*>(base + L.ex_out);
  h->prop = reinterpret_cast<mca_trace_rec*>(base + L.prop);
  h->gimg = L.gimg != SIZE_MAX ? reinterpret_cast<float*>(base + L.gimg) : nullptr;
  int* scratch = reinterpret_cast<int*>(base + L.scratch);
  CTRY(cudaMemsetAsync(h->st, 0, sizeof(DevState), h->stream));
  CTRY(cudaMemsetAsync(h->bar, 0, sizeof(GridBarrier), h->stream));
  CTRY(cudaMemsetAsync(h->partial, 0, L.st - L.partial, h->stream));

  // dataset: X -> XT (feature-major, zero-padded), CSR by feature, labels
  const size_t nx = (size_t)h->N * h->D;
  const float* Xd = data->x;
  float* Xtmp = nullptr;
  if (!is_device_ptr(data->x)) {
    CTRY(cudaMalloc(&Xtmp, sizeof(float) * nx));
    CTRY(cudaMemcpyAsync(Xtmp, data->x, sizeof(float) * nx, cudaMemcpyHostToDevice, h->stream));
    Xd = Xtmp;
  }
  CTRY(cudaMemsetAsync(scratch, 0, sizeof(int), h->stream));
  CTRY(mca::launch_count_nonfinite(Xd, nx, scratch, h->stream));
  CTRY(mca::launch_transpose_pad(Xd, (int)h->N, h->D, h->XT, h->Np, h->stream));
  if (!h->deep) {
    CTRY(mca::launch_csr_count(h->XT, h->Np, (int)h->N, h->D, scratch + 8, h->stream));
    h->launches++;
  }
  h->launches += 2;
  std::vector<int> cnt(h->D + 8);
  CTRY(cudaMemcpyAsync(cnt.data(), scratch, sizeof(int) * (h->D + 8), cudaMemcpyDeviceToHost,
                       h->stream));
  CTRY(cudaStreamSynchronize(h->stream));
  if (Xtmp) cudaFree(Xtmp);
  if (cnt[0]) return bail(fail(h, MCA_ERR_NUMERIC, "non-finite value in x"));
  if (!h->deep) {
  std::vector<int> offs(h->D + 1, 0);
  long long acc = 0;
  for (int i = 0; i < h->D; ++i) {
    offs[i] = (int)acc;
    acc += cnt[8 + i];
    h->max_nnz = std::max(h->max_nnz, cnt[8 + i]);
  }
  offs[h->D] = (int)acc;
  if (acc != h->nnz) return bail(fail(h, MCA_ERR_INVALID, "nnz mismatch %lld vs %lld", acc, h->nnz));
  CTRY(cudaMemcpyAsync(h->xs_off, offs.data(), sizeof(int) * (h->D + 1), cudaMemcpyHostToDevice,
                       h->stream));
  CTRY(mca::launch_csr_fill(h->XT, h->Np, (int)h->N, h->D, h->xs_off, h->xs_n, h->xs_v, h->stream));
  CTRY(mca::launch_csr_sectors(h->xs_off, h->xs_n, h->D, h->xs_sect, h->stream));
  CTRY(mca::launch_csr_range_offsets(h->xs_off, h->xs_n, h->D, h->NR, h->RS, h->xs_roff,
                                     h->stream));
  h->launches += 3;
  }
  {
    std::vector<int> yh(h->N);
    CTRY(cudaMemcpyAsync(yh.data(), data->y, sizeof(int) * h->N, cudaMemcpyDefault, h->stream));
    CTRY(cudaStreamSynchronize(h->stream));
    for (long long n = 0; n < h->N; ++n)
      if (yh[n] < 0 || yh[n] >= h->C)
        return bail(fail(h, MCA_ERR_INVALID, "label %d of sample %lld outside [0, %d)", yh[n], n,
                         h->C));
    CTRY(cudaMemcpyAsync(h->y, yh.data(), sizeof(int) * h->N, cudaMemcpyHostToDevice, h->stream));
    CTRY(cudaStreamSynchronize(h->stream));
  }
  TRY(load_params(h, init_params, nullptr));
  TRY(resync(h));
  DevState ds;
  TRY(read_state(h, &ds));
  if (ds.err == MCA_ERR_TIMEOUT)
    return bail(fail(h, MCA_ERR_TIMEOUT, "device-side wait timed out in the forward pass"));
  if (!std::isfinite(ds.S)) return bail(fail(h, MCA_ERR_NUMERIC, "initial loss is not finite"));
#undef TRY
#undef CTRY
  *out = h;
  return MCA_OK;
}

mca_status mca_run(mca_handle* h, uint64_t n_trials, uint64_t seed, mca_run_stats* stats) {
  if (!h) return fail(nullptr, MCA_ERR_INVALID, "NULL handle");
  NvtxRange nv_run("mca_run");
  if (h->broken) return fail(h, MCA_ERR_CUDA, "handle unusable after an earlier device error");
  uint64_t remaining = n_trials;
  if (h->deep || h->tfm) {
    // one batch per round trip: evaluate, decide, commit, then read how many trials it consumed
    mca::DeepArgs a = h->deep ? deep_args(h) : mca::DeepArgs{};
    mca::TfmArgs ta = h->tfm ? tfm_args(h) : mca::TfmArgs{};
    a.seed = seed;
    ta.seed = seed;
    const uint64_t R = (uint64_t)h->opt.resync_period;
    if (h->tfm && h->tc && R == 0 && remaining > 0) {
      mca_status rc = run_tfm_pipelined(h, ta, remaining);
      if (rc != MCA_OK) return rc;
      remaining = 0;
    }
    while (remaining > 0) {
      NvtxRange nv_batch(h->tfm ? "mca batch (transformer)" : "mca batch (deep)");
      const int Kw = h->opt.fixed_K ? h->opt.K
                                    : mca::batch_width_cost(h->rate_acc, h->rate_trials,
                                                            h->tfm ? mca::kBatchCostTfm
                                                                   : mca::kBatchCostDeep,
                                                            h->opt.K);
      uint64_t kb = std::min<uint64_t>(remaining, (uint64_t)Kw);
      if (R > 0) kb = std::min<uint64_t>(kb, R - h->tau % R);
      if (!h->ev[0]) {
        for (auto& e : h->ev) CUDA_TRY(h, cudaEventCreate(&e));
      }
      CUDA_TRY(h, cudaEventRecord(h->ev[0], h->stream));
      if (h->tfm) {
        ta.tau = h->tau;
        ta.Kb = (int)kb;
        ta.nscr = h->nscr;
        ta.scrX = h->tfm_scrX;
        ta.scr_ell = h->tfm_scr_ell;
        CUDA_TRY(h, mca::launch_tfm_eval(ta, h->stream));
        CUDA_TRY(h, cudaEventRecord(h->ev[1], h->stream));
        CUDA_TRY(h, mca::launch_tfm_decide(ta, h->stream));
        // the commit kernel recomputes an accepted candidate beyond the scratch slots (and
        // returns at once otherwise); then the accepted weight's image entry and, for a
        // candidate with a slot, its adoption
        CUDA_TRY(h, mca::launch_tfm_commit(ta, h->stream));
        if (ta.tc) {
          CUDA_TRY(h, mca::launch_tfm_tc_adopt(ta, h->stream));
          h->launches += 1;
        }
      } else {
        a.tau = h->tau;
        a.Kb = (int)kb;
        a.scr = h->scr_dev;
        a.nscr = h->nscr;
        CUDA_TRY(h, mca::launch_deep_eval(a, h->stream));
        CUDA_TRY(h, cudaEventRecord(h->ev[1], h->stream));
        CUDA_TRY(h, mca::launch_deep_decide(a, h->stream));
        // with scratch slots the commit follows the decision on the host (below)
        if (h->nscr == 0) CUDA_TRY(h, mca::launch_deep_commit(a, h->stream));
        else h->launches -= 1;
      }
      CUDA_TRY(h, cudaEventRecord(h->ev[2], h->stream));
      h->launches += 3;
      mca::DeepCtl ctl;
      CUDA_TRY(h, cudaMemcpyAsync(&ctl, h->ctl, sizeof(ctl), cudaMemcpyDeviceToHost, h->stream));
      CUDA_TRY(h, cudaStreamSynchronize(h->stream));
      {
        float ms_eval = 0.0f, ms_rest = 0.0f, ms_c = 0.0f;
        CUDA_TRY(h, cudaEventElapsedTime(&ms_eval, h->ev[0], h->ev[1]));
        CUDA_TRY(h, cudaEventElapsedTime(&ms_rest, h->ev[1], h->ev[2]));
        if (h->ev_c_pending) {             // the previous batch's adoption or commit
          CUDA_TRY(h, cudaEventElapsedTime(&ms_c, h->ev_c[0], h->ev_c[1]));
          h->ev_c_pending = false;
        }
        h->eval_ns += (uint64_t)(ms_eval * 1e6f);
        h->rest_ns += (uint64_t)((ms_rest + ms_c) * 1e6f);
      }
      if (ctl.kstar == -2 || ctl.consumed <= 0) {
        h->broken = true;
        return fail(h, MCA_ERR_NUMERIC, "non-finite loss change");
      }
      if (!h->tfm && h->nscr > 0 && ctl.kstar >= 0) {
        // The accepted candidate's fields: adopted from its scratch slot (row j of its layer
        // copied, the later layers' arrays and the losses swapped with the slot's), or, for a
        // candidate without a dense chain or beyond the slots, recomputed by the commit kernel.
        if (!h->ev_c[0]) {
          for (auto& e : h->ev_c) CUDA_TRY(h, cudaEventCreate(&e));
        }
        CUDA_TRY(h, cudaEventRecord(h->ev_c[0], h->stream));
        const mca::DeepCand& c = ctl.acc;
        const int L = (int)h->layers.size();
        if (ctl.kstar < h->nscr && c.valid && c.delta != 0.0f && c.layer <= L - 3) {
          float** sk = h->scr.data() + (size_t)ctl.kstar * (L + 1);
          const size_t row = (size_t)c.row * h->Np;
          CUDA_TRY(h, cudaMemcpyAsync(h->Z[c.layer] + row, sk[c.layer] + row,
                                      sizeof(float) * (size_t)h->N, cudaMemcpyDeviceToDevice,
                                      h->stream));
          for (int m = c.layer + 1; m < L; ++m) std::swap(h->Z[m], sk[m]);
          std::swap(h->ell, sk[L]);
          CUDA_TRY(h, cudaMemcpyAsync(h->scr_dev + (size_t)ctl.kstar * (L + 1), sk,
                                      sizeof(float*) * (size_t)(L + 1), cudaMemcpyHostToDevice,
                                      h->stream));
          const uint64_t sd = a.seed;
          a = deep_args(h);
          a.seed = sd;
        } else {
          CUDA_TRY(h, mca::launch_deep_commit(a, h->stream));
          h->launches += 1;
        }
        CUDA_TRY(h, cudaEventRecord(h->ev_c[1], h->stream));
        h->ev_c_pending = true;
        if (remaining == (uint64_t)ctl.consumed) {   // the run's last batch: its time now
          float ms_c = 0.0f;
          CUDA_TRY(h, cudaEventSynchronize(h->ev_c[1]));
          CUDA_TRY(h, cudaEventElapsedTime(&ms_c, h->ev_c[0], h->ev_c[1]));
          h->rest_ns += (uint64_t)(ms_c * 1e6f);
          h->ev_c_pending = false;
        }
      }
      h->tau += (uint64_t)ctl.consumed;
      remaining -= (uint64_t)ctl.consumed;
      h->rate_acc = h->rate_acc * mca::kRateDecay + (ctl.kstar >= 0 ? 1.0f : 0.0f);
      h->rate_trials = h->rate_trials * mca::kRateDecay + (float)ctl.consumed;
      if (R > 0 && h->tau % R == 0) {
        mca_status rc = resync(h);
        if (rc != MCA_OK) return rc;
        h->resyncs++;
      }
    }
  }
  while (remaining > 0) {
    NvtxRange nv_seg("mca trial-loop segment");
    uint64_t seg = remaining;
    const uint64_t R = (uint64_t)h->opt.resync_period;
    if (R > 0) seg = std::min<uint64_t>(seg, R - h->tau % R);
    mca::Mlp2Args a = mlp2_args(h);
    a.seed = seed;
    a.tau0 = h->tau;
    a.n_trials = seg;
    CUDA_TRY(h, cudaMemsetAsync(h->bar, 0, sizeof(GridBarrier), h->stream));
    CUDA_TRY(h, cudaMemsetAsync(h->accum, 0, sizeof(unsigned long long) * 3 * mca::kAccStride,
                                h->stream));
    CUDA_TRY(h, mca::launch_mlp2_loop(a, h->stream));
    h->launches++;
    h->tau += seg;
    remaining -= seg;
    if (R > 0 && h->tau % R == 0) {
      mca_status rc = resync(h);
      if (rc != MCA_OK) return rc;
      h->resyncs++;
    }
  }
  DevState ds;
  mca_status rc = read_state(h, &ds);
  if (rc != MCA_OK) return rc;
  if (stats) fill_stats(h, ds, stats);
  if (ds.err != 0) {
    h->broken = true;
    return fail(h, (mca_status)ds.err, ds.err == MCA_ERR_TIMEOUT
                                           ? "device-side wait timed out"
                                           : "non-finite loss change");
  }
  return MCA_OK;
}

mca_status mca_loss(mca_handle* h, double* L) {
  if (!h || !L) return fail(h, MCA_ERR_INVALID, "NULL argument");
  DevState ds;
  mca_status rc = read_state(h, &ds);
  if (rc != MCA_OK) return rc;
  *L = ds.S / (double)h->N;
  return MCA_OK;
}

mca_status mca_get_stats(mca_handle* h, mca_run_stats* stats) {
  if (!h || !stats) return fail(h, MCA_ERR_INVALID, "NULL argument");
  DevState ds;
  mca_status rc = read_state(h, &ds);
  if (rc != MCA_OK) return rc;
  fill_stats(h, ds, stats);
  return MCA_OK;
}

mca_status mca_get_params(mca_handle* h, float* dst, size_t n) {
  if (!h || !dst) return fail(h, MCA_ERR_INVALID, "NULL argument");
  if (n != h->P) return fail(h, MCA_ERR_INVALID, "n = %zu, P = %llu", n, h->P);
  for (size_t l = 0; l < h->layers.size(); ++l) {
    const size_t m = (size_t)h->layers[l].n_in * h->layers[l].n_out;
    CUDA_TRY(h, cudaMemcpyAsync(dst + h->off[l], h->w_eff[l], sizeof(float) * m, cudaMemcpyDefault,
                                h->stream));
  }
  CUDA_TRY(h, cudaStreamSynchronize(h->stream));
  return MCA_OK;
}

mca_status mca_get_codes(mca_handle* h, int8_t* dst, size_t n) {
  if (!h || !dst) return fail(h, MCA_ERR_INVALID, "NULL argument");
  if (n != h->P) return fail(h, MCA_ERR_INVALID, "n = %zu, P = %llu", n, h->P);
  const bool dev = is_device_ptr(dst);
  for (size_t l = 0; l < h->layers.size(); ++l) {
    const size_t m = (size_t)h->layers[l].n_in * h->layers[l].n_out;
    if (h->code[l]) {
      CUDA_TRY(h, cudaMemcpyAsync(dst + h->off[l], h->code[l], m, cudaMemcpyDefault, h->stream));
    } else if (dev) {
      CUDA_TRY(h, cudaMemsetAsync(dst + h->off[l], 0, m, h->stream));
    } else {
      CUDA_TRY(h, cudaStreamSynchronize(h->stream));
      std::memset(dst + h->off[l], 0, m);
    }
  }
  CUDA_TRY(h, cudaStreamSynchronize(h->stream));
  return MCA_OK;
}

mca_status mca_set_params(mca_handle* h, const float* params, const int8_t* codes, size_t n,
                          uint64_t tau) {
  if (!h || !params) return fail(h, MCA_ERR_INVALID, "NULL argument");
  if (h->broken) return fail(h, MCA_ERR_CUDA, "handle unusable after an earlier device error");
  if (n != h->P) return fail(h, MCA_ERR_INVALID, "n = %zu, P = %llu", n, h->P);
  mca_status rc = load_params(h, params, reinterpret_cast<const signed char*>(codes));
  if (rc != MCA_OK) return rc;
  rc = resync(h);
  if (rc != MCA_OK) return rc;
  h->tau = tau;
  return MCA_OK;
}

mca_status mca_resync(mca_handle* h) {
  if (!h) return fail(nullptr, MCA_ERR_INVALID, "NULL handle");
  if (h->broken) return fail(h, MCA_ERR_CUDA, "handle unusable after an earlier device error");
  mca_status rc = resync(h);
  if (rc != MCA_OK) return rc;
  DevState ds;
  rc = read_state(h, &ds);
  if (rc != MCA_OK) return rc;
  if (ds.err == MCA_ERR_TIMEOUT) {
    h->broken = true;
    return fail(h, MCA_ERR_TIMEOUT, "device-side wait timed out in the forward pass");
  }
  return MCA_OK;
}

mca_status mca_get_trace(mca_handle* h, mca_trace_rec* dst, size_t cap, size_t* n) {
  if (!h || !n || (!dst && cap)) return fail(h, MCA_ERR_INVALID, "NULL argument");
  if (h->trace_cap <= 0) return fail(h, MCA_ERR_INVALID, "created without a trace");
  DevState ds;
  mca_status rc = read_state(h, &ds);
  if (rc != MCA_OK) return rc;
  const unsigned long long tc = (unsigned long long)h->trace_cap;
  const unsigned long long have = std::min<unsigned long long>(ds.trace_written, tc);
  const unsigned long long take = std::min<unsigned long long>(have, cap);
  std::vector<mca_trace_rec> ring(tc);
  CUDA_TRY(h, cudaMemcpyAsync(ring.data(), h->trace, sizeof(mca_trace_rec) * tc,
                              cudaMemcpyDeviceToHost, h->stream));
  CUDA_TRY(h, cudaStreamSynchronize(h->stream));
  const unsigned long long first = ds.trace_written - take;
  for (unsigned long long m = 0; m < take; ++m) dst[m] = ring[(first + m) % tc];
  *n = (size_t)take;
  return MCA_OK;
}

mca_status mca_force_decisions(mca_handle* h, const uint64_t* tau, const uint8_t* accept,
                               size_t n) {
  if (!h) return fail(nullptr, MCA_ERR_INVALID, "NULL handle");
  if (n && (!tau || !accept)) return fail(h, MCA_ERR_INVALID, "NULL argument");
  for (size_t m = 1; m < n; ++m)
    if (tau[m] <= tau[m - 1]) return fail(h, MCA_ERR_INVALID, "tau not strictly increasing");
  if (h->ftau) cudaFree(h->ftau);
  if (h->facc) cudaFree(h->facc);
  h->ftau = nullptr;
  h->facc = nullptr;
  h->nforce = 0;
  if (n == 0) return MCA_OK;
  CUDA_TRY(h, cudaMalloc(&h->ftau, sizeof(unsigned long long) * n));
  CUDA_TRY(h, cudaMalloc(&h->facc, n));
  CUDA_TRY(h, cudaMemcpyAsync(h->ftau, tau, sizeof(unsigned long long) * n, cudaMemcpyHostToDevice,
                              h->stream));
  CUDA_TRY(h, cudaMemcpyAsync(h->facc, accept, n, cudaMemcpyHostToDevice, h->stream));
  CUDA_TRY(h, cudaStreamSynchronize(h->stream));
  h->nforce = (int)n;
  return MCA_OK;
}

namespace {

// Loss changes of the n candidates in h->ex_idx / h->ex_new against the current state, no commit,
// into dS (host). The evaluation kernels of mca_run's evaluation step.
mca_status eval_explicit(mca_handle* h, size_t n, double* dS) {
  if (h->tfm) {
    mca::TfmArgs a = tfm_args(h);
    a.n_explicit = (int)n;
    a.ex_idx = h->ex_idx;
    a.ex_new = h->ex_new;
    a.ex_out = h->ex_out;
    CUDA_TRY(h, mca::launch_tfm_eval(a, h->stream));
    CUDA_TRY(h, mca::launch_tfm_decide(a, h->stream));
    h->launches += 2;
  } else if (h->deep) {
    mca::DeepArgs a = deep_args(h);
    a.n_explicit = (int)n;
    a.ex_idx = h->ex_idx;
    a.ex_new = h->ex_new;
    a.ex_out = h->ex_out;
    CUDA_TRY(h, mca::launch_deep_eval(a, h->stream));
    CUDA_TRY(h, mca::launch_deep_decide(a, h->stream));
    h->launches += 2;
  } else {
    mca::Mlp2Args a = mlp2_args(h);
    a.n_explicit = (int)n;
    a.ex_idx = h->ex_idx;
    a.ex_new = h->ex_new;
    a.ex_out = h->ex_out;
    CUDA_TRY(h, cudaMemsetAsync(h->bar, 0, sizeof(GridBarrier), h->stream));
    CUDA_TRY(h, mca::launch_mlp2_loop(a, h->stream));
    h->launches++;
  }
  CUDA_TRY(h, cudaMemcpyAsync(dS, h->ex_out, sizeof(double) * n, cudaMemcpyDeviceToHost,
                              h->stream));
  CUDA_TRY(h, cudaStreamSynchronize(h->stream));
  DevState ds;
  mca_status rc = read_state(h, &ds);
  if (rc != MCA_OK) return rc;
  if (ds.err == MCA_ERR_TIMEOUT) {
    h->broken = true;
    return fail(h, MCA_ERR_TIMEOUT, "device-side wait timed out");
  }
  return MCA_OK;
}

}  // namespace

mca_status mca_eval_candidates(mca_handle* h, const uint32_t* flat_idx, const float* new_w,
                               size_t n, double* dS) {
  if (!h || (n && (!flat_idx || !new_w || !dS))) return fail(h, MCA_ERR_INVALID, "NULL argument");
  if (n > (size_t)mca::kKmax) return fail(h, MCA_ERR_INVALID, "n = %zu > %d", n, mca::kKmax);
  if (h->broken) return fail(h, MCA_ERR_CUDA, "handle unusable after an earlier device error");
  if (n == 0) return MCA_OK;
  for (size_t m = 0; m < n; ++m) {
    if (flat_idx[m] >= h->P) return fail(h, MCA_ERR_INVALID, "flat_idx[%zu] >= P", m);
    if (!std::isfinite(new_w[m])) return fail(h, MCA_ERR_INVALID, "new_w[%zu] not finite", m);
  }
  CUDA_TRY(h, cudaMemcpyAsync(h->ex_idx, flat_idx, sizeof(unsigned int) * n, cudaMemcpyHostToDevice,
                              h->stream));
  CUDA_TRY(h, cudaMemcpyAsync(h->ex_new, new_w, sizeof(float) * n, cudaMemcpyHostToDevice,
                              h->stream));
  return eval_explicit(h, n, dS);
}

mca_status mca_eval_trials(mca_handle* h, uint64_t seed, uint64_t tau, size_t n,
                           mca_trace_rec* out) {
  if (!h) return fail(nullptr, MCA_ERR_INVALID, "NULL handle");
  if (n && !out) return fail(h, MCA_ERR_INVALID, "NULL out");
  if (n > (size_t)mca::kKmax) return fail(h, MCA_ERR_INVALID, "n = %zu > %d", n, mca::kKmax);
  if (h->broken) return fail(h, MCA_ERR_CUDA, "handle unusable after an earlier device error");
  if (n == 0) return MCA_OK;
  mca::ProposeArgs a;
  std::memset(&a, 0, sizeof(a));
  a.L = (int)h->layers.size();
  a.n = (int)n;
  for (int l = 0; l < a.L; ++l) {
    a.off[l] = h->off[l];
    a.wk[l] = h->layers[l].wkind;
    a.sc[l] = h->layers[l].scale;
    a.w[l] = h->w_eff[l];
    a.code[l] = h->code[l];
    a.wfix[l] = h->wfix[l];
  }
  a.off[a.L] = h->P;
  a.op = h->dom.op;
  a.lo = h->dom.lo;
  a.hi = h->dom.hi;
  a.delta = h->dom.delta;
  a.bound = h->dom.bound;
  a.stretch = h->dom.layer_stretch;
  a.seed = seed;
  a.tau0 = tau;
  a.rec = h->prop;
  a.ex_idx = h->ex_idx;
  a.ex_new = h->ex_new;
  CUDA_TRY(h, mca::launch_propose(a, h->stream));
  h->launches++;
  CUDA_TRY(h, cudaMemcpyAsync(out, h->prop, sizeof(mca_trace_rec) * n, cudaMemcpyDeviceToHost,
                              h->stream));
  double dS[mca::kKmax];
  mca_status rc = eval_explicit(h, n, dS);
  if (rc != MCA_OK) return rc;
  double S = 0.0;
  rc = mca_loss(h, &S);
  if (rc != MCA_OK) return rc;
  S *= (double)h->N;
  for (size_t k = 0; k < n; ++k) {
    out[k].dS = out[k].valid ? dS[k] : std::nan("");
    out[k].S = S;
  }
  return MCA_OK;
}

mca_status mca_decide_batch(mca_handle* h, uint64_t seed, uint64_t tau, size_t n,
                            const uint8_t* valid, const double* dS, int64_t n_samples,
                            int32_t* kstar) {
  if (!h || !kstar || (n && (!valid || !dS))) return fail(h, MCA_ERR_INVALID, "NULL argument");
  if (n_samples < 0) return fail(h, MCA_ERR_INVALID, "n_samples < 0");
  const double N = n_samples > 0 ? (double)n_samples : (double)h->N;
  const int metro = h->dom.temperature > 0.0f ? 1 : 0;
  const double msc = N * (double)h->dom.temperature;
  *kstar = -1;
  for (size_t k = 0; k < n; ++k) {
    if (!valid[k]) continue;
    if (!std::isfinite(dS[k]))
      return fail(h, MCA_ERR_NUMERIC, "non-finite loss change of trial %llu",
                  (unsigned long long)(tau + k));
    if (mca::accept_change((float)dS[k], h->dom.strict, metro, seed, tau + k, msc)) {
      *kstar = (int32_t)k;
      break;
    }
  }
  return MCA_OK;
}

mca_status mca_tfm_workspace_size(const mca_tfm_spec* spec, int64_t n_seq, const mca_options* opt,
                                  size_t* bytes) {
  mca_status rc = tfm_check(spec, n_seq);
  if (rc != MCA_OK) return rc;
  if (!bytes) return fail(nullptr, MCA_ERR_INVALID, "bytes is NULL");
  const mca_options o = opt ? *opt : default_options();
  *bytes = tfm_plan(*spec, n_seq, o.trace_cap, tfm_use_tc(*spec, n_seq), o.K).total;
  return MCA_OK;
}

mca_status mca_create_transformer(const mca_tfm_spec* spec, const mca_domain* dom,
                                  const int32_t* tokens, int64_t n_seq, const float* init_params,
                                  const mca_options* opt, mca_handle** out) {
  NvtxRange nv("mca_create_transformer");
  if (!out) return fail(nullptr, MCA_ERR_INVALID, "out is NULL");
  *out = nullptr;
  mca_status rc = tfm_check(spec, n_seq);
  if (rc != MCA_OK) return rc;
  if (!tokens || !init_params) return fail(nullptr, MCA_ERR_INVALID, "NULL tokens or params");
  const mca_options o = opt ? *opt : default_options();
  if (o.K < 1 || o.K > mca::kKmax)
    return fail(nullptr, MCA_ERR_INVALID, "K = %d outside 1..%d", o.K, mca::kKmax);
  if (o.resync_period < 0 || o.trace_cap < 0) return fail(nullptr, MCA_ERR_INVALID, "negative option");
  const mca_domain d = dom ? *dom : default_domain();
  if (d.op != MCA_OP_REPLACE && d.op != MCA_OP_PERTURB)
    return fail(nullptr, MCA_ERR_INVALID, "unknown op %d", d.op);
  if (!std::isfinite(d.lo) || !std::isfinite(d.hi) || !std::isfinite(d.delta) || !(d.hi > d.lo))
    return fail(nullptr, MCA_ERR_INVALID, "bad domain");
  if (!std::isfinite(d.temperature) || d.temperature < 0.0f)
    return fail(nullptr, MCA_ERR_INVALID, "temperature %g: must be finite and >= 0", d.temperature);
  if (d.layer_stretch < 0)
    return fail(nullptr, MCA_ERR_INVALID, "layer_stretch = %d < 0", d.layer_stretch);
  if (d.layer_stretch > 0)
    return fail(nullptr, MCA_ERR_UNSUPPORTED, "the current-layer schedule is for MLPs");
  mca_handle* h = new (std::nothrow) mca_handle();
  if (!h) return fail(nullptr, MCA_ERR_OOM, "host allocation failed");
  auto bail = [&](mca_status st) {
    g_create_err = h->err;
    mca_destroy(h);
    return st;
  };
  h->tfm = true;
  h->tspec = *spec;
  h->dom = d;
  h->opt = o;
  h->stream = (cudaStream_t)o.stream;
  h->N = n_seq * spec->ctx;
  h->C = spec->vocab;
  h->trace_cap = o.trace_cap;
  const TfmLayout TL = tfm_offsets(*spec);
  h->P = TL.P;
  mca_layer pseudo;
  std::memset(&pseudo, 0, sizeof(pseudo));
  pseudo.n_in = (int32_t)TL.P;
  pseudo.n_out = 1;
  pseudo.wkind = MCA_W_FP32;
  h->layers.push_back(pseudo);
  h->off.push_back(0);
  cudaError_t e = cudaGetDevice(&h->device);
  if (e == cudaSuccess)
    e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
  if (e != cudaSuccess) return bail(fail(h, MCA_ERR_CUDA, "%s", cudaGetErrorString(e)));
  h->tc = tfm_use_tc(*spec, n_seq);
  const TfmMem M = tfm_plan(*spec, n_seq, o.trace_cap, h->tc, o.K);
  if (o.workspace) {
    if (o.workspace_bytes < M.total)
      return bail(fail(h, MCA_ERR_OOM, "workspace of %zu bytes < %zu needed", o.workspace_bytes,
                       M.total));
    if (reinterpret_cast<uintptr_t>(o.workspace) % 256 != 0)
      return bail(fail(h, MCA_ERR_INVALID, "workspace not 256-byte aligned"));
    h->ws = o.workspace;
    h->ws_bytes = o.workspace_bytes;
  } else {
    e = cudaMalloc(&h->ws, M.total);
    if (e != cudaSuccess) return bail(fail(h, MCA_ERR_OOM, "%s", cudaGetErrorString(e)));
    h->ws_owned = true;
    h->ws_bytes = M.total;
  }
  char* base = static_cast<char*>(h->ws);
  h->params = reinterpret_cast<float*>(base + M.params);
  h->w_eff.push_back(h->params);
  h->code.push_back(nullptr);
  h->wfix.push_back(nullptr);
  h->tokens = reinterpret_cast<int*>(base + M.tokens);
  h->X = reinterpret_cast<float*>(base + M.X);
  h->ell = reinterpret_cast<float*>(base + M.ell);
  h->partial = reinterpret_cast<float*>(base + M.partial);
  h->st = reinterpret_cast<DevState*>(base + M.st);
  h->ctl = reinterpret_cast<mca::DeepCtl*>(base + M.ctl);
  h->trace = o.trace_cap > 0 ? reinterpret_cast<mca_trace_rec*>(base + M.trace) : nullptr;
  h->ex_idx = reinterpret_cast<unsigned int*>(base + M.ex_idx);
  h->ex_new = reinterpret_cast<float*>(base + M.ex_new);
  h->ex_out = reinterpret_cast<double*>(base + M.ex_out);
  h->prop = reinterpret_cast<mca_trace_rec*>(base + M.prop);
  h->tfm_img = h->tc ? reinterpret_cast<float*>(base + M.wimg) : nullptr;
  h->tfm_Xmid = h->tc ? reinterpret_cast<float*>(base + M.Xmid) : nullptr;
  h->ctl2 = reinterpret_cast<mca::DeepCtl*>(base + M.ctl2);
  h->tau_dev = reinterpret_cast<unsigned long long*>(base + M.tau_dev);
  h->nscr = M.nscr;
  h->tfm_scrX = reinterpret_cast<float*>(base + M.scrX);
  h->tfm_scr_ell = reinterpret_cast<float*>(base + M.scr_ell);
  e = cudaMemsetAsync(h->st, 0, sizeof(DevState), h->stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(h->ctl, 0, sizeof(mca::DeepCtl), h->stream);
  if (e != cudaSuccess) return bail(fail(h, MCA_ERR_CUDA, "%s", cudaGetErrorString(e)));
  {
    const size_t nt = (size_t)n_seq * (spec->ctx + 1);
    std::vector<int> th(nt);
    e = cudaMemcpyAsync(th.data(), tokens, sizeof(int) * nt, cudaMemcpyDefault, h->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
    if (e != cudaSuccess) return bail(fail(h, MCA_ERR_CUDA, "%s", cudaGetErrorString(e)));
    for (size_t q = 0; q < nt; ++q)
      if (th[q] < 0 || th[q] >= spec->vocab)
        return bail(fail(h, MCA_ERR_INVALID, "token %d outside [0, %d)", th[q], spec->vocab));
    e = cudaMemcpyAsync(h->tokens, th.data(), sizeof(int) * nt, cudaMemcpyHostToDevice, h->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
    if (e != cudaSuccess) return bail(fail(h, MCA_ERR_CUDA, "%s", cudaGetErrorString(e)));
  }
  rc = load_params(h, init_params, nullptr);
  if (rc != MCA_OK) return bail(rc);
  rc = resync(h);
  if (rc != MCA_OK) return bail(rc);
  DevState ds;
  rc = read_state(h, &ds);
  if (rc != MCA_OK) return bail(rc);
  if (!std::isfinite(ds.S)) return bail(fail(h, MCA_ERR_NUMERIC, "initial loss is not finite"));
  *out = h;
  return MCA_OK;
}

mca_status mca_run_channels(mca_handle* h, uint64_t n_trials, uint64_t seed, int32_t scheme,
                            uint8_t* accepted, double* dS) {
  if (!h) return fail(nullptr, MCA_ERR_INVALID, "NULL handle");
  if (h->broken) return fail(h, MCA_ERR_CUDA, "handle unusable after an earlier device error");
  if (scheme != MCA_CHANNEL_HE && scheme != MCA_CHANNEL_ZERO)
    return fail(h, MCA_ERR_INVALID, "unknown channel scheme %d", scheme);
  if (h->tfm) return fail(h, MCA_ERR_UNSUPPORTED, "channel mutations are for MLPs");
  const int L = (int)h->layers.size();
  for (int m = 0; m < L; ++m)
    if (h->layers[m].wkind != MCA_W_FP32)
      return fail(h, MCA_ERR_UNSUPPORTED, "layer %d is not fp32", m);
  NvtxRange nv("mca_run_channels");
  // forced decisions, as a host copy of the device lists
  std::vector<unsigned long long> ftau(h->nforce);
  std::vector<unsigned char> facc(h->nforce);
  if (h->nforce > 0) {
    CUDA_TRY(h, cudaMemcpyAsync(ftau.data(), h->ftau, sizeof(unsigned long long) * h->nforce,
                                cudaMemcpyDeviceToHost, h->stream));
    CUDA_TRY(h, cudaMemcpyAsync(facc.data(), h->facc, h->nforce, cudaMemcpyDeviceToHost,
                                h->stream));
    CUDA_TRY(h, cudaStreamSynchronize(h->stream));
  }
  std::vector<int> node(L + 1);
  std::vector<float> oldw(L), neww(L);
  std::vector<float*> at(L);
  DevState ds;
  mca_status rc = read_state(h, &ds);
  if (rc != MCA_OK) return rc;
  double S = ds.S;
  for (uint64_t t = 0; t < n_trials; ++t) {
    const uint64_t tau = h->tau;
    for (int m = 0; m <= L; ++m) {
      const unsigned long long n_m =
          m == 0 ? (unsigned long long)h->layers[0].n_in : (unsigned long long)h->layers[m - 1].n_out;
      node[m] = mca::channel_node(mca::channel_word(seed, tau, m), n_m);
    }
    for (int m = 0; m < L; ++m) {
      const mca_layer& ly = h->layers[m];
      at[m] = h->w_eff[m] + (size_t)node[m + 1] * ly.n_in + node[m];
      neww[m] = scheme == MCA_CHANNEL_HE
                    ? mca::channel_he_value(mca::channel_word(seed, tau, L + 1 + m), ly.n_in)
                    : 0.0f;
      CUDA_TRY(h, cudaMemcpyAsync(&oldw[m], at[m], sizeof(float), cudaMemcpyDeviceToHost,
                                  h->stream));
    }
    CUDA_TRY(h, cudaStreamSynchronize(h->stream));
    for (int m = 0; m < L; ++m)
      CUDA_TRY(h, cudaMemcpyAsync(at[m], &neww[m], sizeof(float), cudaMemcpyHostToDevice,
                                  h->stream));
    rc = resync(h);
    if (rc != MCA_OK) return rc;
    rc = read_state(h, &ds);
    if (rc != MCA_OK) return rc;
    const double d = ds.S - S;
    if (!std::isfinite(d)) {
      h->broken = true;
      return fail(h, MCA_ERR_NUMERIC, "non-finite loss change");
    }
    bool acc;
    const auto it = std::lower_bound(ftau.begin(), ftau.end(), (unsigned long long)tau);
    if (it != ftau.end() && *it == tau) {
      acc = facc[it - ftau.begin()] != 0;
    } else {
      acc = mca::accept_change((float)d, h->dom.strict, h->dom.temperature > 0.0f ? 1 : 0, seed,
                               tau, (double)h->N * (double)h->dom.temperature);
    }
    if (accepted) accepted[t] = acc ? 1 : 0;
    if (dS) dS[t] = d;
    if (acc) {
      S = ds.S;
    } else {
      for (int m = L - 1; m >= 0; --m)
        CUDA_TRY(h, cudaMemcpyAsync(at[m], &oldw[m], sizeof(float), cudaMemcpyHostToDevice,
                                    h->stream));
      rc = resync(h);
      if (rc != MCA_OK) return rc;
      CUDA_TRY(h, cudaStreamSynchronize(h->stream));
    }
    h->tau = tau + 1;
  }
  return MCA_OK;
}

mca_status mca_selftest_wait_timeout(int32_t* status, double* waited_ms) {
  if (!status) return fail(nullptr, MCA_ERR_INVALID, "status is NULL");
  NvtxRange nv("mca wait self-test");
  void* mem = nullptr;
  cudaError_t e = cudaMalloc(&mem, 256);
  if (e != cudaSuccess) return fail(nullptr, MCA_ERR_CUDA, "%s", cudaGetErrorString(e));
  GridBarrier* bar = static_cast<GridBarrier*>(mem);
  int* err = reinterpret_cast<int*>(static_cast<char*>(mem) + 64);
  e = cudaMemset(mem, 0, 256);
  const auto t0 = std::chrono::steady_clock::now();
  if (e == cudaSuccess) {
    wait_selftest_kernel<<<1, 32, 0, 0>>>(bar, err);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(0);
  const double ms =
      std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0).count();
  int h_err = -1;
  if (e == cudaSuccess) e = cudaMemcpy(&h_err, err, sizeof(int), cudaMemcpyDeviceToHost);
  const cudaError_t ef = cudaFree(mem);
  if (e == cudaSuccess) e = ef;
  if (e != cudaSuccess) return fail(nullptr, MCA_ERR_CUDA, "%s", cudaGetErrorString(e));
  *status = h_err;
  if (waited_ms) *waited_ms = ms;
  return MCA_OK;
}

void mca_destroy(mca_handle* h) {
  if (!h) return;
  cudaStreamSynchronize(h->stream);
  for (auto& e : h->ev)
    if (e) cudaEventDestroy(e);
  for (auto& e : h->ev_c)
    if (e) cudaEventDestroy(e);
  for (auto& b : h->ev_p)
    for (auto& e : b)
      if (e) cudaEventDestroy(e);
  if (h->pipe_host) cudaFreeHost(h->pipe_host);
  if (h->ws_owned && h->ws) cudaFree(h->ws);
  if (h->ftau) cudaFree(h->ftau);
  if (h->facc) cudaFree(h->facc);
  delete h;
}

}  // extern "C"
