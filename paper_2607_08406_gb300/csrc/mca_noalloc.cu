// mca_eval_candidates_noalloc: the candidate evaluation of mca_eval_candidates for callers that
// cannot allocate device memory (see include/mca.h). The evaluation kernel needs scratch beyond its
// inputs and outputs -- one partial loss change per (candidate, sample range) and a grid barrier --
// and here that scratch is a fixed array of this file instead of the handle's workspace, so the call
// makes no cudaMalloc, cudaFree or other allocating call.
#include <cmath>
#include <cstring>
#include <mutex>
#include <string>

#include "mca_device.cuh"
#include "mca_internal.h"

namespace {

constexpr int kNoAllocMaxCandidates = mca::kKmax;   // 128
constexpr int kNoAllocMaxRanges = 256;              // sample ranges (CTAs) of the handle
constexpr size_t kNoAllocBarrierBytes = 256;
constexpr size_t kNoAllocBytes =
    kNoAllocBarrierBytes + sizeof(float) * (size_t)kNoAllocMaxCandidates * kNoAllocMaxRanges;

// 128 KB + 256 B of device memory, held by every GPU that loads the library until the process
// exits. Shared by every call: the barrier slot is cleared at the start of each call; the partials
// are written before they are read.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up once per device).
cudaError_t scratch_address(int dev, void** out) {
  std::lock_guard<std::mutex> lock(g_mutex);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return cudaSuccess;
}

bool on_device(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

mca_status set_err(mca_handle* h, mca_status st, const std::string& msg) {
  h->err = msg;
  return st;
}

}  // namespace

extern "C" mca_status mca_eval_candidates_noalloc(mca_handle* h, const uint32_t* flat_idx,
                                                  const float* new_w, size_t n, double* dS) {
  if (!h) return MCA_ERR_INVALID;
  if (n == 0) return MCA_OK;
  if (!flat_idx || !new_w || !dS) return set_err(h, MCA_ERR_INVALID, "NULL argument");
  if (h->broken)
    return set_err(h, MCA_ERR_CUDA, "handle unusable after an earlier device error");
  // single-hidden-layer handles only; refused before any CUDA call, the handle stays usable
  if (h->deep || h->tfm)
    return set_err(h, MCA_ERR_UNSUPPORTED,
                   "the no-allocation evaluation runs single-hidden-layer handles only");
  if (n > (size_t)kNoAllocMaxCandidates)
    return set_err(h, MCA_ERR_INVALID,
                   "n = " + std::to_string(n) + " candidates exceeds the no-allocation maximum of " +
                       std::to_string(kNoAllocMaxCandidates));
  if (h->NR > kNoAllocMaxRanges)
    return set_err(h, MCA_ERR_INVALID,
                   "handle uses " + std::to_string(h->NR) +
                       " sample ranges; the no-allocation scratch holds at most " +
                       std::to_string(kNoAllocMaxRanges));
  // the scratch address and the handle's stream both belong to the current device, so the
  // caller must have made the handle's device current (a mistake, not a device error)
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    return set_err(h, MCA_ERR_INVALID, "no usable current device");
  }
  if (dev != h->device)
    return set_err(h, MCA_ERR_INVALID,
                   "current device " + std::to_string(dev) + " is not the handle's device " +
                       std::to_string(h->device) + "; make the handle's device current first");
  if (!on_device(flat_idx) || !on_device(new_w) || !on_device(dS))
    return set_err(h, MCA_ERR_INVALID, "flat_idx, new_w and dS must be device pointers");
  // the kernel trusts its indices: check them (and the values) on the host, on the stack
  uint32_t hidx[kNoAllocMaxCandidates];
  float hnew[kNoAllocMaxCandidates];
  cudaError_t e = cudaMemcpyAsync(hidx, flat_idx, sizeof(uint32_t) * n, cudaMemcpyDeviceToHost,
                                  h->stream);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(hnew, new_w, sizeof(float) * n, cudaMemcpyDeviceToHost, h->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
  if (e != cudaSuccess) {
    h->broken = true;
    return set_err(h, MCA_ERR_CUDA, std::string("reading candidates: ") + cudaGetErrorString(e));
  }
  for (size_t m = 0; m < n; ++m) {
    if (hidx[m] >= h->P)
      return set_err(h, MCA_ERR_INVALID, "flat_idx[" + std::to_string(m) + "] >= P");
    if (!std::isfinite(hnew[m]))
      return set_err(h, MCA_ERR_INVALID, "new_w[" + std::to_string(m) + "] not finite");
  }
  void* base = nullptr;
  e = scratch_address(dev, &base);
  if (e != cudaSuccess)
    return set_err(h, MCA_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));

  mca::Mlp2Args a = mca::handle_mlp2_args(h);
  a.n_explicit = (int)n;
  a.ex_idx = flat_idx;
  a.ex_new = new_w;
  a.ex_out = dS;
  a.bar = reinterpret_cast<mca::GridBarrier*>(base);
  a.partial = reinterpret_cast<float*>(static_cast<char*>(base) + kNoAllocBarrierBytes);
  e = cudaMemsetAsync(base, 0, sizeof(mca::GridBarrier), h->stream);
  if (e == cudaSuccess) e = mca::launch_mlp2_loop(a, h->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
  int derr = 0;
  if (e == cudaSuccess)
    e = cudaMemcpy(&derr, &h->st->err, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) {
    h->broken = true;
    return set_err(h, MCA_ERR_CUDA, std::string("evaluation launch: ") + cudaGetErrorString(e));
  }
  h->launches++;
  if (derr == MCA_ERR_TIMEOUT) {
    h->broken = true;
    return set_err(h, MCA_ERR_TIMEOUT, "device-side wait timed out");
  }
  return MCA_OK;
}
