// crf_kl_logits_noalloc: the first-step KL from logits (forward KL, fresh
// model as reference, Section S2.1) with its scratch in a fixed device array
// instead of a caller-provided workspace.
//
// Some callers cannot allocate device memory at the point where they need the
// fidelity number: a serving loop that runs under a fixed device-memory budget
// partitioned at start-up, or a C host without a device allocator of its own.
// This entry point lets them call the KL reduction with only their inputs and
// outputs. Its per-split partial sums live in g_kl_scratch, a file-scope
// device array that every GPU which loads this library holds until the
// process exits.
#include "../../include/crf.h"
#include "common.cuh"
#include "kernels.h"

#include <mutex>

namespace crf {
void set_last_error(const char* msg);
}

namespace {

constexpr int kNoallocMaxRows = 32;
constexpr int kPartFloats = 5;  // (max*, sum*, dot*, max, sum) per (row, split)
constexpr int kMaxDevices = 64;

// Per-(row, split) partials of one call: 32 x 256 x 5 floats = 160 KiB.
static __device__ __align__(256) float g_kl_scratch[kNoallocMaxRows * crf::kKlMaxSplits * kPartFloats];

using CtxGetCurrentFn = CUresult (*)(CUcontext*);

// cuCtxGetCurrent from the driver, through the runtime's entry-point query (the library links
// only the runtime). Null if the driver does not provide it.
CtxGetCurrentFn ctx_get_current() {
  static CtxGetCurrentFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<CtxGetCurrentFn>(p);
    return static_cast<CtxGetCurrentFn>(nullptr);
  }();
  return fn;
}

std::mutex g_setup_mu;
struct Setup {
  CUcontext ctx;
  float* addr;
};
Setup g_setup[kMaxDevices] = {};

// Device address of g_kl_scratch on `device`, which must be current. The host-side name of the
// array is not a device address, so the address is looked up with cudaGetSymbolAddress: once
// per device and context. A device reset followed by a new primary context gives a new context
// handle, and the address is looked up again for it instead of reusing the old context's.
crf_status scratch_on(int device, float** out) {
  CtxGetCurrentFn get = ctx_get_current();
  if (!get) {
    crf::set_last_error("crf_kl_logits_noalloc: cuCtxGetCurrent is unavailable");
    return CRF_ECUDA;
  }
  // the runtime binds the device's primary context on first use; make that happen first
  if (cudaFree(nullptr) != cudaSuccess) {
    crf::set_last_error("crf_kl_logits_noalloc: cannot initialise the device context");
    return CRF_ECUDA;
  }
  CUcontext cur = nullptr;
  if (get(&cur) != CUDA_SUCCESS || !cur) {
    crf::set_last_error("crf_kl_logits_noalloc: no current CUDA context");
    return CRF_ECUDA;
  }
  std::lock_guard<std::mutex> lock(g_setup_mu);
  Setup& s = g_setup[device];
  if (s.ctx != cur || !s.addr) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_kl_scratch);
    if (e != cudaSuccess || !p) {
      crf::set_last_error(cudaGetErrorString(e));
      return CRF_ECUDA;
    }
    s.ctx = cur;
    s.addr = static_cast<float*>(p);
  }
  *out = s.addr;
  return CRF_OK;
}

}  // namespace

extern "C" crf_status crf_kl_logits_noalloc(int device, const float* z_ref, const float* z_cur,
                                            int n_rows, int vocab, float* out_kl, void* stream) {
  if (!z_ref || !z_cur || !out_kl) {
    crf::set_last_error("crf_kl_logits_noalloc: null pointer");
    return CRF_EINVAL;
  }
  if (vocab < 1 || n_rows < 1) {
    crf::set_last_error("crf_kl_logits_noalloc: n_rows and vocab must be positive");
    return CRF_EINVAL;
  }
  if (n_rows > kNoallocMaxRows) {
    crf::set_last_error("crf_kl_logits_noalloc: n_rows exceeds the 32 rows of its fixed scratch");
    return CRF_EUNSUPPORTED;
  }
  int count = 0;
  if (cudaGetDeviceCount(&count) != cudaSuccess || device < 0 || device >= count ||
      device >= kMaxDevices) {
    crf::set_last_error("crf_kl_logits_noalloc: device out of range");
    return CRF_EINVAL;
  }
  int prev = 0;
  if (cudaGetDevice(&prev) != cudaSuccess || cudaSetDevice(device) != cudaSuccess) {
    crf::set_last_error("crf_kl_logits_noalloc: cannot make the device current");
    return CRF_ECUDA;
  }
  float* part = nullptr;
  crf_status st = scratch_on(device, &part);
  if (st == CRF_OK) {
    int sms = 1;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
    // the same split count as crf_kl, so both reduce in the same order; at most kKlMaxSplits
    const int splits = crf::kl_split_count(sms, n_rows, vocab);
    // Every (row, split) partial is written before it is read: nothing needs clearing.
    const cudaError_t e = crf::launch_kl(z_ref, z_cur, n_rows, vocab, out_kl, part, splits,
                                         static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) {
      crf::set_last_error(cudaGetErrorString(e));
      st = CRF_ECUDA;
    }
  }
  cudaSetDevice(prev);
  return st;
}
