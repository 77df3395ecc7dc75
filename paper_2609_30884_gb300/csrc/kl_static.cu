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
constexpr int kNoallocMaxSplits = 256;
constexpr int kPartFloats = 5;  // (max*, sum*, dot*, max, sum) per (row, split)
constexpr int kMaxDevices = 64;

// Per-(row, split) partials of one call: 32 x 256 x 5 floats = 160 KiB.
static __device__ __align__(256) float g_kl_scratch[kNoallocMaxRows * kNoallocMaxSplits * kPartFloats];

std::mutex g_setup_mu;
float* g_scratch_addr[kMaxDevices] = {};

// Device address of g_kl_scratch on `device` (which must be current). Looked
// up once per device; the host-side name of the array is not a device address.
crf_status scratch_on(int device, float** out) {
  std::lock_guard<std::mutex> lock(g_setup_mu);
  if (!g_scratch_addr[device]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_kl_scratch);
    if (e != cudaSuccess || !p) {
      crf::set_last_error(cudaGetErrorString(e));
      return CRF_ECUDA;
    }
    g_scratch_addr[device] = static_cast<float*>(p);
  }
  *out = g_scratch_addr[device];
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
    int splits = (2 * sms + n_rows - 1) / n_rows;
    splits = splits < (vocab + 1023) / 1024 ? splits : (vocab + 1023) / 1024;
    splits = splits < kNoallocMaxSplits ? splits : kNoallocMaxSplits;
    splits = splits < 1 ? 1 : splits;
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
