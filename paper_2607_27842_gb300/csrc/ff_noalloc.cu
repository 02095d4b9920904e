// featfix_op_verify_noalloc: the paid-check kernel of featfix_op_verify with
// its scratch in a fixed array compiled into this library, for callers that
// cannot allocate device memory (see include/featfix_ops.h).
#include "featfix_ops.h"
#include "ff_common.cuh"

namespace {

// Scratch of the verify reduction: one 4-double partial per 8-CTA cluster
// of a launch.  512 partials = 16 KiB, held by every GPU that loads the
// library until the process exits.
constexpr size_t kNoallocScratchBytes = FEATFIX_VERIFY_NOALLOC_SCRATCH_BYTES;
static __device__ __align__(256) double g_verify_scratch[kNoallocScratchBytes / sizeof(double)];

// Device address of the array on the current device.  Host code only sees a
// host-side stand-in under the array's name, so the address is looked up with
// the device current -- on every call: after a device reset or a re-created
// primary context the module may be loaded at another address, and once the
// module is loaded the lookup is cheap.
cudaError_t scratch_address(void** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_verify_scratch);
  if (e != cudaSuccess) return e;
  *out = p;
  return cudaSuccess;
}

}  // namespace

extern "C" {

featfix_status featfix_op_verify_noalloc(int dtype, void* dev_u, const void* const* dev_hist, const double* w,
                                         int n_terms, const void* dev_hf, long long n, int write_draft,
                                         double* dev_sums, void* stream) {
  if ((dtype != FEATFIX_DTYPE_F32 && dtype != FEATFIX_DTYPE_BF16) || !dev_u || !dev_hist || !w || !dev_hf ||
      !dev_sums || n_terms < 1 || n_terms > 4 || n <= 0)
    return FEATFIX_ERR_INVALID_ARG;
  if (((uintptr_t)dev_u & 15) || ((uintptr_t)dev_hf & 15)) return FEATFIX_ERR_INVALID_ARG;
  if (ff::verify_workspace_bytes(n) > kNoallocScratchBytes) return FEATFIX_ERR_INVALID_ARG;
  ff::Hist4 h = {{nullptr, nullptr, nullptr, nullptr}};
  float wf[4] = {0, 0, 0, 0};
  for (int j = 0; j < n_terms; ++j) {
    if (!dev_hist[j] || ((uintptr_t)dev_hist[j] & 15)) return FEATFIX_ERR_INVALID_ARG;
    h.p[j] = dev_hist[j];
    wf[j] = (float)w[j];
  }
  void* scratch = nullptr;
  if (scratch_address(&scratch) != cudaSuccess) return FEATFIX_ERR_CUDA;
  // Every partial the launch reads back is written by the same launch, so
  // the array needs no clearing between calls.
  const cudaError_t e = ff::launch_verify((ff::DType)dtype, dev_u, h, wf, n_terms, dev_hf, n, write_draft, dev_sums,
                                          scratch, (cudaStream_t)stream);
  if (e == cudaSuccess) return FEATFIX_OK;
  return e == cudaErrorInvalidValue ? FEATFIX_ERR_INVALID_ARG : FEATFIX_ERR_CUDA;
}

}  // extern "C"
