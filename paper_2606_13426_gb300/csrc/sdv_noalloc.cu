// sdv_noalloc.cu - sdv_verify_noalloc: the whole verification step with its
// scratch memory in a static device array instead of a caller-provided workspace.
//
// Who needs this: code that may not call cudaMalloc at all.  Typical cases are
// plug-ins loaded into a host program that owns every device allocation through
// its own allocator (custom operators of an inference server, stages of a media
// or rendering pipeline), and real-time loops where cudaMalloc's implicit device
// synchronisation and its possible failure at run time are not acceptable.  Such
// callers can still hand over their input and output buffers; only the scratch
// has to come from somewhere else.
//
// The scratch is a file-scope __device__ array of SDV_NOALLOC_SCRATCH_BYTES.  Every
// GPU on which this library is loaded holds it until the process exits.  Host code
// cannot use the array's name as a device address (it is a host-side stand-in), so
// the device address is fetched with cudaGetSymbolAddress, on every call with the
// caller's device current, and passed to the kernels as their workspace.
#include <cuda_runtime.h>

#include "sdv_host.h"

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[SDV_NOALLOC_SCRATCH_BYTES];

// Device address of the scratch on the current device.  It is looked up on every call
// (a host-side lookup that allocates nothing): a cached address would go stale when
// the device's primary context is torn down (cudaDeviceReset) and the module is
// loaded again at another address.
cudaError_t noalloc_scratch(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  return cudaGetSymbolAddress(out, g_noalloc_scratch);
}

}  // namespace

extern "C" int sdv_verify_noalloc(const void* x_draft, const void* mu_target, const void* mu_draft,
                                  const float* sigma, int64_t sigma_stride_b, int B, int L,
                                  int64_t d, int dtype, uint64_t seed, int mode,
                                  int32_t* accepted_len, void* y_out, float* log_ratio_out,
                                  float* delta_norm_out, uint32_t* status_out,
                                  sdv_stream_t stream) {
  const size_t need = sdv_workspace_bytes(B, L, d, dtype);
  if (need == 0) return SDV_EINVAL;
  if (need > (size_t)SDV_NOALLOC_SCRATCH_BYTES) return SDV_ENOWORKSPACE;
  void* scratch = nullptr;
  if (noalloc_scratch(&scratch) != cudaSuccess) {
    // record the failure for sdv_last_cuda_error() and clear the runtime's last-error
    // slot, so that a later launch check does not report it again
    sdv::set_last_cuda_error((int)cudaGetLastError());
    return SDV_ECUDA;
  }
  // The tickets of the fused kernel, which must start at zero, are cleared by the call
  // itself (a memset on `stream`); k_tiles' partials carry the call's tag; everything
  // else in the workspace is written before it is read.
  return sdv_verify(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype, seed, mode,
                    accepted_len, y_out, log_ratio_out, delta_norm_out, status_out, scratch,
                    (size_t)SDV_NOALLOC_SCRATCH_BYTES, stream);
}
