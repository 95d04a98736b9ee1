// kdn_noalloc.cu -- a Diagonal-KDN forward for callers that cannot allocate.
//
// kdn_diag_fwd needs a scratch workspace that the caller allocates.  Some
// callers cannot do that: their interface hands them only input and output
// buffers, and they may not call cudaMalloc themselves -- for instance a
// latency-critical serving thread, where cudaMalloc can stall on an implicit
// device synchronisation, or a host framework that forbids any allocation
// outside its own allocator once it is running.  kdn_diag_fwd_noalloc serves
// them: its scratch is a fixed array in the library's own device memory, so
// the call itself allocates nothing.
//
// The array is a file-scope __device__ variable of KDN_NOALLOC_SCRATCH_BYTES.
// A GPU holds that memory from the first use of the library on it (CUDA loads
// the module lazily) until the process exits.  Host code cannot use the
// array's name as a device address, so the first call on each device looks
// the address up with cudaGetSymbolAddress (with that device current) and
// caches it together with the CUDA context it belongs to; a call under a
// different context (after a device reset, say) looks it up again.  Make that
// first call before any stream capture.  All calls on a device share the one
// array and it keeps the previous call's contents; nothing in it needs to
// start at zero (the forward writes every scratch element before reading it,
// and clears its status word itself), but calls whose executions overlap on
// the GPU -- on different streams, or from different host threads -- race on
// it and must be serialised by the caller.  The device status word of the
// last call (the first bytes of the array) is read and cleared by
// kdn_noalloc_device_status.
#include <cuda.h>

#include <mutex>

#include "kdn_internal.cuh"

namespace {

constexpr size_t kScratchBytes = KDN_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char kdn_noalloc_scratch[kScratchBytes];

std::mutex g_mutex;
void *g_scratch[kMaxDevices] = {};
CUcontext g_ctx[kMaxDevices] = {};

using CtxGetCurrent = CUresult (*)(CUcontext *);

// The current CUDA context (the driver's cuCtxGetCurrent, through the runtime's
// entry-point query so that the library needs no link-time driver dependency).
kdn_status_t current_context(CUcontext *ctx) {
  static CtxGetCurrent fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void *p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetCurrent>(p);
  });
  if (!fn || fn(ctx) != CUDA_SUCCESS) return KDN_ERR_CUDA;
  return KDN_OK;
}

// Device address of the scratch array on the current device (set-up on first
// use, and again whenever the device's context has changed).
kdn_status_t scratch_address(void **out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return KDN_ERR_CUDA;
  // cudaSetDevice makes the device's primary context current (initialising it if needed)
  if (cudaSetDevice(dev) != cudaSuccess) return KDN_ERR_CUDA;
  CUcontext ctx = nullptr;
  if (current_context(&ctx) != KDN_OK || !ctx) return KDN_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mutex);
  if (!g_scratch[dev] || g_ctx[dev] != ctx) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, kdn_noalloc_scratch) != cudaSuccess || !p) return KDN_ERR_CUDA;
    g_scratch[dev] = p;
    g_ctx[dev] = ctx;
  }
  *out = g_scratch[dev];
  return KDN_OK;
}

}  // namespace

extern "C" {

kdn_status_t kdn_diag_fwd_noalloc(const kdn_desc_t *desc, const void *q, const void *k,
                                  const void *v, const void *g, const void *omega,
                                  const void *r, const float *S0, const float *p0, void *o,
                                  float *ST, float *pT, void *stream) {
  // the single-pass layout must fit; the sequence-parallel buffers are used
  // when they fit as well (the regular entry point decides)
  const size_t need = kdn::fwd_min_workspace_bytes(desc, 0);
  if (need == 0)  // invalid descriptor: let the regular entry point name the error
    return kdn_diag_fwd(desc, q, k, v, g, omega, r, S0, p0, o, ST, pT, nullptr, 0, stream);
  if (need > kScratchBytes) return KDN_ERR_WORKSPACE;  // problem too large for the array
  void *ws = nullptr;
  kdn_status_t st = scratch_address(&ws);
  if (st != KDN_OK) return st;
  return kdn_diag_fwd(desc, q, k, v, g, omega, r, S0, p0, o, ST, pT, ws, kScratchBytes, stream);
}

kdn_status_t kdn_noalloc_device_status(void *stream) {
  void *ws = nullptr;
  kdn_status_t st = scratch_address(&ws);
  if (st != KDN_OK) return st;
  return kdn_get_device_status(ws, stream);
}

}  // extern "C"
