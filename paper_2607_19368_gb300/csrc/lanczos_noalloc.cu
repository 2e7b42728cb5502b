// sls_lanczos_topr_noalloc: the Lanczos top-r call for callers that may not
// allocate device memory.  Its scratch is one file-scope device array; the
// host looks up that array's device address once per device and hands it to
// the ordinary workspace path as the workspace.
#include <mutex>

#include "common.cuh"
#include "kernels.cuh"

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[SLS_NOALLOC_MAX_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_lock;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_noalloc_scratch on the current device.  In host code
// the array's name is only a stand-in for the symbol, never a device pointer.
// The address is looked up once per device and cached for the process; a
// cudaDeviceReset() destroys the context that holds the array, after which
// the cached address is stale (the header says so).
int scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return SLS_ERR_CUDA;
  std::lock_guard<std::mutex> guard(g_lock);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr)
      return SLS_ERR_CUDA;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return SLS_OK;
}

}  // namespace

extern "C" int sls_lanczos_topr_noalloc(const float* Phi, int64_t N, int D, int r,
                                        const double* q1, double tol, double* theta, float* U,
                                        int32_t* r_eff, double* alpha, double* beta,
                                        void* stream) {
  if (N < 1 || D < 4 || D > SLS_MAX_D || r < 1 || r > SLS_MAX_R || !(tol >= 0.0))
    return SLS_ERR_INVALID_ARG;
  if ((D & 3) != 0) return SLS_ERR_UNSUPPORTED;
  // the same pointer checks as sls_lanczos_topr, before anything is enqueued
  if (Phi == nullptr || ((uintptr_t)Phi & 15u) != 0 || !q1 || !theta || !U || !r_eff)
    return SLS_ERR_INVALID_ARG;
  const size_t need = sls_lanczos_workspace_size(N, D, r);
  if (need == 0) return SLS_ERR_UNSUPPORTED;
  if (need > (size_t)SLS_NOALLOC_MAX_BYTES) return SLS_ERR_WORKSPACE;
  void* ws = nullptr;
  const int st = scratch_address(&ws);
  if (st != SLS_OK) return st;
  return sls_lanczos_topr(Phi, N, D, r, q1, tol, theta, U, r_eff, alpha, beta, ws,
                          (size_t)SLS_NOALLOC_MAX_BYTES, stream);
}
