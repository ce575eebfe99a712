// static_ws.cu -- qwam_asp_linear_static: the layer with a scratch workspace that the library
// reserves statically in device memory, for callers that cannot hand it a device buffer (a C
// host without a device allocator, or a hot loop that must not allocate).  No allocation happens
// here or in the calls it makes.
#include <mutex>

#include "internal.h"

namespace {

// The scratch: one per device (a module-scope __device__ array exists once in every device
// context that loads this library).  Its size is the header's limit.
constexpr size_t kStaticWsBytes = QWAM_STATIC_WS_BYTES;
static __device__ __align__(256) unsigned char g_static_ws[kStaticWsBytes];

constexpr int kMaxDevices = 64;
std::mutex g_ws_mu;
void* g_ws_addr[kMaxDevices] = {};  // the scratch's device address, per device, once looked up

// Device address of the current device's scratch.  The first call per device asks the runtime
// for the symbol's address (with that device current) and keeps it.
qwam_status static_ws_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return QWAM_ERR_CUDA;
  }
  if (dev < 0 || dev >= kMaxDevices) return QWAM_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_ws_mu);
  if (!g_ws_addr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_static_ws);
    if (e != cudaSuccess || !p) {
      cudaGetLastError();
      return QWAM_ERR_CUDA;
    }
    g_ws_addr[dev] = p;
  }
  *out = g_ws_addr[dev];
  return QWAM_OK;
}

}  // namespace

qwam_status qwam_asp_linear_static(const void* X_bf16, int M, qwam_asp_handle h, void* Y, int y_dtype,
                                   struct CUstream_st* stream) {
  if (!h || M < 0) return QWAM_ERR_INVALID_ARG;
  // the layout without the per-call float16 weights: the GEMM expands them tile by tile
  const size_t need = qwam::act_layout(h->h, M, true).bytes;
  if (need > kStaticWsBytes) return QWAM_ERR_TOO_LARGE;
  void* ws = nullptr;
  const qwam_status sa = static_ws_address(&ws);
  if (sa != QWAM_OK) return sa;
  return qwam::linear_impl(X_bf16, M, h, Y, y_dtype, ws, stream, true);
}
