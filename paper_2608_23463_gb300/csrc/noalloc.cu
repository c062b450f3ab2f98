// Allocation-free variant of proxy_layer_bwd (see proxyformer.h).
//
// Some callers cannot hand the library a workspace: host frameworks whose
// memory planner owns every device byte and gives plugins no scratch, and
// latency-critical loops that cannot afford cudaMalloc's implicit device
// synchronisation.  For them the backward's scratch lives in the fixed
// file-scope device array below instead of a caller buffer.
#include <stdio.h>

#include <atomic>

#include "kernels.h"
#include "proxyformer.h"

pf_status pf_set_error(pf_status s, const char* msg);

namespace {

// Scratch of the allocation-free backward.  Every GPU that loads the library
// holds these PF_NOALLOC_SCRATCH_BYTES until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[PF_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
// Device address of the array per device, filled on a device's first call.
// Host threads may race on the first call: each looks the (same) address up
// and stores it; readers see either null (and look it up too) or the address.
std::atomic<void*> g_scratch_addr[kMaxDevices] = {};

thread_local char g_noalloc_msg[256];

}  // namespace

extern "C" pf_status proxy_layer_bwd_noalloc(const pf_layer_desc* desc,
                                             const pf_layer_params* params, const void* X,
                                             const float* H_in, const float* t, const void* saved,
                                             const void* dX_out, const float* dH_out, void* dX,
                                             float* dH_in, const pf_layer_grads* grads,
                                             void* stream) {
  pf_status st = proxy_layer_check(desc);
  if (st != PF_OK) return st;
  const size_t need = proxy_layer_workspace_size(desc, 1);
  if (need > (size_t)PF_NOALLOC_SCRATCH_BYTES) {
    snprintf(g_noalloc_msg, sizeof(g_noalloc_msg),
             "proxy_layer_bwd_noalloc: this layer needs %zu bytes of scratch, more than the "
             "fixed %zu bytes; use proxy_layer_bwd with a workspace",
             need, (size_t)PF_NOALLOC_SCRATCH_BYTES);
    return pf_set_error(PF_ERR_WORKSPACE, g_noalloc_msg);
  }
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return pf_set_error(PF_ERR_CUDA, "proxy_layer_bwd_noalloc: no usable current device");
  void* scratch = g_scratch_addr[dev].load(std::memory_order_acquire);
  if (scratch == nullptr) {
    // Host code must not use g_noalloc_scratch directly (on the host it is a
    // stand-in symbol, not a device address): look the device address up once
    // per device, with that device current.
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || p == nullptr) {
      snprintf(g_noalloc_msg, sizeof(g_noalloc_msg),
               "proxy_layer_bwd_noalloc: cudaGetSymbolAddress failed: %s", cudaGetErrorString(e));
      return pf_set_error(PF_ERR_CUDA, g_noalloc_msg);
    }
    g_scratch_addr[dev].store(p, std::memory_order_release);
    scratch = p;
  }
  return proxy_layer_bwd(desc, params, X, H_in, t, saved, dX_out, dH_out, dX, dH_in, grads,
                         scratch, (size_t)PF_NOALLOC_SCRATCH_BYTES, stream);
}
