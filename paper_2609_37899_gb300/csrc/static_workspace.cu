// static_workspace.cu -- soma_spsa_step_static: the SPSA step for callers
// that cannot allocate device memory.
//
// Some callers of this library cannot call cudaMalloc: a host runtime that
// only hands over buffers it was given (a plugin or an embedded interpreter
// with no device allocator of its own), or a control loop that must not risk
// an allocation that blocks or fails in the middle of training.  For them the
// scratch memory lives in a fixed array in this file, reserved when the
// library is loaded on a device and held until the process exits.  The
// caller still passes the parameters, the bytes and the output buffers.
#include <cstdint>

#include "soma_api.h"

namespace {

constexpr size_t kStaticBytes = SOMA_STATIC_WORKSPACE_BYTES;

// The scratch array.  In host code this name is only a host-side stand-in
// for the device symbol: its device address comes from
// cudaGetSymbolAddress, once per device.
static __device__ __align__(256) unsigned char g_static_workspace[kStaticBytes];

constexpr int kMaxDevices = 64;
void* g_static_ptr[kMaxDevices] = {nullptr};

// Device address of the array on the current device (set up on the first
// call made with that device current).
int static_workspace(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return SOMA_ERR_CUDA;
  if (!g_static_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_workspace) != cudaSuccess || !p) return SOMA_ERR_CUDA;
    g_static_ptr[dev] = p;
  }
  *out = g_static_ptr[dev];
  return SOMA_OK;
}

}  // namespace

extern "C" int soma_spsa_step_static(float* params, int n_experts, soma_dims d, int n_pert,
                                     float eps, float lr, uint64_t seed, uint64_t step,
                                     const uint8_t* byte_batch, int batch, int seq_len,
                                     float* losses_out, float* coef_out, void* stream) {
  if (soma_param_count(d) < 0) return SOMA_ERR_UNSUPPORTED;
  const size_t need = soma_workspace_bytes(d, n_experts, n_pert, batch, seq_len);
  if (need == 0) return SOMA_ERR_INVALID_ARG;
  if (need > kStaticBytes) return SOMA_ERR_WORKSPACE;
  void* ws = nullptr;
  const int rc = static_workspace(&ws);
  if (rc != SOMA_OK) return rc;
  return soma_spsa_step(params, n_experts, d, n_pert, eps, lr, seed, step, byte_batch, batch,
                        seq_len, losses_out, coef_out, ws, kStaticBytes, stream);
}
