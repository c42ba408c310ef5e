// soma_launch.h -- host-side launchers shared by the translation units of
// libsoma (not part of the public ABI).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "soma_device.cuh"

namespace soma {

// Scratch of one forward sweep, carved out of the caller's workspace.
struct ForwardBuffers {
  int Tc;        // ring length of the h_t history
  float* hist;   // [lanes][Tc][B][H]
  float* cst;    // [lanes][B][H]
  float* nll;    // [lanes][B][T] per-target NLL
};

// Tracing hooks: bracket one kernel launch of class `kind` (SOMA_TRACE_*).
void trace_begin(int kind, cudaStream_t stream);
void trace_end(int kind, cudaStream_t stream);

int forward_hist_slots(const Sweep& s);
cudaError_t launch_forward_simt(const Sweep& s, const ForwardBuffers& fb, cudaStream_t stream);

// losses_out [pairs][n_sign]; coef_out / coef_ws [pairs] (either may be null).
cudaError_t launch_reduce_losses(const float* nll, int pairs, int n_sign, int B, int T, float eps,
                                 float* losses_out, float* coef_out, float* coef_ws, int* status,
                                 cudaStream_t stream);
cudaError_t launch_spsa_update(float* params, const Layout& lay, int n_experts, int n_pert,
                               float lr, uint64_t seed, uint64_t step, const float* coef,
                               cudaStream_t stream);
cudaError_t launch_init(float* params, const Layout& lay, int n_experts, uint64_t seed, float std,
                        cudaStream_t stream);
cudaError_t launch_debug_philox(uint64_t seed, const uint32_t* ctr4, uint32_t* out4, int count,
                                cudaStream_t stream);
cudaError_t launch_debug_rademacher(uint64_t seed, uint64_t step, int expert, int pert, int64_t p0,
                                    int64_t count, int8_t* z, cudaStream_t stream);

}  // namespace soma
