// body.cu -- the paper's expert body (Sec. "Model size"; loss and probes of
// App. E): D pre-norm residual blocks of width d, each a bias-free LSTM and a
// bias-free GELU MLP of width 4d, gain-only LayerNorm, and one frozen tied
// head E [V][d] that embeds the byte and decodes the final normalised state
// (logits = E y).  Only the body is perturbed.  The antithetic forwards run
// in body_tc.cu; this file holds the rest of the step.
//
// Kernels: body_reduce_kernel (L+-, the coefficients (L+ - L-) / (2 eps) in
// fp64) and the probe debug kernel; the SGD and Adam updates are the LSTM
// expert's (spsa_misc.cu) under the body's probe law.
//
// Probe law (App. E): normalisation gains take the dense sign; every other
// coordinate is the dense sign where the activity stream's bit is set, else
// 0 (the sparse probe).  With dense probes every coordinate takes the sign.
#include <cstdint>
#include <cuda_runtime.h>

#include "body_device.cuh"
#include "soma_device.cuh"
#include "soma_launch.h"

namespace soma {
namespace {

constexpr int kD = kBodyWidth;
constexpr int kRows = kBodyRows;

// L[pair][s] = sum over chunks / (B T); coef = (L+ - L-) / (2 eps).
__global__ void body_reduce_kernel(const double* __restrict__ partial, int pairs, int n_sign,
                                   int chunks, int BT, float eps, float* losses_out,
                                   float* coef_out, float* coef_ws, int* status) {
  const int pair = blockIdx.x * blockDim.x + threadIdx.x;
  if (pair >= pairs) return;
  double L[2] = {0.0, 0.0};
  for (int s = 0; s < n_sign; ++s) {
    const double* p = partial + ((int64_t)pair * n_sign + s) * chunks;
    double acc = 0.0;
    for (int c = 0; c < chunks; ++c) acc += p[c];
    L[s] = acc / (double)BT;
  }
  bool finite = isfinite(L[0]);
  if (losses_out) losses_out[(int64_t)pair * n_sign] = (float)L[0];
  if (n_sign == 2) {
    const double c = (eps == 0.f) ? 0.0 : (L[0] - L[1]) / (2.0 * (double)eps);
    finite = finite && isfinite(L[1]) && isfinite(c);
    if (losses_out) losses_out[(int64_t)pair * 2 + 1] = (float)L[1];
    if (coef_out) coef_out[pair] = (float)c;
    if (coef_ws) coef_ws[pair] = (float)c;
  }
  if (!finite && status) atomicCAS(status, 0, kStatusNonFinite);
}

// z[p - p0] for p in [p0, p0 + count): thread w handles run (p0 >> 5) + w.
__global__ void debug_body_probe_kernel(ProbeKey pk, int sparse, int64_t goff, int64_t p0,
                                        int64_t count, int8_t* z) {
  const int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t q = (p0 >> 5) + w;
  if (q * 32 >= p0 + count) return;
  uint32_t neg, act;
  body_probe_words(pk, (int)q, sparse, goff, neg, act);
  for (int j = 0; j < 32; ++j) {
    const int64_t p = q * 32 + j;
    if (p < p0 || p >= p0 + count) continue;
    z[p - p0] = ((act >> j) & 1u) ? (((neg >> j) & 1u) ? -1 : 1) : 0;
  }
}

}  // namespace

int body_rows_per_cta() { return kRows; }

cudaError_t launch_body_reduce(const double* partial, int pairs, int n_sign, int B, int T,
                               float eps, float* losses_out, float* coef_out, float* coef_ws,
                               int* status, cudaStream_t stream) {
  const int chunks = (B + kRows - 1) / kRows;
  trace_begin(SOMA_TRACE_REDUCE, stream);
  body_reduce_kernel<<<(pairs + 127) / 128, 128, 0, stream>>>(partial, pairs, n_sign, chunks,
                                                              B * T, eps, losses_out, coef_out,
                                                              coef_ws, status);
  trace_end(SOMA_TRACE_REDUCE, stream);
  return cudaGetLastError();
}

cudaError_t launch_body_sgd(float* params, int n_experts, int blocks, int n_pert, int sparse,
                            float lr, uint64_t seed, uint64_t step, const float* coef,
                            cudaStream_t stream) {
  return launch_sgd_update(params, body_param_count(kD, blocks), body_gain_offset(kD, blocks),
                           n_experts, n_pert, sparse, lr, seed, step, coef, stream);
}

cudaError_t launch_body_adam(float* params, float* m, float* v, int n_experts, int blocks,
                             int n_pert, int sparse, uint64_t seed, const AdamSteps& steps,
                             const float* coef, const AdamArgs& h, cudaStream_t stream) {
  return launch_probe_adam(params, m, v, body_param_count(kD, blocks),
                           body_gain_offset(kD, blocks), n_experts, n_pert, sparse, seed, steps,
                           coef, h, stream);
}

cudaError_t launch_debug_body_probe(uint64_t seed, uint64_t step, int expert, int pert, int blocks,
                                    int sparse, int64_t p0, int64_t count, int8_t* z,
                                    cudaStream_t stream) {
  const ProbeKey pk = make_probe_key(seed, step, (uint32_t)expert, (uint32_t)pert);
  const int64_t runs = ((p0 + count + 31) >> 5) - (p0 >> 5);
  debug_body_probe_kernel<<<(unsigned)((runs + 127) / 128), 128, 0, stream>>>(
      pk, sparse, body_gain_offset(kD, blocks), p0, count, z);
  return cudaGetLastError();
}

}  // namespace soma
