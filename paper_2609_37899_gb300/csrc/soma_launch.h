// soma_launch.h -- host-side launchers shared by the translation units of
// libsoma (not part of the public ABI).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "soma_api.h"
#include "soma_device.cuh"

namespace soma {

// Tracing hooks: bracket one kernel launch of class `kind` (SOMA_TRACE_*).
void trace_begin(int kind, cudaStream_t stream);
void trace_end(int kind, cudaStream_t stream);


// ---- tensor-core path ------------------------------------------------------
// Geometry of one sweep on the tensor cores.  K of the gate GEMM is
// [x part padded to Ep | h part padded to Hp], in stages of 64; rows are
// 32-unit tiles of 4 gates; sequences are padded to Bp and P <= 2 probes
// share one operand group tile of rowsB = 3 Bp P rows (vbar, dhat and
// eps^2 dhat per probe, forward_tc.cu).
//
// The unperturbed layout (inf = 1: evaluation and routed inference, eps = 0,
// one sign) uses the same tile shape, but the four row blocks that the W
// product reads hold four blocks of Bp = 32 different sequences, so a group
// is 128 sequences and every MMA column does useful work; G groups cover
// the whole batch in one sweep.
struct TcGeom {
  int E, H, Ep, Hp, S, Sx, Sh, MT, Bp, P, G, rowsB;
  uint32_t tileB;  // bytes of one operand group tile of one stage
  int n_experts, n_pert, B, T;
  int Bm;          // sequences of the whole batch (the loss partials); B <= 64 of them per sweep
  int inf;         // the unperturbed layout
};

// Sequences of one group of the unperturbed layout.
constexpr int kInfGroupSeqs = 128;

struct TcSizes {
  size_t w16, wo16, op, cst, pm, ply, zb, cnt, xall;
};

struct TcBuffers {
  uint8_t* w16;    // gate weight tiles, fp16
  uint8_t* wo16;   // head weight tiles, fp16
  uint8_t* op[2];  // operands of timesteps t and t + 1
  float* cst;      // cell state, fp32 per sign
  float* pm;       // head partial max
  float* ps;       // head partial sum-exp
  float* ply;      // target logits
  uint2* zbits;    // probe-word table of the sweep
  int* cnt;        // phase counters of the persistent kernel
  uint8_t* xall;   // embedding part of the operand of every timestep of the sweep
};

TcGeom make_tc_geom(const Layout& lay, int n_experts, int n_pert, int B, int T, int B_mem);
// The unperturbed layout for B sequences per expert (all in one sweep).
TcGeom make_tc_geom_inf(const Layout& lay, int n_experts, int B, int T);
// Sequences of one tensor-core sweep; a larger batch runs in chunks of this many.
constexpr int kTcMaxBatch = 64;
TcSizes tc_sizes(const TcGeom& g);
cudaError_t launch_forward_tc(const Sweep& s, const TcGeom& g, const TcBuffers& tb, int* status,
                              cudaStream_t stream);
cudaError_t launch_reduce_tc(const TcBuffers& tb, int pairs, int n_sign, int B, int T, float eps,
                             float* losses_out, float* coef_out, float* coef_ws, int* status,
                             cudaStream_t stream);
cudaError_t launch_debug_tc_gemm(const void* A, const void* B, float* D, int N, int K,
                                 int a_in_tmem, int* status, cudaStream_t stream);

cudaError_t launch_spsa_update(float* params, const Layout& lay, int n_experts, int n_pert,
                               float lr, uint64_t seed, uint64_t step, const float* coef,
                               cudaStream_t stream);
// The update under a probe law (probe_law.cuh): sparse probes are dense from
// coordinate dense_from on (the LSTM expert passes P).
cudaError_t launch_sgd_update(float* params, int64_t P, int64_t dense_from, int n_experts,
                              int n_pert, int sparse, float lr, uint64_t seed, uint64_t step,
                              const float* coef, cudaStream_t stream);
cudaError_t launch_init(float* params, const Layout& lay, int n_experts, uint64_t seed, float std,
                        cudaStream_t stream);
cudaError_t launch_debug_wait_timeout(uint32_t max_polls, int* status, cudaStream_t stream);
cudaError_t launch_debug_check_fail(int* status, cudaStream_t stream);
cudaError_t launch_debug_philox(uint64_t seed, const uint32_t* ctr4, uint32_t* out4, int count,
                                cudaStream_t stream);
cudaError_t launch_debug_rademacher(uint64_t seed, uint64_t step, int expert, int pert, int sparse,
                                    int64_t p0, int64_t count, int8_t* z, cudaStream_t stream);

// Probe step counters of the accumulation batches of one Adam update.
struct AdamSteps {
  int n_acc;
  uint64_t step[SOMA_MAX_ACCUM];
};

// Adam hyper-parameters with the bias corrections of update t folded in:
// inv_bc1 = 1 / (1 - b1^t), inv_bc2 = 1 / (1 - b2^t).
struct AdamArgs {
  float lr, b1, b2, delta, wd, inv_bc1, inv_bc2;
};

// Small experts with the whole recurrence resident in one CTA (resident.cu).
bool res_supported(const Layout& lay, int B);
// n_sign = 2: losses_out [N][n][2] (L+, L-) and the coefficients; n_sign = 1
// (eps = 0, n = 1): losses_out [N] = L(theta).
cudaError_t launch_forward_res(const Sweep& s, int n_sign, float* losses_out, float* coef_out,
                               float* coef_ws, int* status, cudaStream_t stream);

// Routed inference (mixture.cu).
cudaError_t launch_gather_requests(const uint8_t* requests, const int32_t* gather, int N,
                                   int b_max, int b0, int Bc, int T1, uint8_t* grouped,
                                   cudaStream_t stream);
cudaError_t launch_token_nll_tc(const TcBuffers& tb, int N, int Bc, int T, int b_max, int b0,
                                float* nll, cudaStream_t stream);
cudaError_t launch_mixture(const float* nll, const int32_t* route, const int32_t* slot, int R,
                           int k, int T, int t0, int b_max, float* out, cudaStream_t stream);
cudaError_t launch_sum_over_experts(float* coef, int n_experts, int n_pert, cudaStream_t stream);
cudaError_t launch_adam_update(float* params, float* m, float* v, const Layout& lay, int n_experts,
                               int n_pert, int sparse, uint64_t seed, const AdamSteps& steps,
                               const float* coef, const AdamArgs& h, cudaStream_t stream);
cudaError_t launch_probe_adam(float* params, float* m, float* v, int64_t P, int64_t dense_from,
                              int n_experts, int n_pert, int sparse, uint64_t seed,
                              const AdamSteps& steps, const float* coef, const AdamArgs& h,
                              cudaStream_t stream);

// The paper's expert body (body.cu, body_tc.cu): width kBodyWidth, 1 <=
// blocks <= kBodyMaxBlocks.  partial [N * n * n_sign][ceil(B / 16)] fp64 NLL sums.
int body_rows_per_cta();
// The antithetic forwards on the tensor cores (body_tc.cu): one CTA per
// (expert, probe) pair and 16-sequence chunk, both signs in the
// mean/difference form.
cudaError_t launch_body_tc(const float* params, const float* head, const uint8_t* bytes,
                           int n_experts, int blocks, int n_pert, int n_sign, int B, int T,
                           float eps, int sparse, uint64_t seed, uint64_t step, double* partial,
                           int* status, cudaStream_t stream);
cudaError_t launch_body_reduce(const double* partial, int pairs, int n_sign, int B, int T,
                               float eps, float* losses_out, float* coef_out, float* coef_ws,
                               int* status, cudaStream_t stream);
cudaError_t launch_body_sgd(float* params, int n_experts, int blocks, int n_pert, int sparse,
                            float lr, uint64_t seed, uint64_t step, const float* coef,
                            cudaStream_t stream);
cudaError_t launch_body_adam(float* params, float* m, float* v, int n_experts, int blocks,
                             int n_pert, int sparse, uint64_t seed, const AdamSteps& steps,
                             const float* coef, const AdamArgs& h, cudaStream_t stream);
cudaError_t launch_debug_body_probe(uint64_t seed, uint64_t step, int expert, int pert, int blocks,
                                    int sparse, int64_t p0, int64_t count, int8_t* z,
                                    cudaStream_t stream);

}  // namespace soma
