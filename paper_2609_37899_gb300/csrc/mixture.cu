// mixture.cu -- routed inference (Sec. 3, Eq. main-mixture): requests grouped
// by expert, each expert's unperturbed forward on its group, and the average
// of the routed experts' probabilities of every target byte.
#include "soma_api.h"
#include "soma_launch.h"

namespace soma {

namespace {

// grouped[e][b][:] = requests[gather[e][b0 + b]][:], zeros for an empty slot.
// grid (N * Bc), block 128: one block per (expert, slot) row.
__global__ void gather_requests_kernel(const uint8_t* __restrict__ requests,
                                       const int32_t* __restrict__ gather, int b_max, int b0,
                                       int Bc, int T1, uint8_t* __restrict__ grouped) {
  const int e = blockIdx.x / Bc, b = blockIdx.x % Bc;
  const int slot = b0 + b;
  const int r = slot < b_max ? gather[(int64_t)e * b_max + slot] : -1;
  uint8_t* dst = grouped + ((int64_t)e * Bc + b) * T1;
  for (int t = threadIdx.x; t < T1; t += blockDim.x)
    dst[t] = r >= 0 ? requests[(int64_t)r * T1 + t] : (uint8_t)0;
}

// Per-target NLL of the tensor path's partials (the + lane of probe 0 of
// every expert): nll[e][b0 + b][t] = logsumexp of the two vocabulary halves
// minus the target logit.  pm, ps: [lanes][Bc][T][2], ply: [lanes][Bc][T].
__global__ void token_nll_tc_kernel(const float* __restrict__ pm, const float* __restrict__ ps,
                                    const float* __restrict__ ply, int N, int Bc, int T,
                                    int b_max, int b0, float* __restrict__ nll) {
  const int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;  // over N * Bc * T
  if (j >= (int64_t)N * Bc * T) return;
  const int t = (int)(j % T);
  const int b = (int)((j / T) % Bc);
  const int e = (int)(j / ((int64_t)T * Bc));
  if (b0 + b >= b_max) return;
  const int64_t ln = (int64_t)e * 2;  // lanes (e, probe 0, sign +)
  const int64_t k = (ln * Bc + b) * T + t;
  const float m0 = pm[2 * k], m1 = pm[2 * k + 1];
  const float M = fmaxf(m0, m1);
  const float v = M + logf(ps[2 * k] * expf(m0 - M) + ps[2 * k + 1] * expf(m1 - M)) - ply[k];
  nll[((int64_t)e * b_max + b0 + b) * T + t] = v;
}

// out[r][t - t0] = log k - logsumexp_j(-nll[e_j][slot_j][t]): the NLL of the
// average of the k routed experts' probabilities of the target.
__global__ void mixture_kernel(const float* __restrict__ nll, const int32_t* __restrict__ route,
                               const int32_t* __restrict__ slot, int R, int k, int T, int t0,
                               int b_max, float* __restrict__ out) {
  const int Ts = T - t0;
  const int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= (int64_t)R * Ts) return;
  const int r = (int)(j / Ts), t = t0 + (int)(j % Ts);
  float mx = -INFINITY;
  for (int q = 0; q < k; ++q) {
    const int e = route[(int64_t)r * k + q], s = slot[(int64_t)r * k + q];
    mx = fmaxf(mx, -nll[((int64_t)e * b_max + s) * T + t]);
  }
  float acc = 0.f;
  for (int q = 0; q < k; ++q) {
    const int e = route[(int64_t)r * k + q], s = slot[(int64_t)r * k + q];
    acc += expf(-nll[((int64_t)e * b_max + s) * T + t] - mx);
  }
  out[j] = logf((float)k) - (mx + logf(acc));
}

}  // namespace

cudaError_t launch_gather_requests(const uint8_t* requests, const int32_t* gather, int N,
                                   int b_max, int b0, int Bc, int T1, uint8_t* grouped,
                                   cudaStream_t stream) {
  gather_requests_kernel<<<N * Bc, 128, 0, stream>>>(requests, gather, b_max, b0, Bc, T1, grouped);
  return cudaGetLastError();
}

cudaError_t launch_token_nll_tc(const TcBuffers& tb, int N, int Bc, int T, int b_max, int b0,
                                float* nll, cudaStream_t stream) {
  const int64_t n = (int64_t)N * Bc * T;
  token_nll_tc_kernel<<<(unsigned)((n + 255) / 256), 256, 0, stream>>>(tb.pm, tb.ps, tb.ply, N, Bc,
                                                                       T, b_max, b0, nll);
  return cudaGetLastError();
}

cudaError_t launch_mixture(const float* nll, const int32_t* route, const int32_t* slot, int R,
                           int k, int T, int t0, int b_max, float* out, cudaStream_t stream) {
  const int64_t n = (int64_t)R * (T - t0);
  mixture_kernel<<<(unsigned)((n + 255) / 256), 256, 0, stream>>>(nll, route, slot, R, k, T, t0,
                                                                  b_max, out);
  return cudaGetLastError();
}

}  // namespace soma
