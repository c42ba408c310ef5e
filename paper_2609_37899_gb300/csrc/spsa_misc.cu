// spsa_misc.cu -- the loss reduction, the SPSA update, the parameter
// initialisation and the generator test kernels.
#include "soma_api.h"
#include "probe_law.cuh"
#include "soma_launch.h"
#include "tc_primitives.cuh"

namespace soma {

namespace {

constexpr int kRedThreads = 256;

// One block per (expert, probe) pair: L+, L- = mean NLL of each sign (fp64
// sums in a fixed order), the pairwise mean D = mean(nll+ - nll-) and the
// coefficient D / (2 eps) (Eq. main-spsa).  nll: [pairs][n_sign][B*T].
__global__ void __launch_bounds__(kRedThreads)
reduce_losses_kernel(const float* __restrict__ nll, int n_sign, int BT, float eps,
                     float* losses_out, float* coef_out, float* coef_ws, int* status) {
  __shared__ double red[3][kRedThreads];
  const int pair = blockIdx.x;
  const float* np = nll + (int64_t)pair * n_sign * BT;
  double sp = 0.0, sm = 0.0, sd = 0.0;
  for (int j = threadIdx.x; j < BT; j += kRedThreads) {
    const float a = np[j];
    sp += (double)a;
    if (n_sign == 2) {
      const float b = np[BT + j];
      sm += (double)b;
      sd += (double)a - (double)b;  // exact in fp64 for any two fp32 values
    }
  }
  red[0][threadIdx.x] = sp;
  red[1][threadIdx.x] = sm;
  red[2][threadIdx.x] = sd;
  __syncthreads();
  for (int w = kRedThreads / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) {
      red[0][threadIdx.x] += red[0][threadIdx.x + w];
      red[1][threadIdx.x] += red[1][threadIdx.x + w];
      red[2][threadIdx.x] += red[2][threadIdx.x + w];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const double inv = 1.0 / (double)BT;
    const double Lp = red[0][0] * inv;
    bool finite = isfinite(Lp);
    if (losses_out) losses_out[(int64_t)pair * n_sign] = (float)Lp;
    if (n_sign == 2) {
      const double Lm = red[1][0] * inv;
      const double D = red[2][0] * inv;
      const double c = (eps == 0.f) ? 0.0 : D / (2.0 * (double)eps);
      finite = finite && isfinite(Lm) && isfinite(c);
      if (losses_out) losses_out[(int64_t)pair * 2 + 1] = (float)Lm;
      if (coef_out) coef_out[pair] = (float)c;
      if (coef_ws) coef_ws[pair] = (float)c;
    }
    if (!finite && status) atomicCAS(status, 0, kStatusNonFinite);
  }
}

constexpr int kUpdThreads = 128;

// theta[e][p] -= lr * (1/n) * sum_i coef[e][i] z_{e,i}[p] (Eq. main-spsa).
// Thread q of expert e owns the 32 parameters 32q .. 32q + 31, whose probe
// bits are one Philox word per probe (two for sparse probes), under the probe
// law of probe_law_words.  An expert whose coefficients are not all finite is
// left unchanged.
__global__ void __launch_bounds__(kUpdThreads)
sgd_update_kernel(float* __restrict__ params, int64_t P, int64_t dense_from, int n_pert,
                  int sparse, float lr, uint64_t seed, uint64_t step,
                  const float* __restrict__ coef) {
  extern __shared__ float cf[];  // [n_pert]
  __shared__ int all_finite;
  const int e = blockIdx.y;
  if (threadIdx.x == 0) all_finite = 1;
  __syncthreads();
  for (int i = threadIdx.x; i < n_pert; i += kUpdThreads) {
    const float c = coef[(int64_t)e * n_pert + i];
    cf[i] = c;
    if (!isfinite(c)) all_finite = 0;
  }
  __syncthreads();
  if (!all_finite) return;
  const int64_t q = (int64_t)blockIdx.x * kUpdThreads + threadIdx.x;
  const int64_t p0 = q * 32;
  if (p0 >= P) return;
  float acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0.f;
  for (int i = 0; i < n_pert; ++i) {
    uint32_t neg, act;
    probe_law_words(make_probe_key(seed, step, (uint32_t)e, (uint32_t)i), (int)q, sparse,
                    dense_from, neg, act);
    const float c = cf[i];
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if ((act >> j) & 1u) acc[j] += ((neg >> j) & 1u) ? -c : c;
  }
  const float scale = lr / (float)n_pert;
  float* th = params + (int64_t)e * P + p0;
  if (p0 + 32 <= P && (P & 3) == 0) {
    // P a multiple of 4 and p0 of 32: 16-byte aligned
#pragma unroll
    for (int j4 = 0; j4 < 8; ++j4) {
      float4 v = reinterpret_cast<float4*>(th)[j4];
      v.x -= scale * acc[4 * j4 + 0];
      v.y -= scale * acc[4 * j4 + 1];
      v.z -= scale * acc[4 * j4 + 2];
      v.w -= scale * acc[4 * j4 + 3];
      reinterpret_cast<float4*>(th)[j4] = v;
    }
  } else {
    for (int j = 0; j < 32 && p0 + j < P; ++j) th[j] -= scale * acc[j];
  }
}

// The paper's optimizer step (App. E, Eq. localspsa) for expert e:
//   g = (1/(A n)) sum_a sum_i coef[a][e][i] z_{e,i}^{(a)} + wd * theta,
//   m = b1 m + (1 - b1) g,  v = b2 v + (1 - b2) g^2,
//   theta -= lr * (m / bc1) / (sqrt(v / bc2) + delta),
// with z^{(a)} drawn with step counter steps[a] under the probe law of
// probe_law_words.  Thread q owns the 32 parameters 32q .. 32q + 31.  An
// expert whose coefficients are not all finite is left unchanged, moments
// included.
__global__ void __launch_bounds__(kUpdThreads)
adam_update_kernel(float* __restrict__ params, float* __restrict__ m, float* __restrict__ v,
                   int64_t P, int64_t dense_from, int n_experts, int n_pert, int sparse,
                   uint64_t seed, AdamSteps steps, const float* __restrict__ coef, AdamArgs h) {
  __shared__ int all_finite;
  const int e = blockIdx.y;
  if (threadIdx.x == 0) all_finite = 1;
  __syncthreads();
  for (int j = threadIdx.x; j < steps.n_acc * n_pert; j += kUpdThreads) {
    const int a = j / n_pert, i = j % n_pert;
    if (!isfinite(coef[((int64_t)a * n_experts + e) * n_pert + i])) all_finite = 0;
  }
  __syncthreads();
  if (!all_finite) return;
  const int64_t q = (int64_t)blockIdx.x * kUpdThreads + threadIdx.x;
  const int64_t p0 = q * 32;
  if (p0 >= P) return;
  float acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0.f;
  for (int a = 0; a < steps.n_acc; ++a) {
    const float* ca = coef + ((int64_t)a * n_experts + e) * n_pert;
    for (int i = 0; i < n_pert; ++i) {
      uint32_t neg, act;
      probe_law_words(make_probe_key(seed, steps.step[a], (uint32_t)e, (uint32_t)i), (int)q,
                      sparse, dense_from, neg, act);
      const float c = ca[i];
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if ((act >> j) & 1u) acc[j] += ((neg >> j) & 1u) ? -c : c;
    }
  }
  const float inv = 1.f / ((float)steps.n_acc * (float)n_pert);
  const int64_t base = (int64_t)e * P + p0;
  const int cnt = P - p0 < 32 ? (int)(P - p0) : 32;
  for (int j = 0; j < cnt; ++j) {
    const float th = params[base + j];
    const float g = fmaf(h.wd, th, acc[j] * inv);
    const float mj = fmaf(h.b1, m[base + j], (1.f - h.b1) * g);
    const float vj = fmaf(h.b2, v[base + j], (1.f - h.b2) * g * g);
    m[base + j] = mj;
    v[base + j] = vj;
    params[base + j] = th - h.lr * (mj * h.inv_bc1) / (sqrtf(vj * h.inv_bc2) + h.delta);
  }
}

// The summed-loss control arm (App. D): the N experts' losses are summed
// before each finite difference, so every expert's coefficient of probe i is
// sum_e (L+_{e,i} - L-_{e,i}) / (2 eps) = sum_e c_{e,i}.  One thread per
// probe, experts summed in order in fp64.
__global__ void sum_over_experts_kernel(float* coef, int n_experts, int n_pert) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n_pert) return;
  double acc = 0.0;
  for (int e = 0; e < n_experts; ++e) acc += (double)coef[(int64_t)e * n_pert + i];
  for (int e = 0; e < n_experts; ++e) coef[(int64_t)e * n_pert + i] = (float)acc;
}

// Box-Muller normals from Philox4x32-10 in the init domain (counter word 3
// = 0x80000001): parameters 2q and 2q+1 of expert e use counter (q, e, 0, .).
__global__ void init_kernel(float* __restrict__ params, Layout lay, uint64_t seed, float std) {
  const int e = blockIdx.y;
  const int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t p = 2 * q;
  if (p >= lay.P) return;
  const uint4 w = philox4x32_10(make_uint4((uint32_t)q, (uint32_t)e, 0u, 0x80000001u),
                                (uint32_t)(seed & 0xffffffffu), (uint32_t)(seed >> 32));
  const float u1 = (float)((w.x >> 8) + 1u) * (1.0f / 16777216.0f);  // (0, 1]
  const float u2 = (float)(w.y >> 8) * (1.0f / 16777216.0f);         // [0, 1)
  const float r = sqrtf(-2.0f * logf(u1));
  float nv[2] = {r * cospif(2.0f * u2), r * sinpif(2.0f * u2)};
  for (int j = 0; j < 2; ++j) {
    const int64_t pp = p + j;
    if (pp >= lay.P) break;
    float sd;
    if (std > 0.f) {
      sd = std;
    } else if (pp < lay.w_ih) {
      sd = 0.1f;
    } else if (pp < lay.b) {
      sd = rsqrtf((float)(lay.E + lay.H));
    } else if (pp < lay.w_out) {
      sd = 0.f;
    } else if (pp < lay.b_out) {
      sd = rsqrtf((float)lay.H);
    } else {
      sd = 0.f;
    }
    params[(int64_t)e * lay.P + pp] = sd * nv[j];
  }
}

__global__ void debug_philox_kernel(uint64_t seed, const uint32_t* ctr4, uint32_t* out4,
                                    int count) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= count) return;
  const uint4 c = make_uint4(ctr4[4 * j], ctr4[4 * j + 1], ctr4[4 * j + 2], ctr4[4 * j + 3]);
  const uint4 o = philox4x32_10(c, (uint32_t)(seed & 0xffffffffu), (uint32_t)(seed >> 32));
  out4[4 * j] = o.x;
  out4[4 * j + 1] = o.y;
  out4[4 * j + 2] = o.z;
  out4[4 * j + 3] = o.w;
}

// z[q] for p = p0 + q, through probe_bits at an arbitrary (unaligned) start
// so that the two-block path of the helper is exercised as well.
__global__ void debug_rademacher_kernel(ProbeKey pk, int sparse, int64_t p0, int64_t count,
                                        int8_t* z) {
  const int64_t q0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * 32;
  if (q0 >= count) return;
  const ProbeBits bits = probe_bits(pk, p0 + q0, sparse != 0);
  for (int j = 0; j < 32 && q0 + j < count; ++j)
    z[q0 + j] = ((bits.act >> j) & 1u) ? (((bits.neg >> j) & 1u) ? -1 : 1) : 0;
}


// A wait that nothing completes.  The bounded wait gives up after max_polls
// polls and the kernel records SOMA_ERR_TIMEOUT, as every kernel of the
// library does when one of its waits runs out; the context stays usable.
__global__ void debug_wait_timeout_kernel(uint32_t max_polls, int* status) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar, 1);
    tc::mbar_fence_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && !tc::mbar_wait(&bar, 0u, max_polls))
    atomicCAS(status, 0, kStatusTimeout);
}
}  // namespace

cudaError_t launch_reduce_losses(const float* nll, int pairs, int n_sign, int B, int T, float eps,
                                 float* losses_out, float* coef_out, float* coef_ws, int* status,
                                 cudaStream_t stream) {
  trace_begin(SOMA_TRACE_REDUCE, stream);
  reduce_losses_kernel<<<pairs, kRedThreads, 0, stream>>>(nll, n_sign, B * T, eps, losses_out,
                                                          coef_out, coef_ws, status);
  trace_end(SOMA_TRACE_REDUCE, stream);
  return cudaGetLastError();
}

cudaError_t launch_sgd_update(float* params, int64_t P, int64_t dense_from, int n_experts,
                              int n_pert, int sparse, float lr, uint64_t seed, uint64_t step,
                              const float* coef, cudaStream_t stream) {
  const int64_t words = (P + 31) / 32;
  dim3 grid((unsigned)((words + kUpdThreads - 1) / kUpdThreads), n_experts);
  trace_begin(SOMA_TRACE_UPDATE, stream);
  sgd_update_kernel<<<grid, kUpdThreads, n_pert * sizeof(float), stream>>>(
      params, P, dense_from, n_pert, sparse, lr, seed, step, coef);
  trace_end(SOMA_TRACE_UPDATE, stream);
  return cudaGetLastError();
}

cudaError_t launch_spsa_update(float* params, const Layout& lay, int n_experts, int n_pert,
                               float lr, uint64_t seed, uint64_t step, const float* coef,
                               cudaStream_t stream) {
  return launch_sgd_update(params, lay.P, lay.P, n_experts, n_pert, 0, lr, seed, step, coef,
                           stream);
}

cudaError_t launch_init(float* params, const Layout& lay, int n_experts, uint64_t seed, float std,
                        cudaStream_t stream) {
  const int64_t pairs = (lay.P + 1) / 2;
  dim3 grid((unsigned)((pairs + 255) / 256), n_experts);
  init_kernel<<<grid, 256, 0, stream>>>(params, lay, seed, std);
  return cudaGetLastError();
}

cudaError_t launch_debug_philox(uint64_t seed, const uint32_t* ctr4, uint32_t* out4, int count,
                                cudaStream_t stream) {
  debug_philox_kernel<<<(count + 127) / 128, 128, 0, stream>>>(seed, ctr4, out4, count);
  return cudaGetLastError();
}

cudaError_t launch_debug_rademacher(uint64_t seed, uint64_t step, int expert, int pert, int sparse,
                                    int64_t p0, int64_t count, int8_t* z, cudaStream_t stream) {
  const ProbeKey pk = make_probe_key(seed, step, (uint32_t)expert, (uint32_t)pert);
  const int64_t words = (count + 31) / 32;
  debug_rademacher_kernel<<<(unsigned)((words + 127) / 128), 128, 0, stream>>>(pk, sparse, p0,
                                                                                count, z);
  return cudaGetLastError();
}

cudaError_t launch_sum_over_experts(float* coef, int n_experts, int n_pert, cudaStream_t stream) {
  trace_begin(SOMA_TRACE_REDUCE, stream);
  sum_over_experts_kernel<<<(n_pert + 127) / 128, 128, 0, stream>>>(coef, n_experts, n_pert);
  trace_end(SOMA_TRACE_REDUCE, stream);
  return cudaGetLastError();
}

cudaError_t launch_probe_adam(float* params, float* m, float* v, int64_t P, int64_t dense_from,
                              int n_experts, int n_pert, int sparse, uint64_t seed,
                              const AdamSteps& steps, const float* coef, const AdamArgs& h,
                              cudaStream_t stream) {
  const int64_t words = (P + 31) / 32;
  dim3 grid((unsigned)((words + kUpdThreads - 1) / kUpdThreads), n_experts);
  trace_begin(SOMA_TRACE_UPDATE, stream);
  adam_update_kernel<<<grid, kUpdThreads, 0, stream>>>(params, m, v, P, dense_from, n_experts,
                                                       n_pert, sparse, seed, steps, coef, h);
  trace_end(SOMA_TRACE_UPDATE, stream);
  return cudaGetLastError();
}

cudaError_t launch_adam_update(float* params, float* m, float* v, const Layout& lay, int n_experts,
                               int n_pert, int sparse, uint64_t seed, const AdamSteps& steps,
                               const float* coef, const AdamArgs& h, cudaStream_t stream) {
  return launch_probe_adam(params, m, v, lay.P, lay.P, n_experts, n_pert, sparse, seed, steps,
                           coef, h, stream);
}

cudaError_t launch_debug_wait_timeout(uint32_t max_polls, int* status, cudaStream_t stream) {
  debug_wait_timeout_kernel<<<1, 32, 0, stream>>>(max_polls, status);
  return cudaGetLastError();
}

}  // namespace soma
