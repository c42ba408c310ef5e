// spsa_misc.cu -- the SPSA and Adam updates, the summed-loss arm, the
// parameter initialisation and the generator test kernels.
#define SOMA_CHECK_FILE 4
#include "checked.cuh"
#include "soma_api.h"
#include "probe_law.cuh"
#include "soma_launch.h"
#include "tc_primitives.cuh"

namespace soma {

namespace {

constexpr int kUpdThreads = 128;
constexpr int kUpdParams = kUpdThreads * 32;  // parameters of one block

// Adds the probe terms c_i z_i of probes i0 .. i0 + 3 to the 32 parameters of
// run q (32q .. 32q + 31) owned by this thread.  One Philox block covers the
// 128 parameters of four consecutive runs, i.e. of a group of four
// consecutive lanes (q % 4 == lane % 4), so lane j of the group draws the
// block of probe i0 + j (and its activity block for sparse probes) and the
// four lanes pass words round: in round k every lane sends word (j - k) % 4
// of its block and receives, from lane (j + k) % 4 of the group, the word of
// its own run for probe i0 + (j + k) % 4.  One Philox block per 128
// parameters and probe, one shuffle per probe and word kind.  All 32 lanes
// of the warp take part.
__device__ __forceinline__ void accumulate_x4(float (&acc)[32], const float* cf, int n_pert,
                                              int i0, const ProbeKey& pk0, int64_t q, int sparse,
                                              int64_t dense_from) {
  const int lane = threadIdx.x & 31;
  const int j = lane & 3, base = lane & ~3;
  uint4 wn = make_uint4(0u, 0u, 0u, 0u), wa = make_uint4(0u, 0u, 0u, 0u);
  if (i0 + j < n_pert) {
    ProbeKey pk = pk0;
    pk.probe = (uint32_t)(i0 + j);
    const uint32_t blk = (uint32_t)(q >> 2);
    wn = probe_block(pk, blk);
    if (sparse) wa = probe_block(activity_key(pk), blk);
  }
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int send = (j - k) & 3, from = (j + k) & 3;
    const uint32_t rn =
        __shfl_sync(0xffffffffu, word_of(wn, send), base | from);
    uint32_t act = 0xFFFFFFFFu;
    if (sparse) act = probe_law_act(__shfl_sync(0xffffffffu, word_of(wa, send), base | from), q,
                                    dense_from);
    const int i = i0 + from;
    if (i >= n_pert) continue;
    const uint32_t neg = raw_to_natural(rn);
    const float c = cf[i];
#pragma unroll
    for (int b = 0; b < 32; ++b)
      if ((act >> b) & 1u) acc[b] += ((neg >> b) & 1u) ? -c : c;
  }
}

// Writes the block's 32 x kUpdThreads accumulators to shared memory in
// parameter order (thread t: parameters 32t .. 32t + 31 of the block).
__device__ __forceinline__ void stage_acc(float* sacc, const float (&acc)[32], float scale) {
  float4* dst = reinterpret_cast<float4*>(sacc + 32 * threadIdx.x);
#pragma unroll
  for (int j4 = 0; j4 < 8; ++j4)
    dst[j4] = make_float4(scale * acc[4 * j4], scale * acc[4 * j4 + 1], scale * acc[4 * j4 + 2],
                          scale * acc[4 * j4 + 3]);
}

// theta[e][p] -= lr * (1/n) * sum_i coef[e][i] z_{e,i}[p] (Eq. main-spsa).
// Thread q of expert e accumulates the 32 parameters 32q .. 32q + 31 under
// the probe law of probe_law_words (accumulate_x4); the block then stages its
// 4096 steps in shared memory and reads and writes theta as consecutive
// float4s, so a warp's access covers 512 contiguous bytes.  An expert whose
// coefficients are not all finite is left unchanged.
__global__ void __launch_bounds__(kUpdThreads)
sgd_update_kernel(float* __restrict__ params, int64_t P, int64_t dense_from, int n_pert,
                  int sparse, float lr, uint64_t seed, uint64_t step,
                  const float* __restrict__ coef) {
  extern __shared__ float cf[];  // [n_pert]
  __shared__ __align__(16) float sacc[kUpdParams];
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
  float acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0.f;
  const ProbeKey pk0 = make_probe_key(seed, step, (uint32_t)e, 0u);
  // runs past the end draw probe words too (their Philox counters exist) and
  // are simply not written back
  for (int i0 = 0; i0 < n_pert; i0 += 4) accumulate_x4(acc, cf, n_pert, i0, pk0, q, sparse,
                                                       dense_from);
  stage_acc(sacc, acc, lr / (float)n_pert);
  __syncthreads();
  const int64_t p0 = (int64_t)blockIdx.x * kUpdParams;
  float* th = params + (int64_t)e * P + p0;
  const int64_t left = P - p0;
  for (int k = threadIdx.x; k < kUpdParams / 4; k += kUpdThreads) {
    const int64_t p = 4LL * k;
    if (p >= left) break;
    if (p + 4 <= left && (P & 3) == 0) {
      // P a multiple of 4: theta + p is 16-byte aligned
      float4 v = reinterpret_cast<float4*>(th)[k];
      const float4 d = reinterpret_cast<const float4*>(sacc)[k];
      v.x -= d.x;
      v.y -= d.y;
      v.z -= d.z;
      v.w -= d.w;
      reinterpret_cast<float4*>(th)[k] = v;
    } else {
      for (int64_t pp = p; pp < p + 4 && pp < left; ++pp) th[pp] -= sacc[pp];
    }
  }
}

// The paper's optimizer step (App. E, Eq. localspsa) for expert e:
//   g = (1/(A n)) sum_a sum_i coef[a][e][i] z_{e,i}^{(a)} + wd * theta,
//   m = b1 m + (1 - b1) g,  v = b2 v + (1 - b2) g^2,
//   theta -= lr * (m / bc1) / (sqrt(v / bc2) + delta),
// with z^{(a)} drawn with step counter steps[a] under the probe law of
// probe_law_words.  Thread q accumulates the 32 parameters 32q .. 32q + 31;
// the block stages the averaged estimate in shared memory and updates
// theta, m and v as consecutive float4s.  An expert whose coefficients are
// not all finite is left unchanged, moments included.
__global__ void __launch_bounds__(kUpdThreads)
adam_update_kernel(float* __restrict__ params, float* __restrict__ m, float* __restrict__ v,
                   int64_t P, int64_t dense_from, int n_experts, int n_pert, int sparse,
                   uint64_t seed, AdamSteps steps, const float* __restrict__ coef, AdamArgs h) {
  extern __shared__ float cf[];  // [n_pert]: the coefficients of one accumulation batch
  __shared__ __align__(16) float sacc[kUpdParams];
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
  float acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0.f;
  for (int a = 0; a < steps.n_acc; ++a) {
    for (int i = threadIdx.x; i < n_pert; i += kUpdThreads)
      cf[i] = coef[((int64_t)a * n_experts + e) * n_pert + i];
    __syncthreads();
    const ProbeKey pk0 = make_probe_key(seed, steps.step[a], (uint32_t)e, 0u);
    for (int i0 = 0; i0 < n_pert; i0 += 4)
      accumulate_x4(acc, cf, n_pert, i0, pk0, q, sparse, dense_from);
    __syncthreads();  // cf is refilled for the next batch
  }
  stage_acc(sacc, acc, 1.f / ((float)steps.n_acc * (float)n_pert));
  __syncthreads();
  const int64_t p0 = (int64_t)blockIdx.x * kUpdParams;
  const int64_t base = (int64_t)e * P + p0;
  const int64_t left = P - p0;
  for (int k = threadIdx.x; k < kUpdParams / 4; k += kUpdThreads) {
    const int64_t p = 4LL * k;
    if (p >= left) break;
    if (p + 4 <= left && (P & 3) == 0) {
      float4 t4 = reinterpret_cast<float4*>(params + base)[k];
      float4 m4 = reinterpret_cast<float4*>(m + base)[k];
      float4 v4 = reinterpret_cast<float4*>(v + base)[k];
      const float4 g4 = reinterpret_cast<const float4*>(sacc)[k];
      float* tt = &t4.x;
      float* mm = &m4.x;
      float* vv = &v4.x;
      const float* gg = &g4.x;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const float g = fmaf(h.wd, tt[c], gg[c]);
        mm[c] = fmaf(h.b1, mm[c], (1.f - h.b1) * g);
        vv[c] = fmaf(h.b2, vv[c], (1.f - h.b2) * g * g);
        tt[c] = tt[c] - h.lr * (mm[c] * h.inv_bc1) / (sqrtf(vv[c] * h.inv_bc2) + h.delta);
      }
      reinterpret_cast<float4*>(params + base)[k] = t4;
      reinterpret_cast<float4*>(m + base)[k] = m4;
      reinterpret_cast<float4*>(v + base)[k] = v4;
    } else {
      for (int64_t pp = p; pp < p + 4 && pp < left; ++pp) {
        const float th = params[base + pp];
        const float g = fmaf(h.wd, th, sacc[pp]);
        const float mj = fmaf(h.b1, m[base + pp], (1.f - h.b1) * g);
        const float vj = fmaf(h.b2, v[base + pp], (1.f - h.b2) * g * g);
        m[base + pp] = mj;
        v[base + pp] = vj;
        params[base + pp] = th - h.lr * (mj * h.inv_bc1) / (sqrtf(vj * h.inv_bc2) + h.delta);
      }
    }
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

// An index check whose condition is false and that guards no access: the
// reporting path of the checked build (nothing happens in the default one).
__global__ void debug_check_fail_kernel(int* status) {
  if (threadIdx.x == 0) (void)SOMA_CHECK(blockDim.x == 0, status);
}
}  // namespace

cudaError_t launch_sgd_update(float* params, int64_t P, int64_t dense_from, int n_experts,
                              int n_pert, int sparse, float lr, uint64_t seed, uint64_t step,
                              const float* coef, cudaStream_t stream) {
  const int64_t words = (P + 31) / 32;
  dim3 grid((unsigned)((words + kUpdThreads - 1) / kUpdThreads), n_experts);
  const size_t smem = (size_t)n_pert * sizeof(float);  // plus the 16 KB staging array
  cudaError_t e = cudaFuncSetAttribute(sgd_update_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  trace_begin(SOMA_TRACE_UPDATE, stream);
  sgd_update_kernel<<<grid, kUpdThreads, smem, stream>>>(params, P, dense_from, n_pert, sparse,
                                                          lr, seed, step, coef);
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
  const size_t smem = (size_t)n_pert * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(adam_update_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  trace_begin(SOMA_TRACE_UPDATE, stream);
  adam_update_kernel<<<grid, kUpdThreads, smem, stream>>>(params, m, v, P, dense_from, n_experts,
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

cudaError_t launch_debug_check_fail(int* status, cudaStream_t stream) {
  debug_check_fail_kernel<<<1, 32, 0, stream>>>(status);
  return cudaGetLastError();
}

cudaError_t launch_debug_wait_timeout(uint32_t max_polls, int* status, cudaStream_t stream) {
  debug_wait_timeout_kernel<<<1, 32, 0, stream>>>(max_polls, status);
  return cudaGetLastError();
}

}  // namespace soma
