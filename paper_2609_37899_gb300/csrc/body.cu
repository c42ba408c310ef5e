// body.cu -- the paper's expert body (Sec. "Model size"; loss and probes of
// App. E): D pre-norm residual blocks of width d, each a bias-free LSTM and a
// bias-free GELU MLP of width 4d, gain-only LayerNorm, and one frozen tied
// head E [V][d] that embeds the byte and decodes the final normalised state
// (logits = E y).  Only the body is perturbed.
//
// Kernels:
//   body_sweep_kernel   the antithetic forwards.  One CTA runs one sign of one
//                       (expert, probe) pair over up to 16 sequences for all T
//                       timesteps, on CUDA cores in fp32.  Its perturbed
//                       weights theta + s eps z sit in shared memory for the
//                       whole sequence, and the state never leaves the CTA.
//   body_reduce_kernel  L+-, the coefficients (L+ - L-) / (2 eps) in fp64.
//   body_sgd_kernel     theta -= lr (1/n) sum_i c_i z_i (Eq. main-spsa).
//   body_adam_kernel    Eq. localspsa with coupled weight decay.
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

constexpr int kD = kBodyWidth;          // d_t = d_E
constexpr int kG = 4 * kD;              // gate / MLP width
constexpr int kRows = 16;               // sequences of one CTA (one sign)
constexpr int kThreads = 256;
constexpr int kBlockW = 16 * kD * kD;   // weights of one residual block
constexpr float kLnEps = 1e-5f;

// Shared-memory layout (floats).  Each block's weights are stored transposed
// (input feature major): W_ih^T, W_hh^T, W_1^T [d][4d] and W_2^T [4d][d], so
// that consecutive lanes read consecutive output features.  Activations are
// row-major [row][feature].
constexpr int kSmW = 0;
constexpr int kSmGain = kSmW + kBodyMaxBlocks * kBlockW;
constexpr int kSmET = kSmGain + (2 * kBodyMaxBlocks + 1) * kD;  // E^T [d][V]
constexpr int kSmX = kSmET + kD * kVocab;                       // residual stream [R][d]
constexpr int kSmU = kSmX + kRows * kD;                         // normalised stream [R][d]
constexpr int kSmH = kSmU + kRows * kD;                         // LSTM h per block [D][R][d]
constexpr int kSmGt = kSmH + kBodyMaxBlocks * kRows * kD;       // gates / MLP hidden [R][4d]
constexpr int kSmRed = kSmGt + kRows * kG;                      // MLP2 partials [4][R][d]
constexpr int kSmRow = kSmRed + 4 * kRows * kD;                 // head: max [4][R], sum [4][R], target [R]
constexpr int kSmFloats = kSmRow + 9 * kRows;
static_assert(kSmET % 4 == 0 && kSmX % 4 == 0 && kSmGt % 4 == 0, "float4 alignment");

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float sigmoidf_(float a) { return 1.f / (1.f + expf(-a)); }

__device__ __forceinline__ float gelu_erf(float a) {
  return 0.5f * a * (1.f + erff(a * 0.70710678118654752f));
}

// Shared-memory slot of body coordinate p (p < 16 D d^2: a weight).
__device__ __forceinline__ int weight_slot(int p) {
  const int blk = p / kBlockW;
  const int f = p - blk * kBlockW;
  const int region = f / (4 * kD * kD);
  const int loc = f - region * 4 * kD * kD;
  int s;
  if (region < 3) {  // [4d][d] row-major -> [d][4d]
    const int j = loc / kD, k = loc - j * kD;
    s = region * 4 * kD * kD + k * kG + j;
  } else {           // W_2 [d][4d] -> [4d][d]
    const int j = loc / kG, k = loc - j * kG;
    s = 3 * 4 * kD * kD + k * kD + j;
  }
  return kSmW + blk * kBlockW + s;
}

// out[r][k] = LN(x[r]) * g for rows 2w, 2w + 1 (warp w, lane = feature).
__device__ __forceinline__ void layer_norm_rows(const float* __restrict__ x,
                                                float* __restrict__ out,
                                                const float* __restrict__ g, int warp, int lane) {
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    const int r = 2 * warp + q;
    const float v = x[r * kD + lane];
    const float mu = warp_sum(v) * (1.f / kD);
    const float dv = v - mu;
    const float var = warp_sum(dv * dv) * (1.f / kD);
    out[r * kD + lane] = dv * rsqrtf(var + kLnEps) * g[lane];
  }
}

// acc[q] += sum_{k < K} in[r0 + q][k] * WT[k][j] for 8 rows, K a multiple of 4.
template <int K, int LDW, int LDI>
__device__ __forceinline__ void rows8_dot(float (&acc)[8], const float* __restrict__ in, int r0,
                                          const float* __restrict__ WT, int j) {
#pragma unroll 2
  for (int k = 0; k < K; k += 4) {
    const float w0 = WT[(k + 0) * LDW + j];
    const float w1 = WT[(k + 1) * LDW + j];
    const float w2 = WT[(k + 2) * LDW + j];
    const float w3 = WT[(k + 3) * LDW + j];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const float4 a = *reinterpret_cast<const float4*>(in + (r0 + q) * LDI + k);
      acc[q] = fmaf(a.x, w0, acc[q]);
      acc[q] = fmaf(a.y, w1, acc[q]);
      acc[q] = fmaf(a.z, w2, acc[q]);
      acc[q] = fmaf(a.w, w3, acc[q]);
    }
  }
}

struct BodySweep {
  const float* params;   // [N][P]
  const float* head;     // [V][d]
  const uint8_t* bytes;  // [N][B][T+1]
  double* partial;       // [N * n * n_sign][chunks] NLL sums
  int n_experts, n_pert, n_sign, blocks, B, T, chunks;
  int64_t P, goff;
  float eps;
  int sparse;
  uint64_t seed, step;
};

__global__ void __launch_bounds__(kThreads, 1) body_sweep_kernel(BodySweep a) {
  extern __shared__ __align__(16) float sm[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int cta = blockIdx.x;  // (pair, sign)
  const int s = cta % a.n_sign;
  const int pair = cta / a.n_sign;
  const int e = pair / a.n_pert, i = pair % a.n_pert;
  const int chunk = blockIdx.y;
  const int b0 = chunk * kRows;
  const int rows = min(kRows, a.B - b0);
  const int D = a.blocks;
  const float se = (s == 0) ? a.eps : -a.eps;

  // ---- theta + s eps z into shared memory (transposed), E^T ---------------
  const float* th = a.params + (int64_t)e * a.P;
  const ProbeKey pk = make_probe_key(a.seed, a.step, (uint32_t)e, (uint32_t)i);
  const int runs = (int)((a.P + 31) / 32);
  for (int q = tid; q < runs; q += kThreads) {
    uint32_t neg, act;
    body_probe_words(pk, q, a.sparse, a.goff, neg, act);
    const int p0 = 32 * q;
#pragma unroll 4
    for (int j = 0; j < 32; ++j) {
      const int p = p0 + j;
      if (p >= a.P) break;
      const float w = th[p];
      const float v = ((act >> j) & 1u) ? w + (((neg >> j) & 1u) ? -se : se) : w;
      sm[p < a.goff ? weight_slot(p) : kSmGain + (p - (int)a.goff)] = v;
    }
  }
  for (int idx = tid; idx < kD * kVocab; idx += kThreads) {
    const int k = idx / kVocab, v = idx - k * kVocab;
    sm[kSmET + idx] = a.head[v * kD + k];
  }
  for (int idx = tid; idx < kBodyMaxBlocks * kRows * kD; idx += kThreads) sm[kSmH + idx] = 0.f;

  float* xs = sm + kSmX;
  float* us = sm + kSmU;
  float* gt = sm + kSmGt;
  float* red = sm + kSmRed;
  float* rmax = sm + kSmRow;
  float* rsum = rmax + 4 * kRows;
  float* rtgt = rsum + 4 * kRows;
  const float* ET = sm + kSmET;

  // the bytes of this CTA's rows (rows past the batch read row 0's bytes;
  // they are computed and never counted)
  const int T1 = a.T + 1;
  const uint8_t* bx = a.bytes + ((int64_t)e * a.B + b0) * T1;
  // embedding prefetch: thread -> (row, 2 features)
  const int er = tid >> 4, ek = (tid & 15) * 2;
  const uint8_t* brow = bx + (int64_t)(er < rows ? er : 0) * T1;
  float2 emb = *reinterpret_cast<const float2*>(a.head + (int)brow[0] * kD + ek);

  float cst[kBodyMaxBlocks][2];
#pragma unroll
  for (int b = 0; b < kBodyMaxBlocks; ++b) cst[b][0] = cst[b][1] = 0.f;
  double loss = 0.0;  // thread r < rows: its row's NLL sum
  __syncthreads();

  for (int t = 0; t < a.T; ++t) {
    // ---- x = E[byte_t] ----------------------------------------------------
    *reinterpret_cast<float2*>(xs + er * kD + ek) = emb;
    if (t + 1 < a.T)
      emb = *reinterpret_cast<const float2*>(a.head + (int)brow[t + 1] * kD + ek);
    __syncthreads();

#pragma unroll
    for (int b = 0; b < kBodyMaxBlocks; ++b) {
      if (b >= D) break;
      const float* W = sm + kSmW + b * kBlockW;
      float* hs = sm + kSmH + b * kRows * kD;
      // ---- LSTM sublayer on LN(x) ----------------------------------------
      layer_norm_rows(xs, us, sm + kSmGain + 2 * b * kD, warp, lane);
      __syncthreads();
      {
        const int j = tid & (kG - 1), r0 = (tid >> 7) * 8;
        float acc[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] = 0.f;
        rows8_dot<kD, kG, kD>(acc, us, r0, W, j);                    // W_ih u
        rows8_dot<kD, kG, kD>(acc, hs, r0, W + 4 * kD * kD, j);      // W_hh h_{t-1}
#pragma unroll
        for (int q = 0; q < 8; ++q) gt[(r0 + q) * kG + j] = acc[q];
      }
      __syncthreads();
      {
        const int j = lane;
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          const int r = warp + 8 * q;
          const float* g = gt + r * kG;
          const float ig = sigmoidf_(g[j]);
          const float fg = sigmoidf_(g[kD + j]);
          const float gg = tanhf(g[2 * kD + j]);
          const float og = sigmoidf_(g[3 * kD + j]);
          const float c = fmaf(fg, cst[b][q], ig * gg);
          cst[b][q] = c;
          const float h = og * tanhf(c);
          hs[r * kD + j] = h;
          xs[r * kD + j] += h;
        }
      }
      __syncthreads();
      // ---- MLP sublayer on LN(x) -----------------------------------------
      layer_norm_rows(xs, us, sm + kSmGain + 2 * b * kD + kD, warp, lane);
      __syncthreads();
      {
        const int j = tid & (kG - 1), r0 = (tid >> 7) * 8;
        float acc[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] = 0.f;
        rows8_dot<kD, kG, kD>(acc, us, r0, W + 8 * kD * kD, j);      // W_1 v
#pragma unroll
        for (int q = 0; q < 8; ++q) gt[(r0 + q) * kG + j] = gelu_erf(acc[q]);
      }
      __syncthreads();
      {
        // W_2 m: K = 4d split in four quarters, one per thread group
        const int j = lane, r0 = ((tid >> 5) & 1) * 8, kq = tid >> 6;
        float acc[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] = 0.f;
        rows8_dot<kD, kD, kG>(acc, gt + kq * kD, r0, W + 12 * kD * kD + kq * kD * kD, j);
#pragma unroll
        for (int q = 0; q < 8; ++q) red[(kq * kRows + r0 + q) * kD + j] = acc[q];
      }
      __syncthreads();
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const int idx = tid + q * kThreads;  // (row, feature)
        xs[idx] += (red[idx] + red[kRows * kD + idx]) +
                   (red[2 * kRows * kD + idx] + red[3 * kRows * kD + idx]);
      }
      __syncthreads();
    }

    // ---- y = LN(x) gf; logits = E y; NLL ----------------------------------
    layer_norm_rows(xs, us, sm + kSmGain + 2 * D * kD, warp, lane);
    __syncthreads();
    {
      const int v0 = tid & 127, r0 = (tid >> 7) * 8, wq = (tid >> 5) & 3;
      float l0[8], l1[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) l0[q] = l1[q] = 0.f;
      rows8_dot<kD, kVocab, kD>(l0, us, r0, ET, v0);
      rows8_dot<kD, kVocab, kD>(l1, us, r0, ET, v0 + 128);
      float mx[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        mx[q] = warp_max(fmaxf(l0[q], l1[q]));
        const int r = r0 + q;
        const int y = (int)bx[(int64_t)(r < rows ? r : 0) * T1 + t + 1];
        if (y == v0) rtgt[r] = l0[q];
        if (y == v0 + 128) rtgt[r] = l1[q];
        if (lane == 0) rmax[wq * kRows + r] = mx[q];
      }
      __syncthreads();
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int r = r0 + q;
        const float m = fmaxf(fmaxf(rmax[r], rmax[kRows + r]),
                              fmaxf(rmax[2 * kRows + r], rmax[3 * kRows + r]));
        mx[q] = m;
        const float se_ = warp_sum(expf(l0[q] - m) + expf(l1[q] - m));
        if (lane == 0) rsum[wq * kRows + r] = se_;
      }
      __syncthreads();
      if (tid < rows) {
        const int r = tid;
        const float m = fmaxf(fmaxf(rmax[r], rmax[kRows + r]),
                              fmaxf(rmax[2 * kRows + r], rmax[3 * kRows + r]));
        const float sum = (rsum[r] + rsum[kRows + r]) + (rsum[2 * kRows + r] + rsum[3 * kRows + r]);
        loss += (double)(m + logf(sum) - rtgt[r]);
      }
    }
    // the next timestep writes xs (read by nothing here) before its first
    // barrier, and rmax / rsum / rtgt only after several
  }

  // ---- the CTA's NLL sum, rows in order -----------------------------------
  __syncthreads();
  double* dred = reinterpret_cast<double*>(sm + kSmRed);
  if (tid < kRows) dred[tid] = (tid < rows) ? loss : 0.0;
  __syncthreads();
  if (tid == 0) {
    double tot = 0.0;
    for (int r = 0; r < kRows; ++r) tot += dred[r];
    a.partial[(int64_t)cta * a.chunks + chunk] = tot;
  }
}

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

constexpr int kUpd = 128;

// theta[e][p] -= lr (1/n) sum_i coef[e][i] z_{e,i}[p]; thread q owns the 32
// coordinates 32q .. 32q + 31.  An expert with a non-finite coefficient is
// left unchanged.
__global__ void __launch_bounds__(kUpd) body_sgd_kernel(float* __restrict__ params, int64_t P,
                                                        int64_t goff, int n_pert, int sparse,
                                                        float lr, uint64_t seed, uint64_t step,
                                                        const float* __restrict__ coef) {
  extern __shared__ float cf[];
  __shared__ int all_finite;
  const int e = blockIdx.y;
  if (threadIdx.x == 0) all_finite = 1;
  __syncthreads();
  for (int i = threadIdx.x; i < n_pert; i += kUpd) {
    const float c = coef[(int64_t)e * n_pert + i];
    cf[i] = c;
    if (!isfinite(c)) all_finite = 0;
  }
  __syncthreads();
  if (!all_finite) return;
  const int64_t q = (int64_t)blockIdx.x * kUpd + threadIdx.x;
  const int64_t p0 = q * 32;
  if (p0 >= P) return;
  float acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0.f;
  for (int i = 0; i < n_pert; ++i) {
    uint32_t neg, act;
    body_probe_words(make_probe_key(seed, step, (uint32_t)e, (uint32_t)i), (int)q, sparse, goff,
                     neg, act);
    const float c = cf[i];
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if ((act >> j) & 1u) acc[j] += ((neg >> j) & 1u) ? -c : c;
  }
  const float scale = lr / (float)n_pert;
  float* th = params + (int64_t)e * P + p0;
  const int cnt = P - p0 < 32 ? (int)(P - p0) : 32;
  for (int j = 0; j < cnt; ++j) th[j] -= scale * acc[j];
}

// Eq. localspsa: the estimate averaged over n_acc batches, coupled decay,
// bias-corrected Adam moments.
__global__ void __launch_bounds__(kUpd) body_adam_kernel(float* __restrict__ params,
                                                         float* __restrict__ m,
                                                         float* __restrict__ v, int64_t P,
                                                         int64_t goff, int n_experts, int n_pert,
                                                         int sparse, uint64_t seed, AdamSteps st,
                                                         const float* __restrict__ coef,
                                                         AdamArgs h) {
  __shared__ int all_finite;
  const int e = blockIdx.y;
  if (threadIdx.x == 0) all_finite = 1;
  __syncthreads();
  for (int j = threadIdx.x; j < st.n_acc * n_pert; j += kUpd) {
    const int aa = j / n_pert, i = j % n_pert;
    if (!isfinite(coef[((int64_t)aa * n_experts + e) * n_pert + i])) all_finite = 0;
  }
  __syncthreads();
  if (!all_finite) return;
  const int64_t q = (int64_t)blockIdx.x * kUpd + threadIdx.x;
  const int64_t p0 = q * 32;
  if (p0 >= P) return;
  float acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0.f;
  for (int aa = 0; aa < st.n_acc; ++aa) {
    const float* ca = coef + ((int64_t)aa * n_experts + e) * n_pert;
    for (int i = 0; i < n_pert; ++i) {
      uint32_t neg, act;
      body_probe_words(make_probe_key(seed, st.step[aa], (uint32_t)e, (uint32_t)i), (int)q,
                       sparse, goff, neg, act);
      const float c = ca[i];
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if ((act >> j) & 1u) acc[j] += ((neg >> j) & 1u) ? -c : c;
    }
  }
  const float inv = 1.f / ((float)st.n_acc * (float)n_pert);
  const int64_t base = (int64_t)e * P + p0;
  const int cnt = P - p0 < 32 ? (int)(P - p0) : 32;
  for (int j = 0; j < cnt; ++j) {
    const float w = params[base + j];
    const float g = fmaf(h.wd, w, acc[j] * inv);
    const float mj = fmaf(h.b1, m[base + j], (1.f - h.b1) * g);
    const float vj = fmaf(h.b2, v[base + j], (1.f - h.b2) * g * g);
    m[base + j] = mj;
    v[base + j] = vj;
    params[base + j] = w - h.lr * (mj * h.inv_bc1) / (sqrtf(vj * h.inv_bc2) + h.delta);
  }
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

size_t body_smem_bytes() { return (size_t)kSmFloats * sizeof(float); }
int body_rows_per_cta() { return kRows; }

cudaError_t launch_body_sweep(const float* params, const float* head, const uint8_t* bytes,
                              int n_experts, int blocks, int n_pert, int n_sign, int B, int T,
                              float eps, int sparse, uint64_t seed, uint64_t step,
                              double* partial, cudaStream_t stream) {
  BodySweep a;
  a.params = params;
  a.head = head;
  a.bytes = bytes;
  a.partial = partial;
  a.n_experts = n_experts;
  a.n_pert = n_pert;
  a.n_sign = n_sign;
  a.blocks = blocks;
  a.B = B;
  a.T = T;
  a.chunks = (B + kRows - 1) / kRows;
  a.P = body_param_count(kD, blocks);
  a.goff = body_gain_offset(kD, blocks);
  a.eps = eps;
  a.sparse = sparse;
  a.seed = seed;
  a.step = step;
  // per device and cheap: set on every launch
  cudaError_t err = cudaFuncSetAttribute(body_sweep_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)body_smem_bytes());
  if (err != cudaSuccess) return err;
  dim3 grid((unsigned)((int64_t)n_experts * n_pert * n_sign), (unsigned)a.chunks);
  trace_begin(SOMA_TRACE_GATE, stream);
  body_sweep_kernel<<<grid, kThreads, body_smem_bytes(), stream>>>(a);
  trace_end(SOMA_TRACE_GATE, stream);
  return cudaGetLastError();
}

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
  const int64_t P = body_param_count(kD, blocks);
  const int64_t words = (P + 31) / 32;
  dim3 grid((unsigned)((words + kUpd - 1) / kUpd), n_experts);
  trace_begin(SOMA_TRACE_UPDATE, stream);
  body_sgd_kernel<<<grid, kUpd, n_pert * sizeof(float), stream>>>(
      params, P, body_gain_offset(kD, blocks), n_pert, sparse, lr, seed, step, coef);
  trace_end(SOMA_TRACE_UPDATE, stream);
  return cudaGetLastError();
}

cudaError_t launch_body_adam(float* params, float* m, float* v, int n_experts, int blocks,
                             int n_pert, int sparse, uint64_t seed, const AdamSteps& steps,
                             const float* coef, const AdamArgs& h, cudaStream_t stream) {
  const int64_t P = body_param_count(kD, blocks);
  const int64_t words = (P + 31) / 32;
  dim3 grid((unsigned)((words + kUpd - 1) / kUpd), n_experts);
  trace_begin(SOMA_TRACE_UPDATE, stream);
  body_adam_kernel<<<grid, kUpd, 0, stream>>>(params, m, v, P, body_gain_offset(kD, blocks),
                                              n_experts, n_pert, sparse, seed, steps, coef, h);
  trace_end(SOMA_TRACE_UPDATE, stream);
  return cudaGetLastError();
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
