// forward_simt.cu -- fp32 CUDA-core forward sweep of the perturbed LSTM
// experts: one gate/cell kernel per timestep and one head + log-softmax +
// NLL kernel per chunk of timesteps.
//
// Every (expert e, probe i, sign s) "lane" runs the LSTM of App. C with its
// parameters theta_e + s*eps*z_{e,i}; each perturbed weight is formed in
// fp32 when its tile is staged (w + s*eps*z, z regenerated from Philox), so
// no perturbed copy of theta exists in memory.  All arithmetic is fp32 and the
// per-target NLL of every lane is written out for the loss reduction.
#include "soma_api.h"
#include "soma_device.cuh"
#include "soma_launch.h"

namespace soma {

namespace {

constexpr int kUnits = 32;     // hidden units per gate CTA (4 x 32 gate rows)
constexpr int kKc = 32;        // reduction chunk
constexpr int kCols = 32;      // sequences per gate CTA
constexpr int kColsPerThr = 8; // sequences per thread in the gate CTA
constexpr int kHeadCols = 32;  // (timestep, sequence) columns per head CTA

struct GateStep {
  Sweep sw;
  int t, slot, prev_slot, Tc;
  float* hist;  // [lanes][Tc][B][H]
  float* cst;   // [lanes][B][H]
};

__device__ __forceinline__ float sigmoidf_(float a) { return 1.0f / (1.0f + expf(-a)); }

// grid (lanes, ceil(H / 32), ceil(B / 32)), block 128.
// Thread (cu = tid % 32, cg = tid / 32) owns hidden unit u0 + cu (all four
// gates) for the 8 sequences b0 + 8 cg .. +7.
__global__ void __launch_bounds__(128) gate_step_kernel(const GateStep g) {
  __shared__ __align__(16) float Wt[kKc][kUnits][4];  // perturbed W rows, (k, unit, gate)
  __shared__ __align__(16) float Vt[kKc][kCols];      // inputs [x; h_{t-1}], (k, sequence)

  const Sweep& s = g.sw;
  const int lane_id = blockIdx.x;
  const int u0 = blockIdx.y * kUnits;
  const int b0 = blockIdx.z * kCols;
  int e, i;
  float se;
  lane_parts(s, lane_id, e, i, se);
  const Layout& L = s.lay;
  const int E = L.E, H = L.H, B = s.B;
  const float* th = s.params + (int64_t)e * L.P;
  const ProbeKey pk = make_probe_key(s.seed, s.step, (uint32_t)e, (uint32_t)i);
  const bool pert = s.eps != 0.f;
  const int tid = threadIdx.x;

  // staging roles
  const int lg = tid & 3, lu = tid >> 2;  // weight row: gate lg of unit u0 + lu
  const int wrow = lg * H + u0 + lu;
  const bool wrow_ok = (u0 + lu) < H;
  const int lc = tid & 31, lk0 = (tid >> 5) * 8;  // input column lc, k range lk0..+7
  const int bcol = b0 + lc;
  const bool col_ok = bcol < B;
  const uint8_t* seq = s.bytes + seq_offset(s, e, i, col_ok ? bcol : 0);
  const int xbyte = seq[g.t];
  const float* hprev =
      (g.t == 0 || !col_ok)
          ? nullptr
          : g.hist + (((int64_t)lane_id * g.Tc + g.prev_slot) * B + bcol) * (int64_t)H;

  // compute roles
  const int cu = tid & 31, cg = tid >> 5;
  float acc[4][kColsPerThr];
#pragma unroll
  for (int q = 0; q < 4; ++q)
#pragma unroll
    for (int j = 0; j < kColsPerThr; ++j) acc[q][j] = 0.f;

  const int nk = E + H;
  for (int k0 = 0; k0 < nk;) {
    // a chunk never straddles the x / h boundary of [x; h]
    const bool xpart = k0 < E;
    const int kc = min(kKc, (xpart ? E : nk) - k0);
    {  // perturbed weights: row wrow, reduction indices k0 .. k0 + kc - 1
      const int64_t p = xpart ? L.w_ih + (int64_t)wrow * E + k0
                              : L.w_hh + (int64_t)wrow * H + (k0 - E);
      ProbeBits bits = {0u, 0u};
      if (pert && wrow_ok) bits = probe_bits(pk, p, s.sparse);
#pragma unroll
      for (int k = 0; k < kKc; ++k) {
        float w = 0.f;
        if (wrow_ok && k < kc) w = perturb(th[p + k], (bits.neg >> k) & 1u, (bits.act >> k) & 1u, se);
        Wt[k][lu][lg] = w;
      }
    }
    {  // inputs: perturbed embedding row of byte_t, or h_{t-1}
      ProbeBits xbits = {0u, 0u};
      if (xpart && pert && col_ok)
        xbits = probe_bits(pk, L.emb + (int64_t)xbyte * E + k0 + lk0, s.sparse);
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const int k = lk0 + kk;
        float v = 0.f;
        if (col_ok && k < kc) {
          if (xpart) {
            v = perturb(th[L.emb + (int64_t)xbyte * E + k0 + k], (xbits.neg >> kk) & 1u,
                        (xbits.act >> kk) & 1u, se);
          } else if (hprev) {
            v = hprev[k0 - E + k];
          }
        }
        Vt[k][lc] = v;
      }
    }
    __syncthreads();
    for (int k = 0; k < kc; ++k) {
      const float4 w4 = *reinterpret_cast<const float4*>(&Wt[k][cu][0]);
      const float4 va = *reinterpret_cast<const float4*>(&Vt[k][cg * kColsPerThr]);
      const float4 vb = *reinterpret_cast<const float4*>(&Vt[k][cg * kColsPerThr + 4]);
      const float v[8] = {va.x, va.y, va.z, va.w, vb.x, vb.y, vb.z, vb.w};
#pragma unroll
      for (int j = 0; j < kColsPerThr; ++j) {
        acc[0][j] = fmaf(w4.x, v[j], acc[0][j]);
        acc[1][j] = fmaf(w4.y, v[j], acc[1][j]);
        acc[2][j] = fmaf(w4.z, v[j], acc[2][j]);
        acc[3][j] = fmaf(w4.w, v[j], acc[3][j]);
      }
    }
    __syncthreads();
    k0 += kc;
  }

  // fused epilogue: bias, gates (i, f, g, o), cell and hidden update
  const int u = u0 + cu;
  if (u >= H) return;
  float bias[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int64_t p = L.b + (int64_t)q * H + u;
    ProbeBits bit = {0u, 0u};
    if (pert) bit = probe_bits(pk, p, s.sparse);
    bias[q] = perturb(th[p], bit.neg & 1u, bit.act & 1u, se);
  }
#pragma unroll
  for (int j = 0; j < kColsPerThr; ++j) {
    const int b = b0 + cg * kColsPerThr + j;
    if (b >= B) break;
    const float ig = sigmoidf_(acc[0][j] + bias[0]);
    const float fg = sigmoidf_(acc[1][j] + bias[1]);
    const float gg = tanhf(acc[2][j] + bias[2]);
    const float og = sigmoidf_(acc[3][j] + bias[3]);
    float* cp = g.cst + ((int64_t)lane_id * B + b) * H + u;
    const float cprev = (g.t == 0) ? 0.f : *cp;
    const float c = fg * cprev + ig * gg;
    *cp = c;
    g.hist[(((int64_t)lane_id * g.Tc + g.slot) * B + b) * (int64_t)H + u] = og * tanhf(c);
  }
}

struct HeadChunk {
  Sweep sw;
  int t0, nt, Tc;
  const float* hist;  // [lanes][Tc][B][H]
  float* nll;         // [lanes][B][T]
};

// grid (lanes, ceil(nt * B / 32)), block 256.
// Thread v owns vocabulary row v of the perturbed head for 32 columns; a
// column is one (timestep, sequence) pair of this chunk.
__global__ void __launch_bounds__(256) head_nll_kernel(const HeadChunk hc) {
  __shared__ __align__(16) union {
    struct {
      float Wt[kKc][kVocab];     // perturbed W_out, (k, vocab row)
      float Ht[kKc][kHeadCols];  // h_t, (k, column)
    } g;
    float Lg[kVocab][kHeadCols + 1];  // logits, (vocab row, column)
  } sm;

  const Sweep& s = hc.sw;
  const int lane_id = blockIdx.x;
  const int c0 = blockIdx.y * kHeadCols;
  const int ncols = hc.nt * s.B;
  int e, i;
  float se;
  lane_parts(s, lane_id, e, i, se);
  const Layout& L = s.lay;
  const int H = L.H, B = s.B;
  const float* th = s.params + (int64_t)e * L.P;
  const ProbeKey pk = make_probe_key(s.seed, s.step, (uint32_t)e, (uint32_t)i);
  const bool pert = s.eps != 0.f;
  const int tid = threadIdx.x;

  // staging role for Ht: column hcol, k range hk0 .. hk0 + 3
  const int hcol = tid & 31, hk0 = (tid >> 5) * 4;
  const int cidx = c0 + hcol;
  const float* hsrc = nullptr;
  if (cidx < ncols) {
    const int tc = cidx / B, b = cidx % B;
    const int slot = (hc.t0 + tc) % hc.Tc;
    hsrc = hc.hist + (((int64_t)lane_id * hc.Tc + slot) * B + b) * (int64_t)H;
  }

  float acc[kHeadCols];
#pragma unroll
  for (int j = 0; j < kHeadCols; ++j) acc[j] = 0.f;

  for (int k0 = 0; k0 < H; k0 += kKc) {
    const int kc = min(kKc, H - k0);
    {
      const int64_t p = L.w_out + (int64_t)tid * H + k0;
      ProbeBits bits = {0u, 0u};
      if (pert) bits = probe_bits(pk, p, s.sparse);
#pragma unroll
      for (int k = 0; k < kKc; ++k)
        sm.g.Wt[k][tid] =
            (k < kc) ? perturb(th[p + k], (bits.neg >> k) & 1u, (bits.act >> k) & 1u, se) : 0.f;
    }
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const int k = hk0 + kk;
      sm.g.Ht[k][hcol] = (hsrc && k < kc) ? hsrc[k0 + k] : 0.f;
    }
    __syncthreads();
    for (int k = 0; k < kc; ++k) {
      const float w = sm.g.Wt[k][tid];
#pragma unroll
      for (int j4 = 0; j4 < kHeadCols / 4; ++j4) {
        const float4 h4 = *reinterpret_cast<const float4*>(&sm.g.Ht[k][j4 * 4]);
        acc[j4 * 4 + 0] = fmaf(w, h4.x, acc[j4 * 4 + 0]);
        acc[j4 * 4 + 1] = fmaf(w, h4.y, acc[j4 * 4 + 1]);
        acc[j4 * 4 + 2] = fmaf(w, h4.z, acc[j4 * 4 + 2]);
        acc[j4 * 4 + 3] = fmaf(w, h4.w, acc[j4 * 4 + 3]);
      }
    }
    __syncthreads();
  }
  {
    const int64_t p = L.b_out + tid;
    ProbeBits bit = {0u, 0u};
    if (pert) bit = probe_bits(pk, p, s.sparse);
    const float bo = perturb(th[p], bit.neg & 1u, bit.act & 1u, se);
#pragma unroll
    for (int j = 0; j < kHeadCols; ++j) sm.Lg[tid][j] = acc[j] + bo;
  }
  __syncthreads();

  // log-softmax and NLL: warp w handles columns 4w .. 4w + 3
  const int warp = tid >> 5, ln = tid & 31;
  for (int jj = 0; jj < 4; ++jj) {
    const int j = warp * 4 + jj;
    const int cidx2 = c0 + j;
    if (cidx2 >= ncols) break;
    float mx = -INFINITY;
#pragma unroll
    for (int r = 0; r < kVocab / 32; ++r) mx = fmaxf(mx, sm.Lg[ln + 32 * r][j]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float se_ = 0.f;
#pragma unroll
    for (int r = 0; r < kVocab / 32; ++r) se_ += expf(sm.Lg[ln + 32 * r][j] - mx);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) se_ += __shfl_xor_sync(0xffffffffu, se_, o);
    if (ln == 0) {
      const int tc = cidx2 / B, b = cidx2 % B;
      const int t = hc.t0 + tc;
      const int y = s.bytes[seq_offset(s, e, i, b) + t + 1];
      const float nll = (mx + logf(se_)) - sm.Lg[y][j];
      hc.nll[((int64_t)lane_id * B + b) * s.T + t] = nll;
    }
  }
}

}  // namespace

int forward_hist_slots(const Sweep& s) {
  // ring length of the h_t history: as many timesteps as fit in 2 GiB,
  // between 1 and 64
  const double per_slot = (double)s.lanes() * s.B * s.lay.H * sizeof(float);
  double cap = (2.0 * 1024 * 1024 * 1024) / per_slot;
  int tc = cap >= 64 ? 64 : (int)cap;
  if (tc < 1) tc = 1;
  if (tc > s.T) tc = s.T;
  return tc;
}

cudaError_t launch_forward_simt(const Sweep& s, const ForwardBuffers& fb, cudaStream_t stream) {
  const int Tc = fb.Tc;
  const int lanes = s.lanes();
  for (int t0 = 0; t0 < s.T; t0 += Tc) {
    const int nt = min(Tc, s.T - t0);
    for (int t = t0; t < t0 + nt; ++t) {
      GateStep g;
      g.sw = s;
      g.t = t;
      g.slot = t % Tc;
      g.prev_slot = (t + Tc - 1) % Tc;
      g.Tc = Tc;
      g.hist = fb.hist;
      g.cst = fb.cst;
      dim3 grid(lanes, (s.lay.H + kUnits - 1) / kUnits, (s.B + kCols - 1) / kCols);
      trace_begin(SOMA_TRACE_GATE, stream);
      gate_step_kernel<<<grid, 128, 0, stream>>>(g);
      trace_end(SOMA_TRACE_GATE, stream);
    }
    HeadChunk hc;
    hc.sw = s;
    hc.t0 = t0;
    hc.nt = nt;
    hc.Tc = Tc;
    hc.hist = fb.hist;
    hc.nll = fb.nll;
    dim3 grid(lanes, (nt * s.B + kHeadCols - 1) / kHeadCols);
    trace_begin(SOMA_TRACE_HEAD, stream);
    head_nll_kernel<<<grid, 256, 0, stream>>>(hc);
    trace_end(SOMA_TRACE_HEAD, stream);
  }
  return cudaGetLastError();
}

}  // namespace soma
