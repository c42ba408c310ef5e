// body_tc.cu -- the paper's expert body on the tensor cores (tcgen05 / TMEM).
//
// One CTA runs one (expert, probe) pair, both signs, over a chunk of up to 16
// sequences for all T timesteps, in the mean/difference form of the LSTM
// kernels applied to every linear layer.  With v+- = vbar +- dv (dv the half
// difference), its scaled form dhat = dv / eps, and the perturbed weights
// W +- eps Z:
//   (W +- eps Z)(vbar +- dv) = C +- eps D,  C = W vbar + eps^2 Z dhat,
//   D = W dhat + Z vbar,
// so one MMA of W and one of Z against the operand rows [vbar | dhat] give
// both signs.  dhat is O(1), so its fp16 rounding stays relative (2^-11) at
// any eps, where dv itself would fall into fp16's subnormal range.
// Everything between the linear layers (LayerNorm with perturbed gains, the
// LSTM cell, GELU, the residual stream, the decode's log-sum-exp) runs per
// sign in fp32 on the epilogue warps (the residual stream as fp32 mean and
// half difference), which write the next operand back as [vbar | dhat] in
// fp16.  The tied head E is not perturbed: its logits are E ybar +- eps E dhat_y.
//
// Per timestep and block (17 warps: 16 epilogue warps, one MMA warp; one
// barrier between phases):
//   LN_a -> [u | h] operand -> gates MMA (W_ih|W_hh, gate-major tile) -> cells
//   (state in registers; h and x updated) -> LN_b -> MLP1 MMA -> GELU -> the
//   MLP hidden operand -> MLP2 MMA (the hidden rows as the A operand,
//   W_2 as B) -> residual;
// then the final LN, the decode MMA (E, two 128-row tiles) and the NLL.
// The CTA's NLL sums per sign go to partial[(pair, sign)][chunk], which
// body_reduce_kernel (body.cu) turns into L+- and the coefficients.
//
// Precision.  With plain fp16 operands the losses were off by up to ~2e-4
// nats/byte and the coefficients by ~1-2% on small batches: the rounding of
// W and vbar shifts the model both signs see, and the LayerNorms pass the
// shift on.  So, except in the MLP's second layer:
//  - every operand value is split, v = hi + lo (both fp16), as four row
//    groups [vbar_hi | dhat_hi | vbar_lo | dhat_lo], so one W and one Z MMA
//    (N = 64) give both parts of both halves;
//  - W = W_hi + W_lo: W_hi in shared memory, W_lo in tensor memory as the A
//    operand of one more MMA (N = 32, the hi rows);
//  - the tied head likewise, E = E_hi + E_lo (E_lo in shared memory).
#include <cuda_fp16.h>

#define SOMA_CHECK_FILE 3
#include "checked.cuh"
#include "body_device.cuh"
#include "soma_device.cuh"
#include "soma_launch.h"
#include "tc_primitives.cuh"

namespace soma {

using namespace tc;

namespace {

constexpr int kD = kBodyWidth;  // 32
constexpr int kG = 4 * kD;      // 128
constexpr int kBp = kBodyRows;  // sequences per CTA (16)
constexpr int kN = 2 * kBp;     // operand rows [vbar | dhat] (hi parts; MLP2 operand)
constexpr int kNQ = 4 * kBp;    // operand rows [vbar_hi | dhat_hi | vbar_lo | dhat_lo]
constexpr int kEpiWarps = 16;
constexpr int kMmaWarp = kEpiWarps;
constexpr int kThreads = (kEpiWarps + 1) * 32;
constexpr uint32_t kLbo = 128;
constexpr float kLnEps = 1e-5f;

// Shared-memory layout (bytes, from a 1024-aligned base).
constexpr uint32_t kGateTile = 128u * 64 * 2;   // [W_ih | W_hh] gate-major, K = 64
constexpr uint32_t kMlp1Tile = 128u * 32 * 2;   // W_1, K = 32
constexpr uint32_t kMlp2Tile = 32u * 128 * 2;   // W_2 as the B operand: 32 rows, K = 128
                                                // (Z_2 right after it: one 64-row operand)
constexpr uint32_t kBlockBytes = 2 * (kGateTile + kMlp1Tile + kMlp2Tile);  // W and Z
constexpr uint32_t kSmBlk = 0;                                     // [D][W/Z tiles]
constexpr uint32_t kSmE = kSmBlk + kBodyMaxBlocks * kBlockBytes;   // E_hi, E_lo: [2][2 tiles][128][32]
constexpr uint32_t kSmO1 = kSmE + 4u * 128 * 32 * 2;              // [D] gate operands [NQ][64]
constexpr uint32_t kSmO2 = kSmO1 + kBodyMaxBlocks * kNQ * 64 * 2; // MLP1 operand [NQ][32]
constexpr uint32_t kSmO3 = kSmO2 + kNQ * 32 * 2;                  // MLP2 A operand [128][128]
constexpr uint32_t kSmO4 = kSmO3 + 128u * 128 * 2;                // decode operand [NQ][32]
constexpr uint32_t kSmX = kSmO4 + kNQ * 32 * 2;                   // xbar, dx fp32 [2][Bp][d]
constexpr uint32_t kSmGain = kSmX + 2u * kBp * kD * 4;            // gains [2 signs][(2D+1) d]
constexpr uint32_t kSmRed = kSmGain + 2u * (2 * kBodyMaxBlocks + 1) * kD * 4;  // [2][4][2][Bp] float2
constexpr uint32_t kSmYlog = kSmRed + 2u * 4 * 2 * kBp * 8;       // [2][Bp]
constexpr uint32_t kSmAcc = kSmYlog + 2u * kBp * 4;               // [2][Bp] double
constexpr uint32_t kSmCtl = kSmAcc + 2u * kBp * 8;                // mbarrier, tmem slot
constexpr uint32_t kSmBytes = kSmCtl + 64 + 1024;                 // + alignment slack
static_assert(kSmBytes <= 227 * 1024, "shared memory");
static_assert(kSmE % 1024 == 0 && kSmO1 % 16 == 0 && kSmO3 % 16 == 0 && kSmAcc % 8 == 0,
              "alignment");

// TMEM columns (each region starts at a multiple of 32): the W and Z
// accumulators of the current layer (gates, MLP1 or MLP2; 64 each); the
// decode halves, E_hi [ybar | dy] (64 each) and E_lo ybar_hi (16 each); the
// A operands W_lo of the gates (32 columns = K / 2) and of MLP1 (16) per block.
constexpr uint32_t kTW = 0, kTZ = 64, kTHead = 128, kTHeadLo = 256, kTWloGate = 320,
                   kTWloMlp1 = 384, kTmemCols = 512;

__device__ __forceinline__ float sigm_b(float x) { return __fdividef(1.0f, 1.0f + __expf(-x)); }

__device__ __forceinline__ float gelu_b(float a) {
  return 0.5f * a * (1.f + erff(a * 0.70710678118654752f));
}

__device__ __forceinline__ float wsum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

struct BodyTcArgs {
  const float* params;   // [N][P]
  const float* head;     // [V][d]
  const uint8_t* bytes;  // [N][B][T+1]
  double* partial;       // [N * n * n_sign][chunks]
  int* status;
  int n_pert, n_sign, blocks, B, T, chunks;
  int64_t P, goff;
  float eps;
  int sparse;
  uint64_t seed, step;
};

// fp16 +-1 / 0 probe values of coordinates p0 .. p0 + 7 (p0 % 8 == 0) and
// their weights, as two 16-byte chunks.
__device__ __forceinline__ void chunk8(const float* th, int64_t p0, int kmax, const ProbeKey& pk,
                                       const BodyTcArgs& a, bool do_z, uint4& wout, uint4& zout) {
  if (!SOMA_CHECK(p0 >= 0 && p0 + kmax <= a.P, a.status)) kmax = 0;  // inside the expert
  uint32_t neg = 0, act = 0;
  if (do_z && kmax > 0) {
    body_probe_words(pk, (int)(p0 >> 5), a.sparse, a.goff, neg, act);
    const int sh = (int)(p0 & 31);
    neg >>= sh;
    act >>= sh;
  }
  __align__(16) __half w[8], z[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const bool ok = j < kmax;
    w[j] = __float2half_rn(ok ? th[p0 + j] : 0.f);
    const bool on = ok && ((act >> j) & 1u);
    z[j] = __float2half_rn(on ? (((neg >> j) & 1u) ? -1.f : 1.f) : 0.f);
  }
  wout = *reinterpret_cast<const uint4*>(w);
  zout = *reinterpret_cast<const uint4*>(z);
}

// Operand rows of sequence b at column k (fp16): b <- hi(mean), Bp + b <-
// hi(dif), 2 Bp + b <- mean - hi(mean), 3 Bp + b <- dif - hi(dif).
__device__ __forceinline__ void store_split(uint8_t* op, int K, int b, int k, float mean,
                                            float dif) {
  const __half mh = __float2half_rn(mean), dh = __float2half_rn(dif);
  *reinterpret_cast<__half*>(op + kmajor_offset(b, k, K)) = mh;
  *reinterpret_cast<__half*>(op + kmajor_offset(kBp + b, k, K)) = dh;
  *reinterpret_cast<__half*>(op + kmajor_offset(2 * kBp + b, k, K)) =
      __float2half_rn(mean - __half2float(mh));
  *reinterpret_cast<__half*>(op + kmajor_offset(3 * kBp + b, k, K)) =
      __float2half_rn(dif - __half2float(dh));
}

// fp16 pair word (lo parts of w0, w1): the residual w - fp16(w) of each.
__device__ __forceinline__ uint32_t lo_pair(float w0, float w1) {
  const __half a = __float2half_rn(w0 - __half2float(__float2half_rn(w0)));
  const __half b = __float2half_rn(w1 - __half2float(__float2half_rn(w1)));
  return (uint32_t)__half_as_ushort(a) | ((uint32_t)__half_as_ushort(b) << 16);
}

// out rows b + {0, 1, 2, 3} Bp of a K-major operand with K columns, features at
// column offset k0: mean and scaled half difference (times inv_eps = 1 / eps,
// 0 when eps = 0) of the two signs' LN outputs.  Warp w runs sequence b = w
// (lane = feature).
__device__ __forceinline__ void ln_pair(const float* xbar, const float* dx, const float* gp,
                                        const float* gm, uint8_t* op, int K, int k0, int b,
                                        int lane, float inv_eps) {
  const float xb = xbar[b * kD + lane], d = dx[b * kD + lane];
  const float xp = xb + d, xm = xb - d;
  const float mp = wsum(xp) * (1.f / kD), mm = wsum(xm) * (1.f / kD);
  const float cp = xp - mp, cm = xm - mm;
  const float vp = wsum(cp * cp) * (1.f / kD), vm = wsum(cm * cm) * (1.f / kD);
  const float up = cp * rsqrtf(vp + kLnEps) * gp[lane];
  const float um = cm * rsqrtf(vm + kLnEps) * gm[lane];
  store_split(op, K, b, k0 + lane, 0.5f * (up + um), 0.5f * (up - um) * inv_eps);
}

// C and the half difference D of one layer for this thread's 16x128b view
// (TMEM lanes tq: rows 0, 1 of the view; tq2: rows 2, 3; column = the
// thread's sequence):
//   C = W (vbar_hi + vbar_lo) + eps^2 Z (dhat_hi + dhat_lo),
//   D = eps [W (dhat_hi + dhat_lo) + Z (vbar_hi + vbar_lo)],
// from the W accumulator (columns c + {0, 1, 2, 3} Bp; W_lo already added
// to the hi columns) and the Z accumulator.
__device__ __forceinline__ void layer_cd(uint32_t tq, uint32_t tq2, float eps, float (&C)[4],
                                         float (&D)[4]) {
  const float eps2 = eps * eps;
  uint32_t w[4][4], z[4][4];  // [row group][row of the view]
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    tmem_ld_16x128b(tq + g * kBp, w[g][0], w[g][1]);
    tmem_ld_16x128b(tq2 + g * kBp, w[g][2], w[g][3]);
    tmem_ld_16x128b(tq + kTZ + g * kBp, z[g][0], z[g][1]);
    tmem_ld_16x128b(tq2 + kTZ + g * kBp, z[g][2], z[g][3]);
  }
  tmem_wait_ld();
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float wv = __uint_as_float(w[0][k]) + __uint_as_float(w[2][k]);
    const float wd = __uint_as_float(w[1][k]) + __uint_as_float(w[3][k]);
    const float zv = __uint_as_float(z[0][k]) + __uint_as_float(z[2][k]);
    const float zd = __uint_as_float(z[1][k]) + __uint_as_float(z[3][k]);
    C[k] = fmaf(eps2, zd, wv);
    D[k] = eps * (wd + zv);
  }
}

__global__ void __launch_bounds__(kThreads, 1) body_tc_kernel(const BodyTcArgs a) {
  extern __shared__ uint8_t dyn_smem[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(dyn_smem) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int pair = blockIdx.x;
  const int e = pair / a.n_pert, i = pair % a.n_pert;
  const int chunk = blockIdx.y;
  // the CTA's sequences, its expert's parameters and its NLL partials lie
  // inside the caller's buffers (gridDim.x = N n pairs, gridDim.y = chunks)
  if (!SOMA_CHECK(chunk < a.chunks && chunk * kBp < a.B && pair < (int)gridDim.x, a.status))
    return;
  const int b0c = chunk * kBp;
  const int rows = min(kBp, a.B - b0c);
  const int D = a.blocks;
  const float eps = a.eps;
  const bool do_z = eps != 0.f;
  const float eps2 = eps * eps;
  const float inv_eps = do_z ? 1.f / eps : 0.f;  // the operand's difference rows are dv / eps
  const float* th = a.params + (int64_t)e * a.P;
  const ProbeKey pk = make_probe_key(a.seed, a.step, (uint32_t)e, (uint32_t)i);
  uint64_t* mma_bar = reinterpret_cast<uint64_t*>(smem + kSmCtl);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kSmCtl + 8);
  float* xbar = reinterpret_cast<float*>(smem + kSmX);
  float* dx = xbar + kBp * kD;
  float* gains = reinterpret_cast<float*>(smem + kSmGain);  // [sign][(2D+1) d]
  const int ng = (2 * kBodyMaxBlocks + 1) * kD;
  float2* red = reinterpret_cast<float2*>(smem + kSmRed);
  float* ylog = reinterpret_cast<float*>(smem + kSmYlog);
  double* acc = reinterpret_cast<double*>(smem + kSmAcc);

  if (tid == 0) {
    mbar_init(mma_bar, 1);
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(tmem_slot, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // ---- W_lo of the gates and MLP1 into tensor memory (A operands): the
  // thread of TMEM lane r (warps 0-3) writes row r, column c = k pair (2c, 2c+1)
  if (warp < 4) {
    const int r = 32 * warp + lane;
    const uint32_t trow = tmem + ((uint32_t)(32 * warp) << 16);
    for (int b = 0; b < D; ++b) {
      const int64_t base = (int64_t)b * 16 * kD * kD;
      const int64_t R = (int64_t)tile_gate(r) * kD + tile_unit(r);
      const float* wih = th + base + R * kD;
      const float* whh = th + base + 4 * kD * kD + R * kD;
      uint32_t pr[16];
#pragma unroll
      for (int c = 0; c < 16; ++c) pr[c] = lo_pair(wih[2 * c], wih[2 * c + 1]);
      tmem_st16(trow + kTWloGate + 32 * b, pr);
#pragma unroll
      for (int c = 0; c < 16; ++c) pr[c] = lo_pair(whh[2 * c], whh[2 * c + 1]);
      tmem_st16(trow + kTWloGate + 32 * b + 16, pr);
      const float* w1 = th + base + 8 * kD * kD + (int64_t)r * kD;
#pragma unroll
      for (int c = 0; c < 16; ++c) pr[c] = lo_pair(w1[2 * c], w1[2 * c + 1]);
      tmem_st16(trow + kTWloMlp1 + 32 * b, pr);
    }
    tmem_wait_st();
  }

  // ---- resident fp16 tiles of W and Z, and E ------------------------------
  for (int b = 0; b < D; ++b) {
    uint8_t* blk = smem + kSmBlk + b * kBlockBytes;
    const int64_t base = (int64_t)b * 16 * kD * kD;
    // gate tile: row r = gate (r / 8) % 4 of unit 8 (r / 32) + r % 8; K = [u | h]
    for (int c = tid; c < 128 * 8; c += kThreads) {
      const int r = c >> 3, k0 = 8 * (c & 7);
      const int64_t R = (int64_t)tile_gate(r) * kD + tile_unit(r);
      const int64_t p0 = k0 < kD ? base + R * kD + k0 : base + 4 * kD * kD + R * kD + (k0 - kD);
      uint4 w, z;
      chunk8(th, p0, 8, pk, a, do_z, w, z);
      const uint32_t off = kmajor_offset(r, k0, 64);
      *reinterpret_cast<uint4*>(blk + off) = w;
      *reinterpret_cast<uint4*>(blk + kGateTile + off) = z;
    }
    // W_1 [4d][d]
    for (int c = tid; c < 128 * 4; c += kThreads) {
      const int r = c >> 2, k0 = 8 * (c & 3);
      uint4 w, z;
      chunk8(th, base + 8 * kD * kD + (int64_t)r * kD + k0, 8, pk, a, do_z, w, z);
      const uint32_t off = kmajor_offset(r, k0, 32);
      *reinterpret_cast<uint4*>(blk + 2 * kGateTile + off) = w;
      *reinterpret_cast<uint4*>(blk + 2 * kGateTile + kMlp1Tile + off) = z;
    }
    // W_2 [d][4d] as the B operand: row j (output feature), K = 128
    for (int c = tid; c < 32 * 16; c += kThreads) {
      const int r = c >> 4, k0 = 8 * (c & 15);
      uint4 w, z;
      chunk8(th, base + 12 * kD * kD + (int64_t)r * kG + k0, 8, pk, a, do_z, w, z);
      const uint32_t off = kmajor_offset(r, k0, 128);
      *reinterpret_cast<uint4*>(blk + 2 * kGateTile + 2 * kMlp1Tile + off) = w;
      *reinterpret_cast<uint4*>(blk + 2 * kGateTile + 2 * kMlp1Tile + kMlp2Tile + off) = z;
    }
  }
  for (int c = tid; c < 256 * 4; c += kThreads) {  // E [256][32] = E_hi + E_lo, 128-row tiles
    const int v = c >> 2, k0 = 8 * (c & 3);
    __align__(16) __half w[8], wl[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float x = a.head[v * kD + k0 + j];
      w[j] = __float2half_rn(x);
      wl[j] = __float2half_rn(x - __half2float(w[j]));
    }
    const uint32_t off = (v >> 7) * (128u * 32 * 2) + kmajor_offset(v & 127, k0, 32);
    *reinterpret_cast<uint4*>(smem + kSmE + off) = *reinterpret_cast<const uint4*>(w);
    *reinterpret_cast<uint4*>(smem + kSmE + 2u * 128 * 32 * 2 + off) =
        *reinterpret_cast<const uint4*>(wl);
  }
  // perturbed gains per sign (dense probe signs on every gain)
  for (int k = tid; k < (2 * D + 1) * kD; k += kThreads) {
    const int64_t p = a.goff + k;
    float dz = 0.f;
    if (do_z) {
      uint32_t neg, act;
      body_probe_words(pk, (int)(p >> 5), a.sparse, a.goff, neg, act);
      const int j = (int)(p & 31);
      dz = ((act >> j) & 1u) ? (((neg >> j) & 1u) ? -eps : eps) : 0.f;
    }
    gains[k] = th[p] + dz;
    gains[ng + k] = th[p] - dz;
  }
  // operands: zero (the h parts start at h = 0; rows 2 Bp .. 127 of the MLP2
  // operand stay zero)
  for (uint32_t c = tid; c < (kSmX - kSmO1) / 16; c += kThreads)
    reinterpret_cast<uint4*>(smem + kSmO1)[c] = make_uint4(0u, 0u, 0u, 0u);
  for (int c = tid; c < 2 * kBp; c += kThreads) acc[c] = 0.0;

  fence_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  // descriptor words (low word: start address in 16-byte units)
  const uint32_t idesc32 = idesc_f16_f32(128, kN), idesc64 = idesc_f16_f32(128, kNQ),
                 idesc16 = idesc_f16_f32(128, kBp);
  const uint64_t d64 = smem_desc(smem_u32(smem), kLbo, 64 * 16);
  const uint64_t d32 = smem_desc(smem_u32(smem), kLbo, 32 * 16);
  const uint64_t d128 = smem_desc(smem_u32(smem), kLbo, 128 * 16);
  const uint32_t hi64 = (uint32_t)(d64 >> 32), hi32 = (uint32_t)(d32 >> 32),
                 hi128 = (uint32_t)(d128 >> 32);
  const uint32_t lo0 = (uint32_t)d64;  // smem base; same low word for every SBO
  auto lo = [&](uint32_t off) { return lo0 + (off >> 4); };

  // epilogue thread constants
  const int q4 = warp & 3, sg = warp >> 2;  // TMEM lane quarter; sequence group of 4
  const int u8 = lane >> 2, bq = lane & 3;
  const int bseq = 4 * sg + bq;               // sequence of the cell / MLP1 epilogues
  float cst[kBodyMaxBlocks][2];
#pragma unroll
  for (int b = 0; b < kBodyMaxBlocks; ++b) cst[b][0] = cst[b][1] = 0.f;
  // the byte row of warp w's sequence (rows past the batch read row 0)
  const int T1 = a.T + 1;
  const uint8_t* bx = a.bytes + ((int64_t)e * a.B + b0c) * T1;
  const uint8_t* my_row = bx + (int64_t)(warp < rows ? warp : 0) * T1;
  // loads a timestep ahead: the embedding of the next byte (warp = sequence,
  // lane = feature) and the decode targets of this thread's two sequences
  float emb = 0.f;
  if (warp < kEpiWarps) emb = a.head[(int)my_row[0] * kD + lane];
  int tgt[2];
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int b = 4 * (warp >> 3) + 8 * j + bq;
    tgt[j] = (int)bx[(int64_t)(b < rows ? b : 0) * T1 + 1];
  }

  uint32_t nph = 0;  // commits so far: the parity of the next wait
  bool fine = true, ok = true;
  auto mma_wait = [&]() {
    fine = mbar_wait(mma_bar, nph & 1u) && fine;
    ++nph;
    tc_fence_after();
  };
  auto phase_barrier = [&]() {
    fence_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
  };

  for (int t = 0; t < a.T && ok; ++t) {
    // ---- x = E[byte_t] (E is not perturbed: dx = 0) -----------------------
    if (warp < kEpiWarps) {
      xbar[warp * kD + lane] = emb;
      dx[warp * kD + lane] = 0.f;
      if (t + 1 < a.T) emb = a.head[(int)my_row[t + 1] * kD + lane];
    }
    __syncwarp();
#pragma unroll
    for (int b = 0; b < kBodyMaxBlocks; ++b) {
      if (b >= D) break;
      const uint32_t blk = kSmBlk + b * kBlockBytes;
      uint8_t* o1 = smem + kSmO1 + b * (kNQ * 64 * 2);
      // ---- LN_a -> u part of the gate operand ------------------------------
      if (warp < kEpiWarps)
        ln_pair(xbar, dx, gains + 2 * b * kD, gains + ng + 2 * b * kD, o1, 64, 0, warp, lane,
                inv_eps);
      phase_barrier();
      if (warp == kMmaWarp) {
        if (lane == 0) {
          const uint32_t ob = lo(kSmO1 + b * (kNQ * 64 * 2));
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16) {
            const uint32_t ko = 16u * k16, accf = k16 > 0;
            mma_f16_ss_lohi(tmem + kTW, lo(blk) + ko, hi64, ob + ko, hi64, idesc64, accf);
            mma_f16_ss_lohi(tmem + kTZ, lo(blk + kGateTile) + ko, hi64, ob + ko, hi64, idesc64,
                            accf);
            // W_lo [vbar_hi | dhat_hi], added to the hi columns
            mma_f16_ts_lohi(tmem + kTW, tmem + kTWloGate + 32 * b + 8 * k16, ob + ko, hi64,
                            idesc32, 1u);
          }
          mma_commit(mma_bar);
        }
        __syncwarp();
        ++nph;
      } else {
        mma_wait();
        // ---- cells: thread = unit 8 q4 + u8, sequence bseq -----------------
        const uint32_t tq = tmem + kTW + ((uint32_t)(32 * q4) << 16) + (uint32_t)(4 * sg);
        const uint32_t tq2 = tq + (16u << 16);
        float Cg[4], Dg[4];
        layer_cd(tq, tq2, eps, Cg, Dg);
        float ap[4], am[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float C = Cg[k], Dd = Dg[k];
          if (k == 2) {
            ap[k] = fmaf(sigm_b(2.f * (C + Dd)), 2.f, -1.f);
            am[k] = fmaf(sigm_b(2.f * (C - Dd)), 2.f, -1.f);
          } else {
            ap[k] = sigm_b(C + Dd);
            am[k] = sigm_b(C - Dd);
          }
        }
        const float cp = fmaf(ap[1], cst[b][0], ap[0] * ap[2]);
        const float cm = fmaf(am[1], cst[b][1], am[0] * am[2]);
        cst[b][0] = cp;
        cst[b][1] = cm;
        const float hp = ap[3] * fmaf(sigm_b(2.f * cp), 2.f, -1.f);
        const float hm = am[3] * fmaf(sigm_b(2.f * cm), 2.f, -1.f);
        const int U = 8 * q4 + u8;
        const float hb = 0.5f * (hp + hm), hd = 0.5f * (hp - hm);
        store_split(o1, 64, bseq, kD + U, hb, hd * inv_eps);
        xbar[bseq * kD + U] += hb;
        dx[bseq * kD + U] += hd;
      }
      phase_barrier();
      // ---- LN_b -> MLP1 operand ---------------------------------------------
      if (warp < kEpiWarps)
        ln_pair(xbar, dx, gains + 2 * b * kD + kD, gains + ng + 2 * b * kD + kD,
                smem + kSmO2, 32, 0, warp, lane, inv_eps);
      phase_barrier();
      if (warp == kMmaWarp) {
        if (lane == 0) {
          const uint32_t ob = lo(kSmO2);
#pragma unroll
          for (int k16 = 0; k16 < 2; ++k16) {
            const uint32_t ko = 16u * k16, accf = k16 > 0;
            mma_f16_ss_lohi(tmem + kTW, lo(blk + 2 * kGateTile) + ko, hi32, ob + ko, hi32,
                            idesc64, accf);
            mma_f16_ss_lohi(tmem + kTZ, lo(blk + 2 * kGateTile + kMlp1Tile) + ko, hi32, ob + ko,
                            hi32, idesc64, accf);
            mma_f16_ts_lohi(tmem + kTW, tmem + kTWloMlp1 + 32 * b + 8 * k16, ob + ko, hi32,
                            idesc32, 1u);
          }
          mma_commit(mma_bar);
        }
        __syncwarp();
        ++nph;
      } else {
        mma_wait();
        // ---- GELU: thread = features 32 q4 + u8 + {0, 8, 16, 24}, sequence bseq
        const uint32_t tq = tmem + kTW + ((uint32_t)(32 * q4) << 16) + (uint32_t)(4 * sg);
        const uint32_t tq2 = tq + (16u << 16);
        float Cg[4], Dg[4];
        layer_cd(tq, tq2, eps, Cg, Dg);
        uint8_t* o3 = smem + kSmO3;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int j = 32 * q4 + u8 + 8 * k;
          const float C = Cg[k], Dd = Dg[k];
          const float mp = gelu_b(C + Dd), mm = gelu_b(C - Dd);
          *reinterpret_cast<__half*>(o3 + kmajor_offset(bseq, j, 128)) =
              __float2half_rn(0.5f * (mp + mm));
          *reinterpret_cast<__half*>(o3 + kmajor_offset(kBp + bseq, j, 128)) =
              __float2half_rn(0.5f * (mp - mm) * inv_eps);
        }
      }
      phase_barrier();
      // ---- MLP2: [mbar | mhat] (rows) x [W_2 ; Z_2]^T ----------------------
      // W_2 and Z_2 are adjacent 32-row B tiles, i.e. one 64-row B operand:
      // one MMA of N = 64 gives W_2 m (columns 0-31) and Z_2 m (32-63)
      if (warp == kMmaWarp) {
        if (lane == 0) {
          const uint32_t oa = lo(kSmO3);
          const uint32_t wb = lo(blk + 2 * kGateTile + 2 * kMlp1Tile);
#pragma unroll
          for (int k16 = 0; k16 < 8; ++k16) {
            const uint32_t ko = 16u * k16, accf = k16 > 0;
            mma_f16_ss_lohi(tmem + kTW, oa + ko, hi128, wb + ko, hi128, idesc64, accf);
          }
          mma_commit(mma_bar);
        }
        __syncwarp();
        ++nph;
      } else {
        mma_wait();
        if (q4 == 0) {
          // lanes 0-15: rows mbar of sequences, 16-31: mhat; columns: features.
          // Warp 4 sg takes features 8 sg .. 8 sg + 7.
#pragma unroll
          for (int cg = 0; cg < 2; ++cg) {
            const uint32_t col = (uint32_t)(8 * sg + 4 * cg);
            const uint32_t tw = tmem + kTW + col, tz = tw + kD;
            uint32_t wm[2], wdd[2], zm[2], zdd[2];
            tmem_ld_16x128b(tw, wm[0], wm[1]);
            tmem_ld_16x128b(tw + (16u << 16), wdd[0], wdd[1]);
            tmem_ld_16x128b(tz, zm[0], zm[1]);
            tmem_ld_16x128b(tz + (16u << 16), zdd[0], zdd[1]);
            tmem_wait_ld();
            const int j = (int)col + bq;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int s = u8 + 8 * h;  // sequence
              const float C = fmaf(eps2, __uint_as_float(zdd[h]), __uint_as_float(wm[h]));
              const float Dd = eps * (__uint_as_float(wdd[h]) + __uint_as_float(zm[h]));
              xbar[s * kD + j] += C;
              dx[s * kD + j] += Dd;
            }
          }
        }
      }
      phase_barrier();
    }

    // ---- y = LN(x) gf -> decode operand; logits = E y ---------------------
    if (warp < kEpiWarps)
      ln_pair(xbar, dx, gains + 2 * D * kD, gains + ng + 2 * D * kD, smem + kSmO4, 32, 0, warp,
              lane, inv_eps);
    phase_barrier();
    if (warp == kMmaWarp) {
      if (lane == 0) {
        const uint32_t ob = lo(kSmO4);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
#pragma unroll
          for (int k16 = 0; k16 < 2; ++k16) {
            const uint32_t ko = 16u * k16, accf = k16 > 0;
            const uint32_t ea = lo(kSmE + h * (128u * 32 * 2)) + ko;
            mma_f16_ss_lohi(tmem + kTHead + h * 64, ea, hi32, ob + ko, hi32, idesc64, accf);
            mma_f16_ss_lohi(tmem + kTHeadLo + h * 32, ea + ((2u * 128 * 32 * 2) >> 4), hi32,
                            ob + ko, hi32, idesc16, accf);  // E_lo ybar_hi
          }
        }
        mma_commit(mma_bar);
      }
      __syncwarp();
      ++nph;
    } else {
      mma_wait();
      // warp: vocabulary half (w / 4) % 2, quarter w % 4, sequences 4 (w / 8) + 8 j + l % 4;
      // thread l holds rows l / 4 + 8 k (k = 0..3) of the quarter
      const int half = (warp >> 2) & 1, sp = warp >> 3, r4 = lane >> 2;
      const int vq = 128 * half + 32 * q4;
      const uint32_t tq = tmem + kTHead + half * 64 + ((uint32_t)(32 * q4) << 16);
      const uint32_t tq2 = tq + (16u << 16);
      const uint32_t tlo = tmem + kTHeadLo + half * 32 + ((uint32_t)(32 * q4) << 16);
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int b0 = 4 * sp + 8 * j;
        // E_hi times the four row groups, and E_lo ybar_hi
        uint32_t yq[4][4], ye[4];
#pragma unroll
        for (int g = 0; g < 4; ++g) {
          tmem_ld_16x128b(tq + g * kBp + b0, yq[g][0], yq[g][1]);
          tmem_ld_16x128b(tq2 + g * kBp + b0, yq[g][2], yq[g][3]);
        }
        tmem_ld_16x128b(tlo + b0, ye[0], ye[1]);
        tmem_ld_16x128b(tlo + (16u << 16) + b0, ye[2], ye[3]);
        tmem_wait_ld();
        float lp[4], lm[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float C = __uint_as_float(yq[0][k]) +
                          (__uint_as_float(yq[2][k]) + __uint_as_float(ye[k]));
          const float Dh = eps * (__uint_as_float(yq[1][k]) + __uint_as_float(yq[3][k]));
          lp[k] = C + Dh;
          lm[k] = C - Dh;
        }
        float mp = fmaxf(fmaxf(lp[0], lp[1]), fmaxf(lp[2], lp[3]));
        float mm = fmaxf(fmaxf(lm[0], lm[1]), fmaxf(lm[2], lm[3]));
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
          mp = fmaxf(mp, __shfl_xor_sync(0xffffffffu, mp, o));
          mm = fmaxf(mm, __shfl_xor_sync(0xffffffffu, mm, o));
        }
        float sp_ = 0.f, sm_ = 0.f;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          sp_ += __expf(lp[k] - mp);
          sm_ += __expf(lm[k] - mm);
        }
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
          sp_ += __shfl_xor_sync(0xffffffffu, sp_, o);
          sm_ += __shfl_xor_sync(0xffffffffu, sm_, o);
        }
        const int b = b0 + bq;
        if (r4 == 0) {
          red[((half * 4 + q4) * 2 + 0) * kBp + b] = make_float2(mp, sp_);
          red[((half * 4 + q4) * 2 + 1) * kBp + b] = make_float2(mm, sm_);
        }
        const int y = tgt[j] - vq - r4;  // byte t + 1
        if (t + 2 <= a.T) tgt[j] = (int)bx[(int64_t)(b < rows ? b : 0) * T1 + t + 2];
        if (y >= 0 && y < 32 && (y & 7) == 0) {
          const int k = y >> 3;
          ylog[b] = k == 0 ? lp[0] : k == 1 ? lp[1] : k == 2 ? lp[2] : lp[3];
          ylog[kBp + b] = k == 0 ? lm[0] : k == 1 ? lm[1] : k == 2 ? lm[2] : lm[3];
        }
      }
      asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
      if (tid < rows) {
#pragma unroll
        for (int s = 0; s < 2; ++s) {
          float M = -INFINITY;
          for (int h = 0; h < 8; ++h) M = fmaxf(M, red[(h * 2 + s) * kBp + tid].x);
          float S = 0.f;
          for (int h = 0; h < 8; ++h) {
            const float2 q = red[(h * 2 + s) * kBp + tid];
            S += q.y * __expf(q.x - M);
          }
          acc[s * kBp + tid] += (double)(M + logf(S) - ylog[s * kBp + tid]);
        }
      }
    }
    if (!fine) atomicCAS(a.status, 0, kStatusTimeout);
    tc_fence_before();
    ok = (__syncthreads_and(fine) != 0) && ok;
    tc_fence_after();
  }

  // ---- the CTA's NLL sums per sign (sequences in order) -------------------
  if (tid < a.n_sign) {
    double tot = 0.0;
    for (int b = 0; b < rows; ++b) tot += acc[tid * kBp + b];
    if (SOMA_CHECK(((int64_t)pair * a.n_sign + tid) * a.chunks + chunk <
                       (int64_t)gridDim.x * a.n_sign * a.chunks,
                   a.status))
      a.partial[((int64_t)pair * a.n_sign + tid) * a.chunks + chunk] = tot;
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, kTmemCols);
}

}  // namespace

cudaError_t launch_body_tc(const float* params, const float* head, const uint8_t* bytes,
                           int n_experts, int blocks, int n_pert, int n_sign, int B, int T,
                           float eps, int sparse, uint64_t seed, uint64_t step, double* partial,
                           int* status, cudaStream_t stream) {
  BodyTcArgs a;
  a.params = params;
  a.head = head;
  a.bytes = bytes;
  a.partial = partial;
  a.status = status;
  a.n_pert = n_pert;
  a.n_sign = n_sign;
  a.blocks = blocks;
  a.B = B;
  a.T = T;
  a.chunks = (B + kBp - 1) / kBp;
  a.P = body_param_count(kD, blocks);
  a.goff = body_gain_offset(kD, blocks);
  a.eps = eps;
  a.sparse = sparse;
  a.seed = seed;
  a.step = step;
  cudaError_t err = cudaFuncSetAttribute(body_tc_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSmBytes);
  if (err != cudaSuccess) return err;
  dim3 grid((unsigned)((int64_t)n_experts * n_pert), (unsigned)a.chunks);
  trace_begin(SOMA_TRACE_GATE, stream);
  body_tc_kernel<<<grid, kThreads, kSmBytes, stream>>>(a);
  trace_end(SOMA_TRACE_GATE, stream);
  return cudaGetLastError();
}

}  // namespace soma
