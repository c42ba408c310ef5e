// resident.cu -- the SPSA forward of small experts with the whole recurrence
// resident in one CTA (tcgen05 / TMEM).
//
// One CTA runs one (expert, probe) pair, both signs, over all T timesteps in
// the mean/difference form of forward_tc.cu, with the difference operand
// scaled by 1 / eps (dhat = dv / eps, an O(1) quantity):
//   a+- = C +- eps D,  C = W vbar + eps^2 (Z dhat) + b,  D = W dhat + Z vbar + z_b.
// The gate weights W = [W_ih | W_hh], the head weights W_out and the probe
// tiles Z of this pair are converted to fp16 tiles in shared memory once,
// and the probes are therefore drawn once per step, not once per timestep.
// The operand [vbar | dhat] (rows) x [x | h] (K) also lives in shared memory,
// in two buffers: buffer t % 2 holds [x_t | h_{t-1}].  Cell states stay in
// registers, and the losses are summed in the CTA.  Per timestep t, after
// the barrier that publishes buffer t % 2:
//   MMA warp   gate(t) (commit), then head(t - 1) into head accumulator
//              (t - 1) % 2 (its own commit barrier), both reading buffer t % 2;
//   epilogues  head epilogue of t - 1 (max / sum-exp per (sequence, sign)
//              over both vocabulary halves, target logit, NLL summed in fp64)
//              while the gate MMAs of t run; then the gate epilogue of t
//              (gates and cells), which writes h_t and the embedding of
//              t + 1 into buffer (t + 1) % 2; then the barrier.
// The head epilogue, the longest phase, thus overlaps the next gate MMAs,
// and the serial chain of a timestep is gate MMAs -> gate epilogue.
// The shape limits (H <= 64, B <= 32, 2 Bp Ek / 8 <= 256 operand chunks, the
// tiles within shared memory, (MT + 4) 4 Bp <= 512 TMEM columns) are checked
// by res_supported(); other experts use the persistent kernel.
#include <cuda_fp16.h>

#define SOMA_CHECK_FILE 2
#include "checked.cuh"
#include "soma_api.h"
#include "soma_device.cuh"
#include "soma_launch.h"
#include "tc_primitives.cuh"

namespace soma {

using namespace tc;

namespace {

constexpr int kResEpiWarps = 16;  // (two M tiles x four TMEM lane quarters) x two halves
                                   // of the sequences
constexpr int kResMmaWarp = kResEpiWarps;  // issues the MMAs and takes no epilogue work
constexpr int kResThreads = (kResEpiWarps + 1) * 32;
constexpr int kResMaxBp = 32;
constexpr size_t kResMaxSmem = 220 * 1024;
constexpr uint32_t kLboRes = 128;  // bytes between core matrices along K

__device__ __forceinline__ float sigm_res(float x) { return __fdividef(1.0f, 1.0f + __expf(-x)); }

struct ResGeom {
  int E, H, Ek, Hk, K, MTg, Bp, B, T;
  uint32_t wg, zg, wo, zo, op, opsz, emb, dx, red, ylog, acc, ctl, bytes;  // shared-memory offsets
  uint32_t tmem_cols;
};

__host__ __device__ inline uint32_t res_align(uint32_t x) { return (x + 1023u) & ~1023u; }

ResGeom make_res_geom(const Layout& lay, int B, int T) {
  ResGeom r;
  r.E = lay.E;
  r.H = lay.H;
  r.Ek = (lay.E + 15) / 16 * 16;
  r.Hk = (lay.H + 15) / 16 * 16;
  r.K = r.Ek + r.Hk;
  r.MTg = (lay.H + 31) / 32;
  r.Bp = (B + 7) / 8 * 8;
  r.B = B;
  r.T = T;
  uint32_t o = 0;
  const uint32_t gate_tile = 128u * r.K * 2, head_tile = 128u * r.Hk * 2;
  r.wg = o; o = res_align(o + r.MTg * gate_tile);
  r.zg = o; o = res_align(o + r.MTg * gate_tile);
  r.wo = o; o = res_align(o + 2 * head_tile);
  r.zo = o; o = res_align(o + 2 * head_tile);
  r.opsz = 2u * r.Bp * r.K * 2;  // one operand buffer [vbar | dhat] x K, fp16
  r.op = o; o = res_align(o + 2u * r.opsz);
  r.emb = o; o += 256u * r.Ek * 2;   // fp16 Emb rows [V][Ek]
  r.dx = o; o += 256u * r.Ek * 2;    // fp16 z of the Emb rows (dhat of x = z_emb)
  r.red = o; o += 2u * 4 * 2 * r.Bp * sizeof(float2);  // [half][quarter][sign][Bp]
  r.ylog = o; o += 2u * r.Bp * sizeof(float);          // [sign][Bp]
  o = (o + 7u) & ~7u;
  r.acc = o; o += 3u * r.Bp * sizeof(double);          // per sequence: sum nll+, nll-, diff
  o = (o + 7u) & ~7u;
  r.ctl = o; o += 64;
  r.bytes = o + 1024;  // alignment slack of the dynamic shared-memory base
  // gate accumulators, then two head accumulators (4 Bp columns per tile)
  const uint32_t cols = (uint32_t)(r.MTg + 4) * 4 * r.Bp;
  r.tmem_cols = 32;
  while (r.tmem_cols < cols) r.tmem_cols <<= 1;
  return r;
}

struct ResArgs {
  Sweep sw;
  ResGeom g;
  int n_sign;         // 2: (L+, L-) per pair; 1: L per expert (eps = 0)
  float* losses_out;  // [N][n][2] or [N]
  float* coef_out;    // [N][n] or null
  float* coef_ws;     // [N][n] or null
  int* status;
  size_t n_params, n_bytes;  // extents for the index checks of the checked build
};

// z of flat parameter p as an fp16 +-1 / 0 (sparse) value.
__device__ __forceinline__ __half z_half(const ProbeBits& b, int j) {
  return ((b.act >> j) & 1u) ? (((b.neg >> j) & 1u) ? __float2half_rn(-1.f) : __float2half_rn(1.f))
                             : __float2half_rn(0.f);
}

__global__ void __launch_bounds__(kResThreads, 1) res_kernel(const ResArgs a) {
  extern __shared__ uint8_t dyn_smem[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(dyn_smem) + 1023) & ~uintptr_t(1023));
  const ResGeom& g = a.g;
  const Sweep& s = a.sw;
  const Layout& L = s.lay;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int e = blockIdx.x / s.n_pert, i = blockIdx.x % s.n_pert;
  const float* th = s.params + (int64_t)e * L.P;
  const ProbeKey pk = make_probe_key(s.seed, s.step, (uint32_t)e, (uint32_t)i);
  const float eps = s.eps;
  const bool do_z = eps != 0.f;
  const float eps2 = eps * eps;
  // dhat_h = (h+ - h-) / (2 eps); 0 when eps = 0 (both signs coincide)
  const float half_inv_eps = do_z ? 0.5f / eps : 0.f;
  uint64_t* gate_bar = reinterpret_cast<uint64_t*>(smem + g.ctl);
  uint64_t* head_bar = reinterpret_cast<uint64_t*>(smem + g.ctl + 8);  // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + g.ctl + 24);
  float2* red = reinterpret_cast<float2*>(smem + g.red);
  float* ylog = reinterpret_cast<float*>(smem + g.ylog);
  double* acc = reinterpret_cast<double*>(smem + g.acc);

  if (tid == 0) {
    mbar_init(gate_bar, 1);
    mbar_init(head_bar, 1);
    mbar_init(head_bar + 1, 1);
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(tmem_slot, g.tmem_cols);

  // ---- resident tiles: W, Z of the gate (gate-major quarters) and the head
  const int gate_chunks = g.MTg * 128 * (g.K / 8);
  for (int c = tid; c < gate_chunks; c += kResThreads) {
    const int m = c / (128 * (g.K / 8)), rem = c % (128 * (g.K / 8));
    const int r = rem / (g.K / 8), k0 = 8 * (rem % (g.K / 8));
    const int U = 32 * m + tile_unit(r);
    const int64_t R = (int64_t)tile_gate(r) * g.H + U;
    __align__(16) __half w[8], z[8];
    int64_t p0 = -1;
    int kmax = 0;  // valid columns of this chunk
    if (U < g.H) {
      if (k0 < g.Ek) {
        p0 = L.w_ih + R * g.E + k0;
        kmax = min(8, g.E - k0);
      } else {
        p0 = L.w_hh + R * g.H + (k0 - g.Ek);
        kmax = min(8, g.H - (k0 - g.Ek));
      }
    }
    ProbeBits zb = {0u, 0u};
    if (kmax > 0 && do_z) zb = probe_bits(pk, p0, s.sparse);
    if (kmax > 0 && !SOMA_CHECK((size_t)(e * L.P + p0 + kmax) <= a.n_params, a.status)) kmax = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const bool ok = j < kmax;
      w[j] = __float2half_rn(ok ? th[p0 + j] : 0.f);
      z[j] = ok ? z_half(zb, j) : __float2half_rn(0.f);
    }
    const uint32_t off = m * (128u * g.K * 2) + kmajor_offset(r, k0, g.K);
    if (SOMA_CHECK(off + 16 <= g.MTg * 128u * g.K * 2 && g.zg + off + 16 <= g.bytes, a.status)) {
      *reinterpret_cast<uint4*>(smem + g.wg + off) = *reinterpret_cast<const uint4*>(w);
      *reinterpret_cast<uint4*>(smem + g.zg + off) = *reinterpret_cast<const uint4*>(z);
    }
  }
  const int head_chunks = 2 * 128 * (g.Hk / 8);
  for (int c = tid; c < head_chunks; c += kResThreads) {
    const int h = c / (128 * (g.Hk / 8)), rem = c % (128 * (g.Hk / 8));
    const int r = rem / (g.Hk / 8), k0 = 8 * (rem % (g.Hk / 8));
    const int64_t p0 = L.w_out + (int64_t)(128 * h + r) * g.H + k0;
    int kmax = min(8, g.H - k0);
    if (kmax > 0 && !SOMA_CHECK((size_t)(e * L.P + p0 + kmax) <= a.n_params, a.status)) kmax = 0;
    ProbeBits zb = {0u, 0u};
    if (kmax > 0 && do_z) zb = probe_bits(pk, p0, s.sparse);
    __align__(16) __half w[8], z[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const bool ok = j < kmax;
      w[j] = __float2half_rn(ok ? th[p0 + j] : 0.f);
      z[j] = ok ? z_half(zb, j) : __float2half_rn(0.f);
    }
    const uint32_t off = h * (128u * g.Hk * 2) + kmajor_offset(r, k0, g.Hk);
    if (SOMA_CHECK(off + 16 <= 2u * 128u * g.Hk * 2 && g.zo + off + 16 <= g.bytes, a.status)) {
      *reinterpret_cast<uint4*>(smem + g.wo + off) = *reinterpret_cast<const uint4*>(w);
      *reinterpret_cast<uint4*>(smem + g.zo + off) = *reinterpret_cast<const uint4*>(z);
    }
  }
  for (int c = tid; c < 2 * (2 * g.Bp * g.K / 8); c += kResThreads)
    reinterpret_cast<uint4*>(smem + g.op)[c] = make_uint4(0u, 0u, 0u, 0u);
  // the embedding table and its probe z (the scaled difference of the two
  // signs' inputs, dhat_x = (x+ - x-) / (2 eps) = z_emb), so that the operand
  // of a timestep is gathered from shared memory
  for (int c = tid; c < 256 * (g.Ek / 8); c += kResThreads) {
    const int v = c / (g.Ek / 8), k0 = 8 * (c % (g.Ek / 8));
    const int64_t p0 = L.emb + (int64_t)v * g.E + k0;
    const int kmax = min(8, g.E - k0);
    ProbeBits zb = {0u, 0u};
    if (do_z && kmax > 0) zb = probe_bits(pk, p0, s.sparse);
    __align__(16) __half x[8], d[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const bool ok = j < kmax;
      x[j] = __float2half_rn(ok ? th[p0 + j] : 0.f);
      d[j] = ok ? z_half(zb, j) : __float2half_rn(0.f);
    }
    reinterpret_cast<uint4*>(smem + g.emb)[c] = *reinterpret_cast<const uint4*>(x);
    reinterpret_cast<uint4*>(smem + g.dx)[c] = *reinterpret_cast<const uint4*>(d);
  }
  for (int c = tid; c < 3 * g.Bp; c += kResThreads) acc[c] = 0.0;

  // ---- per-thread constants of the epilogues
  // gate: warp w runs tile (w / 4) % 2, TMEM lane quarter w % 4, and the
  // 8-sequence chunks c with c % 2 == w / 8; thread l owns unit 8 (w % 4) +
  // l / 4 of that tile and sequences 8c + l % 4, 8c + 4 + l % 4
  const int q4 = warp & 3, tile = (warp >> 2) & 1, sp = warp >> 3;
  const int u8 = lane >> 2, bq = lane & 3;
  const int U = 32 * tile + 8 * q4 + u8;
  const bool unit_ok = tile < g.MTg && U < g.H;
  float bias[4] = {0.f, 0.f, 0.f, 0.f}, dbias[4] = {0.f, 0.f, 0.f, 0.f};
  if (unit_ok) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int64_t pb = L.b + (int64_t)k * g.H + U;
      bias[k] = th[pb];
      if (do_z) {
        const ProbeBits zb = probe_bits(pk, pb, s.sparse);
        dbias[k] = eps_z(zb.neg & 1u, zb.act & 1u, eps);
      }
    }
  }
  float cst[kResMaxBp / 8][2][2];  // [chunk][sequence half][sign]
#pragma unroll
  for (int c = 0; c < kResMaxBp / 8; ++c)
    cst[c][0][0] = cst[c][0][1] = cst[c][1][0] = cst[c][1][1] = 0.f;
  // head: warp w runs vocabulary half (w / 4) % 2, quarter w % 4, and the
  // 4-sequence groups 4 (w / 8) + 8 j; thread l holds rows l / 4 + 8 k
  // (k = 0..3) of the quarter
  const int half = (warp >> 2) & 1, r4 = lane >> 2;
  const int vq = 128 * half + 32 * q4;
  float bo[4], dbo[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int64_t pb = L.b_out + vq + r4 + 8 * k;
    bo[k] = th[pb];
    dbo[k] = 0.f;
    if (do_z) {
      const ProbeBits zb = probe_bits(pk, pb, s.sparse);
      dbo[k] = eps_z(zb.neg & 1u, zb.act & 1u, eps);
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t gcol0 = 0, hcol0 = (uint32_t)g.MTg * 4 * g.Bp;
  // MMA descriptors as 32-bit words: the low word holds the start address in
  // 16-byte units, so a step along K (256 bytes) or to the next tile is an
  // addition; gate tiles and the operand share their high word (SBO = 16 K)
  const uint32_t n2 = (uint32_t)(2 * g.Bp);
  const uint32_t idesc = idesc_f16_f32(128, 2 * g.Bp);
  const uint64_t dg = smem_desc(smem_u32(smem + g.wg), kLboRes, (uint32_t)g.K * 16);
  const uint64_t dh = smem_desc(smem_u32(smem + g.wo), kLboRes, (uint32_t)g.Hk * 16);
  const uint32_t ghi = (uint32_t)(dg >> 32), wg_lo = (uint32_t)dg;
  const uint32_t hhi = (uint32_t)(dh >> 32), wo_lo = (uint32_t)dh;
  const uint32_t zg_lo = wg_lo + ((g.zg - g.wg) >> 4), op_lo = wg_lo + ((g.op - g.wg) >> 4);
  const uint32_t zo_lo = wo_lo + ((g.zo - g.wo) >> 4);
  const uint32_t gstep = 16u * g.K, hstep = 16u * g.Hk;  // one 128-row tile, in 16-byte units
  bool ok = true;
  // the operand chunk this thread gathers every timestep (one row, 8 columns)
  const int xc = (warp < kResEpiWarps && tid < 2 * g.Bp * (g.Ek / 8)) ? tid : -1;
  const int xrow = xc / (g.Ek / 8), xk0 = 8 * (xc % (g.Ek / 8));
  const bool x_delta = xrow >= g.Bp;
  const int xb = x_delta ? xrow - g.Bp : xrow;
  const uint4* xtab = reinterpret_cast<const uint4*>(smem + (x_delta ? g.dx : g.emb));
  // the embedding part of operand buffer 0 (x_0; h_{-1} = 0): rows
  // [vbar (Bp) | dhat (Bp)], 16-byte chunks of the Emb / z tables
  int ynext = 0;
  if (xc >= 0 && xb < g.B) {
    const int y0 = s.bytes[seq_offset(s, e, i, xb)];
    *reinterpret_cast<uint4*>(smem + g.op + kmajor_offset(xrow, xk0, g.K)) =
        xtab[y0 * (g.Ek / 8) + xk0 / 8];
    if (g.T > 1) ynext = s.bytes[seq_offset(s, e, i, xb) + 1];
  }
  fence_async_smem();
  tc_fence_before();
  __syncthreads();

  // A failed wait marks this thread; the decision is taken for the whole CTA
  // at the barrier that ends the timestep.  Every warp reaches every barrier
  // whatever its waits returned (a wait that times out returns false).
  bool fine = true;
  for (int t = 0; t <= g.T && ok; ++t) {
    const uint32_t cur = (uint32_t)(t & 1), nxt = cur ^ 1u;
    if (warp == kResMmaWarp) {
      if (lane == 0) {
        tc_fence_after();
        const uint32_t ob = op_lo + cur * (g.opsz >> 4);  // operand buffer t % 2
        if (!SOMA_CHECK(hcol0 + 8u * g.Bp <= g.tmem_cols && gcol0 + g.MTg * 4u * g.Bp <= hcol0,
                        a.status)) {
          // columns outside the allocation: no MMA; the epilogue waits time out
        } else if (t < g.T) {  // gate of t: [x_t | h_{t-1}]
#pragma unroll 1
          for (int m = 0; m < g.MTg; ++m) {
            const uint32_t d = tmem + gcol0 + (uint32_t)m * 2 * n2;
            const uint32_t wlo = wg_lo + (uint32_t)m * gstep, zlo = zg_lo + (uint32_t)m * gstep;
            for (int k16 = 0; k16 < g.K / 16; ++k16) {
              const uint32_t ko = (uint32_t)k16 * 16, acc_flag = k16 > 0 ? 1u : 0u;
              mma_f16_ss_lohi(d, wlo + ko, ghi, ob + ko, ghi, idesc, acc_flag);
              mma_f16_ss_lohi(d + n2, zlo + ko, ghi, ob + ko, ghi, idesc, acc_flag);
            }
          }
          mma_commit(gate_bar);
        }
        if (t >= 1) {  // head of t - 1: the h part, h_{t-1}, into accumulator (t - 1) % 2
          const uint32_t hb = (uint32_t)((t - 1) & 1);
          const uint32_t obh = ob + (uint32_t)g.Ek;  // Ek / 8 core matrices further
#pragma unroll 1
          for (int h = 0; h < 2; ++h) {
            const uint32_t d = tmem + hcol0 + hb * 4 * n2 + (uint32_t)h * 2 * n2;
            const uint32_t wlo = wo_lo + (uint32_t)h * hstep, zlo = zo_lo + (uint32_t)h * hstep;
            for (int k16 = 0; k16 < g.Hk / 16; ++k16) {
              const uint32_t ko = (uint32_t)k16 * 16, acc_flag = k16 > 0 ? 1u : 0u;
              mma_f16_ss_lohi(d, wlo + ko, hhi, obh + ko, ghi, idesc, acc_flag);
              mma_f16_ss_lohi(d + n2, zlo + ko, hhi, obh + ko, ghi, idesc, acc_flag);
            }
          }
          mma_commit(head_bar + hb);
        }
      }
      __syncwarp();
    }

    if (t < g.T && warp < kResEpiWarps) {
      fine = mbar_wait(gate_bar, (uint32_t)t & 1u) && fine;
      tc_fence_after();
      if (tile < g.MTg) {
        const uint32_t tq = tmem + gcol0 + (uint32_t)tile * 4 * g.Bp + ((uint32_t)(32 * q4) << 16);
        const uint32_t tq2 = tq + (16u << 16);
#pragma unroll
        for (int c = 0; c < kResMaxBp / 8; ++c) {
          const int b0 = 8 * c;
          if (b0 >= g.Bp) break;
          if ((c & 1) != sp) continue;
          uint32_t wv[2][4], wd[2][4], zv[2][4], zd[2][4];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const uint32_t cw = (uint32_t)(b0 + 4 * h);
            tmem_ld_16x128b(tq + cw, wv[h][0], wv[h][1]);
            tmem_ld_16x128b(tq2 + cw, wv[h][2], wv[h][3]);
            tmem_ld_16x128b(tq + cw + g.Bp, wd[h][0], wd[h][1]);
            tmem_ld_16x128b(tq2 + cw + g.Bp, wd[h][2], wd[h][3]);
            tmem_ld_16x128b(tq + 2 * g.Bp + cw, zv[h][0], zv[h][1]);
            tmem_ld_16x128b(tq2 + 2 * g.Bp + cw, zv[h][2], zv[h][3]);
            tmem_ld_16x128b(tq + 3 * g.Bp + cw, zd[h][0], zd[h][1]);
            tmem_ld_16x128b(tq2 + 3 * g.Bp + cw, zd[h][2], zd[h][3]);
          }
          tmem_wait_ld();
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            float actp[4], actm[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const float C = fmaf(eps2, __uint_as_float(zd[h][k]), __uint_as_float(wv[h][k])) + bias[k];
              const float D = fmaf(eps, __uint_as_float(wd[h][k]) + __uint_as_float(zv[h][k]), dbias[k]);
              if (k == 2) {
                actp[k] = fmaf(sigm_res(2.f * (C + D)), 2.f, -1.f);
                actm[k] = fmaf(sigm_res(2.f * (C - D)), 2.f, -1.f);
              } else {
                actp[k] = sigm_res(C + D);
                actm[k] = sigm_res(C - D);
              }
            }
            const float cp = fmaf(actp[1], cst[c][h][0], actp[0] * actp[2]);
            const float cm = fmaf(actm[1], cst[c][h][1], actm[0] * actm[2]);
            cst[c][h][0] = cp;
            cst[c][h][1] = cm;
            const float hp = actp[3] * fmaf(sigm_res(2.f * cp), 2.f, -1.f);
            const float hm = actm[3] * fmaf(sigm_res(2.f * cm), 2.f, -1.f);
            const int b = b0 + 4 * h + bq;
            if (unit_ok && b < g.B &&
                SOMA_CHECK(kmajor_offset(g.Bp + b, g.Ek + U, g.K) + 2 <= g.opsz, a.status)) {
              *reinterpret_cast<__half*>(smem + g.op + nxt * g.opsz + kmajor_offset(b, g.Ek + U, g.K)) =
                  __float2half_rn(0.5f * (hp + hm));
              *reinterpret_cast<__half*>(smem + g.op + nxt * g.opsz + kmajor_offset(g.Bp + b, g.Ek + U, g.K)) =
                  __float2half_rn((hp - hm) * half_inv_eps);
            }
          }
        }
      }
      // the embedding part of buffer (t + 1) % 2
      if (t + 1 < g.T && xc >= 0) {
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (xb < g.B) v = xtab[ynext * (g.Ek / 8) + xk0 / 8];
        *reinterpret_cast<uint4*>(smem + g.op + nxt * g.opsz + kmajor_offset(xrow, xk0, g.K)) = v;
        if (xb < g.B && t + 2 < g.T) ynext = s.bytes[seq_offset(s, e, i, xb) + t + 2];
      }
    }
    if (!fine) atomicCAS(a.status, 0, kStatusTimeout);
    fence_async_smem();
    tc_fence_before();
    ok = (__syncthreads_and(fine) != 0) && ok;
    fine = true;
    // after the barrier: the head epilogue of t - 1 runs while the MMA warp
    // issues the gate of t + 1
    if (t >= 1 && warp < kResEpiWarps) {
      // head(t - 1) is the ((t - 1) / 2)-th commit to its barrier
      const uint32_t hb = (uint32_t)((t - 1) & 1);
      fine = mbar_wait(head_bar + hb, (uint32_t)((t - 1) >> 1) & 1u) && fine;
      tc_fence_after();
      // ---- head epilogue of t - 1
      const uint32_t tq = tmem + hcol0 + hb * 8u * g.Bp + (uint32_t)half * 4 * g.Bp +
                         ((uint32_t)(32 * q4) << 16);
      const uint32_t tq2 = tq + (16u << 16);
      for (int b0 = 4 * sp; b0 < g.Bp; b0 += 8) {
        uint32_t wv[4], wd[4], zv[4], zd[4];
        const uint32_t cw = (uint32_t)b0;
        tmem_ld_16x128b(tq + cw, wv[0], wv[1]);
        tmem_ld_16x128b(tq2 + cw, wv[2], wv[3]);
        tmem_ld_16x128b(tq + cw + g.Bp, wd[0], wd[1]);
        tmem_ld_16x128b(tq2 + cw + g.Bp, wd[2], wd[3]);
        tmem_ld_16x128b(tq + 2 * g.Bp + cw, zv[0], zv[1]);
        tmem_ld_16x128b(tq2 + 2 * g.Bp + cw, zv[2], zv[3]);
        tmem_ld_16x128b(tq + 3 * g.Bp + cw, zd[0], zd[1]);
        tmem_ld_16x128b(tq2 + 3 * g.Bp + cw, zd[2], zd[3]);
        tmem_wait_ld();
        float lp[4], lm[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float C = fmaf(eps2, __uint_as_float(zd[k]), __uint_as_float(wv[k])) + bo[k];
          const float D = fmaf(eps, __uint_as_float(wd[k]) + __uint_as_float(zv[k]), dbo[k]);
          lp[k] = C + D;
          lm[k] = C - D;
        }
        float mp = fmaxf(fmaxf(lp[0], lp[1]), fmaxf(lp[2], lp[3]));
        float mm = fmaxf(fmaxf(lm[0], lm[1]), fmaxf(lm[2], lm[3]));
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
          mp = fmaxf(mp, __shfl_xor_sync(0xffffffffu, mp, o));
          mm = fmaxf(mm, __shfl_xor_sync(0xffffffffu, mm, o));
        }
        float sp = 0.f, sm_ = 0.f;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          sp += __expf(lp[k] - mp);
          sm_ += __expf(lm[k] - mm);
        }
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
          sp += __shfl_xor_sync(0xffffffffu, sp, o);
          sm_ += __shfl_xor_sync(0xffffffffu, sm_, o);
        }
        const int b = b0 + bq;
        if (r4 == 0) {
          red[((half * 4 + q4) * 2 + 0) * g.Bp + b] = make_float2(mp, sp);
          red[((half * 4 + q4) * 2 + 1) * g.Bp + b] = make_float2(mm, sm_);
        }
        if (b < g.B && SOMA_CHECK((size_t)seq_offset(s, e, i, b) + t < a.n_bytes, a.status)) {
          const int y = s.bytes[seq_offset(s, e, i, b) + t] - vq - r4;  // target of t - 1
          if (y >= 0 && y < 32 && (y & 7) == 0) {
            const int k = y >> 3;
            ylog[b] = k == 0 ? lp[0] : k == 1 ? lp[1] : k == 2 ? lp[2] : lp[3];
            ylog[g.Bp + b] = k == 0 ? lm[0] : k == 1 ? lm[1] : k == 2 ? lm[2] : lm[3];
          }
        }
      }
      // the epilogue warps only: the MMA warp is issuing the gate of t
      asm volatile("bar.sync 1, %0;" ::"n"(kResEpiWarps * 32) : "memory");
      if (tid < g.B) {
        float nll[2];
        for (int sg = 0; sg < 2; ++sg) {
          float M = -INFINITY;
          for (int h = 0; h < 8; ++h) M = fmaxf(M, red[(h * 2 + sg) * g.Bp + tid].x);
          float S = 0.f;
          for (int h = 0; h < 8; ++h) {
            const float2 q = red[(h * 2 + sg) * g.Bp + tid];
            S += q.y * __expf(q.x - M);
          }
          nll[sg] = M + logf(S) - ylog[sg * g.Bp + tid];
        }
        acc[tid] += (double)nll[0];
        acc[g.Bp + tid] += (double)nll[1];
        acc[2 * g.Bp + tid] += (double)nll[0] - (double)nll[1];  // exact in fp64
      }
    }

  }
  if (!fine) atomicCAS(a.status, 0, kStatusTimeout);
  tc_fence_before();
  ok = (__syncthreads_and(fine) != 0) && ok;

  // ---- losses and coefficient of the pair (fp64 sums, sequences in order)
  if (tid == 0) {
    double sp = 0.0, sm = 0.0, sd = 0.0;
    for (int b = 0; b < g.B; ++b) {
      sp += acc[b];
      sm += acc[g.Bp + b];
      sd += acc[2 * g.Bp + b];
    }
    const double inv = 1.0 / ((double)g.B * (double)g.T);
    const double Lp = sp * inv, Lm = sm * inv, D = sd * inv;
    const double c = (eps == 0.f) ? 0.0 : D / (2.0 * (double)eps);
    const int64_t pair = blockIdx.x;
    if (a.n_sign == 2) {
      a.losses_out[pair * 2] = (float)Lp;
      a.losses_out[pair * 2 + 1] = (float)Lm;
    } else {
      a.losses_out[pair] = (float)Lp;
    }
    if (a.coef_out) a.coef_out[pair] = (float)c;
    if (a.coef_ws) a.coef_ws[pair] = (float)c;
    if (!(isfinite(Lp) && isfinite(Lm) && isfinite(c))) atomicCAS(a.status, 0, kStatusNonFinite);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, g.tmem_cols);
}

}  // namespace

bool res_supported(const Layout& lay, int B) {
  if (B < 1 || B > kResMaxBp || lay.H > 64) return false;
  const ResGeom g = make_res_geom(lay, B, 1);
  // one thread gathers each 8-column chunk of the embedding operand
  // and the gate plus two head accumulators fit the 512 TMEM columns
  return g.bytes <= kResMaxSmem && 2 * g.Bp * (g.Ek / 8) <= kResEpiWarps * 32 &&
         (g.MTg + 4) * 4 * g.Bp <= 512;
}

cudaError_t launch_forward_res(const Sweep& s, int n_sign, float* losses_out, float* coef_out,
                               float* coef_ws, int* status, cudaStream_t stream) {
  ResArgs a;
  a.sw = s;
  a.n_sign = n_sign;
  a.g = make_res_geom(s.lay, s.B, s.T);
  a.losses_out = losses_out;
  a.coef_out = coef_out;
  a.coef_ws = coef_ws;
  a.status = status;
  a.n_params = (size_t)s.n_experts * s.lay.P;
  a.n_bytes = (size_t)(s.batch_per_probe ? s.n_experts * s.n_pert : s.n_experts) * s.B_mem *
              (size_t)(s.T + 1);
  cudaError_t e = cudaFuncSetAttribute(res_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)a.g.bytes);
  if (e != cudaSuccess) return e;
  trace_begin(SOMA_TRACE_GATE, stream);
  res_kernel<<<s.n_experts * s.n_pert, kResThreads, a.g.bytes, stream>>>(a);
  trace_end(SOMA_TRACE_GATE, stream);
  return cudaGetLastError();
}

}  // namespace soma
