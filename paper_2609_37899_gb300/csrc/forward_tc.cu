// forward_tc.cu -- tensor-core (tcgen05 / TMEM) forward sweep of the
// perturbed LSTM experts in the mean/difference form.
//
// For one expert e and probe i, the two antithetic copies of the LSTM take
// inputs v+- = [x+-; h+-_{t-1}].  Write vbar = (v+ + v-)/2 and dv = (v+ - v-)/2.
// With the perturbed weights W +- eps Z (Z = z_{e,i} reshaped, entries +-1),
//   (W +- eps Z)(vbar +- dv) = [W vbar + eps Z dv] +- [W dv + eps Z vbar]
// exactly, so the gate pre-activations are a+- = C +- D with
//   C = W vbar + eps (Z dv) + b,       D = W dv + eps (Z vbar) + eps z_b.
// The four products W vbar, W dv, Z vbar, Z dv are fp16 x fp16 -> fp32
// tensor-core GEMMs; eps multiplies only in fp32 (epilogue), so no operand
// ever holds a rounded w +- eps z.  dv is an explicit operand, so the
// rounding of the operands perturbs the difference of the two copies only
// relatively (fp16: 2^-11), never by cancellation.  The cell state c+- and
// the activations are fp32 per sign.  The output head uses the same split:
// logits+- = [W_out hbar + eps Z_out dh + b_out] +- [W_out dh + eps Z_out hbar
// + eps z_bo].
//
// Per timestep t:
//   gate_tc_kernel  one CTA per (expert, 32-unit row tile, group of P probes):
//                   D_W[128 x 2BpP] = W_tile x [vbar|dv]^T (one MMA chain,
//                   shared by the P probes) and D_Z,p[128 x 2Bp] = Z_p x
//                   [vbar_p|dv_p]^T, Z_p generated from Philox into shared
//                   memory stage by stage; epilogue: gates, cell update,
//                   next timestep's operand [hbar|dh] (fp16).
//   head_tc_kernel  one CTA per (expert, 128-row vocabulary half, probe
//                   group): the same MMAs over the h part of the operand,
//                   then per (sequence, sign) max and sum-exp partials of
//                   the half and the target logit.
//   xpart_kernel    the embedding part of the next operand.
// A final reduction merges the two halves into per-target NLL and the
// per-(expert, probe) losses and coefficients.
#include <cuda_fp16.h>

#include "soma_api.h"
#include "soma_device.cuh"
#include "soma_launch.h"
#include "tc_primitives.cuh"

namespace soma {

using namespace tc;

namespace {

constexpr int kThreads = 256;
constexpr int kStages = 3;
constexpr int kKt = 32;                 // K per stage (fp16 elements)
constexpr uint32_t kTileA = 128 * kKt * 2;  // one 128-row A tile per stage
constexpr uint32_t kSbo = kKt * 16;     // bytes between 8-row groups
constexpr uint32_t kLbo = 128;          // bytes between core matrices along K
constexpr uint32_t kZCols = 256;        // TMEM column where the Z products start
constexpr uint32_t kTmemCols = 512;

__device__ __forceinline__ uint32_t compact16(uint32_t x) {
  x &= 0x55555555u;
  x = (x | (x >> 1)) & 0x33333333u;
  x = (x | (x >> 2)) & 0x0F0F0F0Fu;
  x = (x | (x >> 4)) & 0x00FF00FFu;
  x = (x | (x >> 8)) & 0x0000FFFFu;
  return x;
}

// natural-order bits (bit o <=> offset o) -> the raw run order (even offsets
// in the low half, odd offsets in the high half)
__device__ __forceinline__ uint32_t natural_to_raw(uint32_t n) {
  return compact16(n) | (compact16(n >> 1) << 16);
}

__device__ __forceinline__ float sigm(float x) { return __fdividef(1.0f, 1.0f + __expf(-x)); }

// Shared-memory carve-up of one stage.
struct StageLayout {
  uint32_t a_off, b_off, z_off, bytes;
};

__host__ __device__ inline StageLayout stage_layout(const TcGeom& g) {
  StageLayout L;
  L.a_off = 0;
  L.b_off = kTileA;
  L.z_off = L.b_off + g.tileB;
  L.bytes = L.z_off + (uint32_t)g.P * kTileA;
  return L;
}

// Cached Philox block of one (probe, row) slot of the Z generator.
struct ZSlot {
  uint32_t blk;
  uint4 w;
};

// Raw run word for the 32 parameters p0 .. p0+31 of probe key pk.
__device__ __forceinline__ uint32_t z_run_raw(const ProbeKey& pk, int64_t p0, ZSlot& c) {
  if ((p0 & 31) == 0) {
    const uint32_t w = (uint32_t)(p0 >> 5);
    const uint32_t blk = w >> 2;
    if (blk != c.blk) {
      c.w = probe_block(pk, blk);
      c.blk = blk;
    }
    return word_of(c.w, (int)(w & 3));
  }
  return natural_to_raw(probe_bits32(pk, p0));
}

// Writes the 128 x 32 Z tile row r (one 32-parameter run) in the canonical
// K-major layout.
__device__ __forceinline__ void store_z_row(uint8_t* ztile, int r, uint32_t raw) {
  uint4 c0, c1, c2, c3;
  c0.x = pm1_pair<0>(raw);  c0.y = pm1_pair<1>(raw);  c0.z = pm1_pair<2>(raw);  c0.w = pm1_pair<3>(raw);
  c1.x = pm1_pair<4>(raw);  c1.y = pm1_pair<5>(raw);  c1.z = pm1_pair<6>(raw);  c1.w = pm1_pair<7>(raw);
  c2.x = pm1_pair<8>(raw);  c2.y = pm1_pair<9>(raw);  c2.z = pm1_pair<10>(raw); c2.w = pm1_pair<11>(raw);
  c3.x = pm1_pair<12>(raw); c3.y = pm1_pair<13>(raw); c3.z = pm1_pair<14>(raw); c3.w = pm1_pair<15>(raw);
  *reinterpret_cast<uint4*>(ztile + kmajor_offset(r, 0, kKt)) = c0;
  *reinterpret_cast<uint4*>(ztile + kmajor_offset(r, 8, kKt)) = c1;
  *reinterpret_cast<uint4*>(ztile + kmajor_offset(r, 16, kKt)) = c2;
  *reinterpret_cast<uint4*>(ztile + kmajor_offset(r, 24, kKt)) = c3;
}

// Everything the main loop needs for one task.
struct TaskIO {
  const uint8_t* a;      // A1 tile of stage 0
  size_t a_stride;       // bytes between the A1 tiles of consecutive stages
  const uint8_t* b;      // operand group tile of stage 0
  size_t b_stride;
  int nst;               // stages
  int p_valid;           // probes of this group that exist
  bool do_z;             // eps != 0: the Z products are needed
};

// Main loop shared by the gate and head kernels.  zparam(r, s) is the flat
// parameter index of element (row r, k = 0) of the stage-s Z run.
// A wait that times out records SOMA_ERR_TIMEOUT in the status word and sets
// the CTA's abort flag; every later wait and MMA of the task is skipped.
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort,
                                              int* status) {
  if (*abort) return false;
  if (mbar_wait(bar, parity)) return true;
  *abort = 1;
  atomicCAS(status, 0, kStatusTimeout);
  return false;
}

template <class ZParam>
__device__ bool tc_mainloop(const TcGeom& g, const TaskIO& io, uint8_t* smem, uint64_t* load_full,
                            uint64_t* mma_done, uint32_t tmem, const ProbeKey* pks,
                            ZParam zparam, volatile int* abort, int* status) {
  const int tid = threadIdx.x;
  const StageLayout SL = stage_layout(g);
  const uint32_t idesc_w = idesc_f16_f32(128, g.rowsB);
  const uint32_t idesc_z = idesc_f16_f32(128, 2 * g.Bp);
  const uint32_t b_bytes = g.tileB;
  const int nz = io.do_z ? io.p_valid * 128 : 0;  // (probe, row) pairs to generate
  ZSlot cache[2];
  cache[0].blk = 0xFFFFFFFFu;
  cache[1].blk = 0xFFFFFFFFu;

  for (int s = 0; s < io.nst; ++s) {
    const int q = s % kStages;
    const uint32_t use = (uint32_t)(s / kStages);
    uint8_t* st = smem + q * SL.bytes;
    if (s >= kStages) wait_or_abort(&mma_done[q], (use - 1) & 1u, abort, status);
    if (tid == 0 && !*abort) {
      mbar_arrive_expect_tx(&load_full[q], kTileA + b_bytes);
      bulk_g2s(st + SL.a_off, io.a + (size_t)s * io.a_stride, kTileA, &load_full[q]);
      bulk_g2s(st + SL.b_off, io.b + (size_t)s * io.b_stride, b_bytes, &load_full[q]);
    }
    // Z tiles of this stage: thread handles pairs tid and tid + 256
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int pr = tid + j * kThreads;
      if (pr < nz) {
        const int p = pr >> 7, r = pr & 127;
        const uint32_t raw = z_run_raw(pks[p], zparam(r, s), cache[j]);
        store_z_row(st + SL.z_off + p * kTileA, r, raw);
      }
    }
    fence_async_smem();
    __syncthreads();
    if (tid == 0 && !*abort) {
      const bool ok = wait_or_abort(&load_full[q], use & 1u, abort, status);
      tc_fence_after();
      if (ok) {
        const uint32_t a_addr = smem_u32(st + SL.a_off);
        const uint32_t b_addr = smem_u32(st + SL.b_off);
        const uint32_t z_addr = smem_u32(st + SL.z_off);
#pragma unroll
        for (int k16 = 0; k16 < kKt / 16; ++k16) {
          const uint32_t acc = (s > 0 || k16 > 0) ? 1u : 0u;
          mma_f16_ss(tmem, smem_desc(a_addr + k16 * 32 * 8, kLbo, kSbo),
                     smem_desc(b_addr + k16 * 32 * 8, kLbo, kSbo), idesc_w, acc);
          if (io.do_z) {
            for (int p = 0; p < io.p_valid; ++p) {
              const uint32_t brow = (uint32_t)(2 * g.Bp * p);
              mma_f16_ss(tmem + kZCols + brow,
                         smem_desc(z_addr + p * kTileA + k16 * 32 * 8, kLbo, kSbo),
                         smem_desc(b_addr + (brow / 8) * kSbo + k16 * 32 * 8, kLbo, kSbo),
                         idesc_z, acc);
            }
          }
        }
      }
      mma_commit(&mma_done[q]);
    }
  }
  // all MMAs issued by this CTA are complete once the last commit lands
  const int last = io.nst - 1;
  wait_or_abort(&mma_done[last % kStages], (uint32_t)(last / kStages) & 1u, abort, status);
  tc_fence_after();
  __syncthreads();
  return !*abort;
}

struct TcArgs {
  Sweep sw;
  TcGeom g;
  int t;
  const uint8_t* w16;    // [N][MT][S] A tiles
  const uint8_t* wo16;   // [N][2][Sh] A tiles
  const uint8_t* op_in;  // [N][S][G] operand group tiles of this timestep
  uint8_t* op_out;       // next timestep's operand
  float* cst;            // [N*n*2][B][Hp] cell state
  float* pm;             // [N*n*2][B][T][2] head max partials
  float* ps;             // sum-exp partials
  float* ply;            // [N*n*2][B][T] target logits
  int* status;
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

struct KernelShared {
  uint64_t load_full[kStages];
  uint64_t mma_done[kStages];
  uint32_t tmem_slot;
  volatile int abort;
};

__device__ __forceinline__ void kernel_setup(KernelShared* ks, uint32_t& tmem) {
  if (threadIdx.x == 0) {
    ks->abort = 0;
    for (int q = 0; q < kStages; ++q) {
      mbar_init(&ks->load_full[q], 1);
      mbar_init(&ks->mma_done[q], 1);
    }
    mbar_fence_init();
  }
  if (threadIdx.x < 32) tmem_alloc(&ks->tmem_slot, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  tmem = ks->tmem_slot;
}

__device__ __forceinline__ void kernel_teardown(uint32_t tmem) {
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x < 32) tmem_dealloc(tmem, kTmemCols);
}

// grid: N * MT * G blocks, 256 threads.
__global__ void __launch_bounds__(kThreads, 1) gate_tc_kernel(const TcArgs a) {
  extern __shared__ uint8_t dyn_smem[];
  uint8_t* smem = align1024(dyn_smem);
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  KernelShared* ks = reinterpret_cast<KernelShared*>(smem + kStages * stage_layout(g).bytes);
  const int task = blockIdx.x;
  const int grp = task % g.G;
  const int m = (task / g.G) % g.MT;
  const int e = task / (g.G * g.MT);
  const int H = g.H, E = g.E;
  const Layout& L = s.lay;
  const float* th = s.params + (int64_t)e * L.P;

  __shared__ ProbeKey pks[16];
  if (threadIdx.x < g.P)
    pks[threadIdx.x] = make_probe_key(s.seed, s.step, (uint32_t)e, (uint32_t)(grp * g.P + threadIdx.x));
  uint32_t tmem;
  kernel_setup(ks, tmem);

  TaskIO io;
  io.a = a.w16 + (((size_t)e * g.MT + m) * g.S) * kTileA;
  io.a_stride = kTileA;
  io.b = a.op_in + (((size_t)e * g.S) * g.G + grp) * g.tileB;
  io.b_stride = (size_t)g.G * g.tileB;
  io.nst = g.S;
  io.p_valid = min(g.P, s.n_pert - grp * g.P);
  io.do_z = s.eps != 0.f;
  const int Sx = g.Sx;
  auto zparam = [&](int r, int st) -> int64_t {
    const int64_t R = (int64_t)(r & 3) * H + 32 * m + (r >> 2);  // W row of tile row r
    return st < Sx ? L.w_ih + R * E + (int64_t)kKt * st
                   : L.w_hh + R * H + (int64_t)kKt * (st - Sx);
  };
  if (!tc_mainloop(g, io, smem, ks->load_full, ks->mma_done, tmem, pks, zparam, &ks->abort,
                   a.status)) {
    kernel_teardown(tmem);
    return;
  }

  // ---- epilogue: gates, cell update, next operand --------------------------
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int q4 = warp & 3, half = warp >> 2;
  const int r = 32 * q4 + lane;
  const int u_loc = r >> 2, gate = r & 3;
  const int U = 32 * m + u_loc;
  const bool unit_ok = U < H;
  const uint32_t tl = tmem + ((uint32_t)(32 * q4) << 16);
  const float sc = (gate == 2) ? 2.f : 1.f;   // tanh(x) = 2 sigmoid(2x) - 1
  const float add = (gate == 2) ? -1.f : 0.f;
  const int base = lane & ~3;
  const bool sign_lane = gate < 2;             // gate 0 lane: sign +, gate 1 lane: sign -
  const float eps = s.eps;
  uint8_t* out_tile = a.op_out + (((size_t)e * g.S + Sx + m) * g.G + grp) * g.tileB;

  for (int p = half; p < io.p_valid; p += 2) {
    const int i = grp * g.P + p;
    float bias = 0.f, dbias = 0.f;
    if (unit_ok) {
      const int64_t pb = L.b + (int64_t)gate * H + U;
      bias = th[pb];
      if (io.do_z) dbias = (probe_bits32(pks[p], pb) & 1u) ? -eps : eps;
    }
    const int64_t lane_plus = ((int64_t)e * s.n_pert + i) * 2;
    for (int b0 = 0; b0 < g.Bp; b0 += 8) {
      float wv[8], wd[8], zv[8], zd[8];
      const uint32_t cw = (uint32_t)(2 * g.Bp * p + b0);
      tmem_ld8(tl + cw, wv);
      tmem_ld8(tl + cw + g.Bp, wd);
      if (io.do_z) {
        tmem_ld8(tl + kZCols + cw, zv);
        tmem_ld8(tl + kZCols + cw + g.Bp, zd);
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) zv[j] = zd[j] = 0.f;
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int b = b0 + j;
        const float C = fmaf(eps, zd[j], wv[j]) + bias;
        const float D = fmaf(eps, zv[j], wd[j]) + dbias;
        const float actp = fmaf(sigm(sc * (C + D)), sc, add);
        const float actm = fmaf(sigm(sc * (C - D)), sc, add);
        const float ip = __shfl_sync(0xffffffffu, actp, base);
        const float fp = __shfl_sync(0xffffffffu, actp, base + 1);
        const float gp = __shfl_sync(0xffffffffu, actp, base + 2);
        const float op = __shfl_sync(0xffffffffu, actp, base + 3);
        const float im = __shfl_sync(0xffffffffu, actm, base);
        const float fm = __shfl_sync(0xffffffffu, actm, base + 1);
        const float gm = __shfl_sync(0xffffffffu, actm, base + 2);
        const float om = __shfl_sync(0xffffffffu, actm, base + 3);
        const bool active = sign_lane && unit_ok && b < s.B;
        float h = 0.f;
        if (active) {
          const bool plus = gate == 0;
          float* cp = a.cst + ((lane_plus + gate) * s.B + b) * (int64_t)g.Hp + U;
          const float cprev = (a.t == 0) ? 0.f : *cp;
          const float c = plus ? fmaf(fp, cprev, ip * gp) : fmaf(fm, cprev, im * gm);
          *cp = c;
          h = (plus ? op : om) * fmaf(sigm(2.f * c), 2.f, -1.f);
        }
        const float hp = __shfl_sync(0xffffffffu, h, base);
        const float hm = __shfl_sync(0xffffffffu, h, base + 1);
        if (active) {
          const bool plus = gate == 0;
          const float val = plus ? 0.5f * (hp + hm) : 0.5f * (hp - hm);
          const int row = 2 * g.Bp * p + (plus ? b : g.Bp + b);
          *reinterpret_cast<__half*>(out_tile + kmajor_offset(row, u_loc, kKt)) =
              __float2half_rn(val);
        }
      }
    }
  }
  kernel_teardown(tmem);
}

// grid: N * 2 * G blocks, 256 threads.  Head of timestep t: reads the h
// part of the operand of timestep t + 1 (which holds hbar_t and dh_t).
__global__ void __launch_bounds__(kThreads, 1) head_tc_kernel(const TcArgs a) {
  extern __shared__ uint8_t dyn_smem[];
  uint8_t* smem = align1024(dyn_smem);
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  KernelShared* ks = reinterpret_cast<KernelShared*>(smem + kStages * stage_layout(g).bytes);
  const int task = blockIdx.x;
  const int grp = task % g.G;
  const int vh = (task / g.G) % 2;
  const int e = task / (g.G * 2);
  const int H = g.H;
  const Layout& L = s.lay;
  const float* th = s.params + (int64_t)e * L.P;

  __shared__ ProbeKey pks[16];
  if (threadIdx.x < g.P)
    pks[threadIdx.x] = make_probe_key(s.seed, s.step, (uint32_t)e, (uint32_t)(grp * g.P + threadIdx.x));
  uint32_t tmem;
  kernel_setup(ks, tmem);

  TaskIO io;
  io.a = a.wo16 + (((size_t)e * 2 + vh) * g.Sh) * kTileA;
  io.a_stride = kTileA;
  io.b = a.op_in + (((size_t)e * g.S + g.Sx) * g.G + grp) * g.tileB;
  io.b_stride = (size_t)g.G * g.tileB;
  io.nst = g.Sh;
  io.p_valid = min(g.P, s.n_pert - grp * g.P);
  io.do_z = s.eps != 0.f;
  auto zparam = [&](int r, int st) -> int64_t {
    return L.w_out + (int64_t)(128 * vh + r) * H + (int64_t)kKt * st;
  };
  if (!tc_mainloop(g, io, smem, ks->load_full, ks->mma_done, tmem, pks, zparam, &ks->abort,
                   a.status)) {
    kernel_teardown(tmem);
    return;
  }

  // ---- epilogue: logits +-, per-half max / sum-exp, target logit ----------
  // the stage buffers are free now: reuse them for the cross-warp reduction
  float2* red = reinterpret_cast<float2*>(smem);  // [P][Bp][2][4]
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int q4 = warp & 3, half = warp >> 2;
  const int v = 128 * vh + 32 * q4 + lane;
  const uint32_t tl = tmem + ((uint32_t)(32 * q4) << 16);
  const float eps = s.eps;
  const float bo = th[L.b_out + v];
  const int t = a.t;
  for (int p = half; p < io.p_valid; p += 2) {
    const int i = grp * g.P + p;
    const float dbo = io.do_z ? ((probe_bits32(pks[p], L.b_out + v) & 1u) ? -eps : eps) : 0.f;
    const int64_t lane_plus = ((int64_t)e * s.n_pert + i) * 2;
    for (int b0 = 0; b0 < g.Bp; b0 += 8) {
      float wv[8], wd[8], zv[8], zd[8];
      const uint32_t cw = (uint32_t)(2 * g.Bp * p + b0);
      tmem_ld8(tl + cw, wv);
      tmem_ld8(tl + cw + g.Bp, wd);
      if (io.do_z) {
        tmem_ld8(tl + kZCols + cw, zv);
        tmem_ld8(tl + kZCols + cw + g.Bp, zd);
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) zv[j] = zd[j] = 0.f;
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int b = b0 + j;
        const float C = fmaf(eps, zd[j], wv[j]) + bo;
        const float D = fmaf(eps, zv[j], wd[j]) + dbo;
        const float lp = C + D, lm = C - D;
        float mp = lp, mm = lm;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          mp = fmaxf(mp, __shfl_xor_sync(0xffffffffu, mp, o));
          mm = fmaxf(mm, __shfl_xor_sync(0xffffffffu, mm, o));
        }
        float sp = __expf(lp - mp), sm_ = __expf(lm - mm);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          sp += __shfl_xor_sync(0xffffffffu, sp, o);
          sm_ += __shfl_xor_sync(0xffffffffu, sm_, o);
        }
        if (lane == 0) {
          red[((p * g.Bp + b) * 2 + 0) * 4 + q4] = make_float2(mp, sp);
          red[((p * g.Bp + b) * 2 + 1) * 4 + q4] = make_float2(mm, sm_);
        }
        if (b < s.B) {
          const int y = s.bytes[((int64_t)e * s.B + b) * (s.T + 1) + t + 1];
          if (y == v) {
            a.ply[((lane_plus + 0) * s.B + b) * (int64_t)s.T + t] = lp;
            a.ply[((lane_plus + 1) * s.B + b) * (int64_t)s.T + t] = lm;
          }
        }
      }
    }
  }
  __syncthreads();
  // merge the four 32-row quarters of this half
  const int n_red = io.p_valid * g.Bp * 2;
  for (int idx = tid; idx < n_red; idx += kThreads) {
    const int sgn = idx & 1;
    const int pb = idx >> 1;
    const int p = pb / g.Bp, b = pb % g.Bp;
    if (b >= s.B) continue;
    const float2* q = red + (size_t)idx * 4;
    float M = fmaxf(fmaxf(q[0].x, q[1].x), fmaxf(q[2].x, q[3].x));
    float S = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) S += q[k].y * __expf(q[k].x - M);
    const int i = grp * g.P + p;
    const int64_t ln = ((int64_t)e * s.n_pert + i) * 2 + sgn;
    const int64_t o = ((ln * s.B + b) * (int64_t)s.T + t) * 2 + vh;
    a.pm[o] = M;
    a.ps[o] = S;
  }
  kernel_teardown(tmem);
}

// Embedding part of the operand of timestep t: x = Emb[byte_t], dx = eps z_emb.
// grid (Sx * G, N), 128 threads.
__global__ void xpart_kernel(const TcArgs a, uint8_t* op) {
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  const int st = blockIdx.x / g.G, grp = blockIdx.x % g.G;
  const int e = blockIdx.y;
  const Layout& L = s.lay;
  const float* th = s.params + (int64_t)e * L.P;
  uint8_t* tile = op + (((size_t)e * g.S + st) * g.G + grp) * g.tileB;
  const int chunks = g.rowsB * (kKt / 8);
  for (int c = threadIdx.x; c < chunks; c += blockDim.x) {
    const int row = c / (kKt / 8), kc = c % (kKt / 8);
    const int p = row / (2 * g.Bp), rr = row % (2 * g.Bp);
    const int i = grp * g.P + p;
    const bool delta = rr >= g.Bp;
    const int b = delta ? rr - g.Bp : rr;
    __align__(16) __half v[8];
    const int k0 = kKt * st + 8 * kc;
    if (i < s.n_pert && b < s.B) {
      const int y = s.bytes[((int64_t)e * s.B + b) * (s.T + 1) + a.t];
      const int64_t p0 = L.emb + (int64_t)y * g.E + k0;
      uint32_t bits = 0;
      if (delta && s.eps != 0.f)
        bits = probe_bits32(make_probe_key(s.seed, s.step, (uint32_t)e, (uint32_t)i), p0);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        float x = 0.f;
        if (k0 + j < g.E) x = delta ? (((bits >> j) & 1u) ? -s.eps : s.eps) : th[p0 + j];
        v[j] = __float2half_rn(x);
      }
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) v[j] = __float2half_rn(0.f);
    }
    *reinterpret_cast<uint4*>(tile + kmajor_offset(row, 8 * kc, kKt)) =
        *reinterpret_cast<const uint4*>(v);
  }
}

// fp16 A tiles of the gate weights ([x part | h part], rows unit-major:
// tile row r = 4 * unit + gate) and of the head weights.
// grid (MT * S + 2 * Sh, N), 128 threads: thread r writes row r of a tile.
__global__ void prep_tiles_kernel(const TcArgs a) {
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  const Layout& L = s.lay;
  const int e = blockIdx.y;
  const float* th = s.params + (int64_t)e * L.P;
  const int r = threadIdx.x;
  const int tix = blockIdx.x;
  __align__(16) __half v[kKt];
  uint8_t* tile;
  if (tix < g.MT * g.S) {
    const int m = tix / g.S, st = tix % g.S;
    const int U = 32 * m + (r >> 2), gate = r & 3;
    const int64_t R = (int64_t)gate * g.H + U;
    for (int kk = 0; kk < kKt; ++kk) {
      float w = 0.f;
      if (U < g.H) {
        if (st < g.Sx) {
          const int k = kKt * st + kk;
          if (k < g.E) w = th[L.w_ih + R * g.E + k];
        } else {
          const int k = kKt * (st - g.Sx) + kk;
          if (k < g.H) w = th[L.w_hh + R * g.H + k];
        }
      }
      v[kk] = __float2half_rn(w);
    }
    tile = const_cast<uint8_t*>(a.w16) + (((size_t)e * g.MT + m) * g.S + st) * kTileA;
  } else {
    const int t2 = tix - g.MT * g.S;
    const int vh = t2 / g.Sh, st = t2 % g.Sh;
    const int vrow = 128 * vh + r;
    for (int kk = 0; kk < kKt; ++kk) {
      const int k = kKt * st + kk;
      v[kk] = __float2half_rn(k < g.H ? th[L.w_out + (int64_t)vrow * g.H + k] : 0.f);
    }
    tile = const_cast<uint8_t*>(a.wo16) + (((size_t)e * 2 + vh) * g.Sh + st) * kTileA;
  }
#pragma unroll
  for (int kc = 0; kc < kKt / 8; ++kc)
    *reinterpret_cast<uint4*>(tile + kmajor_offset(r, 8 * kc, kKt)) =
        *reinterpret_cast<const uint4*>(v + 8 * kc);
}

// Per (expert, probe) pair: merge the two vocabulary halves into the NLL of
// every target, then L+, L- (fp64 sums), D = mean(nll+ - nll-) and D / (2 eps).
__global__ void __launch_bounds__(256)
reduce_tc_kernel(const float* __restrict__ pm, const float* __restrict__ ps,
                 const float* __restrict__ ply, int n_sign, int BT, float eps, float* losses_out,
                 float* coef_out, float* coef_ws, int* status) {
  __shared__ double red[3][256];
  const int pair = blockIdx.x;
  const int64_t lp = (int64_t)pair * 2, lm = lp + 1;
  double sp = 0.0, sm = 0.0, sd = 0.0;
  for (int j = threadIdx.x; j < BT; j += 256) {
    float nll[2];
    for (int sg = 0; sg < 2; ++sg) {
      const int64_t ln = sg ? lm : lp;
      const float m0 = pm[(ln * BT + j) * 2], m1 = pm[(ln * BT + j) * 2 + 1];
      const float s0 = ps[(ln * BT + j) * 2], s1 = ps[(ln * BT + j) * 2 + 1];
      const float M = fmaxf(m0, m1);
      nll[sg] = M + logf(s0 * expf(m0 - M) + s1 * expf(m1 - M)) - ply[ln * BT + j];
    }
    sp += (double)nll[0];
    sm += (double)nll[1];
    sd += (double)(nll[0] - nll[1]);
  }
  red[0][threadIdx.x] = sp;
  red[1][threadIdx.x] = sm;
  red[2][threadIdx.x] = sd;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
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

// Debug GEMM: D[128][N] = A[128][K] * B[N][K]^T through the same descriptors,
// instruction descriptor and TMEM read-back as the forward kernels.  A and B
// are fp16 row-major in global memory; 128 threads stage them into the
// canonical layout (K <= 256, N <= 256, both multiples of 16).
__global__ void __launch_bounds__(128, 1)
debug_tc_gemm_kernel(const __half* A, const __half* B, float* D, int N, int K, int* status) {
  extern __shared__ uint8_t dyn_smem[];
  uint8_t* smem = align1024(dyn_smem);
  uint8_t* sa = smem;
  uint8_t* sb = smem + 128 * K * 2;
  __shared__ uint64_t bar;
  __shared__ uint32_t slot;
  const int tid = threadIdx.x;
  if (tid == 0) {
    mbar_init(&bar, 1);
    mbar_fence_init();
  }
  if (tid < 32) tmem_alloc(&slot, 256);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = slot;
  for (int c = tid; c < 128 * (K / 8); c += 128) {
    const int r = c / (K / 8), kc = c % (K / 8);
    *reinterpret_cast<uint4*>(sa + kmajor_offset(r, 8 * kc, K)) =
        *reinterpret_cast<const uint4*>(A + (size_t)r * K + 8 * kc);
  }
  for (int c = tid; c < N * (K / 8); c += 128) {
    const int r = c / (K / 8), kc = c % (K / 8);
    *reinterpret_cast<uint4*>(sb + kmajor_offset(r, 8 * kc, K)) =
        *reinterpret_cast<const uint4*>(B + (size_t)r * K + 8 * kc);
  }
  fence_async_smem();
  __syncthreads();
  if (tid == 0) {
    tc_fence_after();
    const uint32_t idesc = idesc_f16_f32(128, N);
    for (int k16 = 0; k16 < K / 16; ++k16)
      mma_f16_ss(tmem, smem_desc(smem_u32(sa) + k16 * 256, 128, K * 16),
                 smem_desc(smem_u32(sb) + k16 * 256, 128, K * 16), idesc, k16 > 0 ? 1u : 0u);
    mma_commit(&bar);
  }
  if (!mbar_wait(&bar, 0) && tid == 0) atomicCAS(status, 0, kStatusTimeout);
  tc_fence_after();
  const int warp = tid >> 5, lane = tid & 31;
  for (int c0 = 0; c0 < N; c0 += 8) {
    float v[8];
    tmem_ld8(tmem + ((uint32_t)(32 * warp) << 16) + c0, v);
    for (int j = 0; j < 8; ++j) D[(size_t)(32 * warp + lane) * N + c0 + j] = v[j];
  }
  tc_fence_before();
  __syncthreads();
  if (tid < 32) tmem_dealloc(tmem, 256);
}

size_t kernel_smem_bytes(const TcGeom& g) {
  // stages + barriers + 1 KB alignment slack; at least 120 KB so that one
  // CTA owns an SM (and all 512 TMEM columns)
  size_t b = (size_t)kStages * stage_layout(g).bytes + sizeof(KernelShared) + 1024 + 256;
  return b < 120 * 1024 ? 120 * 1024 : b;
}

}  // namespace

TcGeom make_tc_geom(const Layout& lay, int n_experts, int n_pert, int B, int T) {
  TcGeom g;
  g.E = lay.E;
  g.H = lay.H;
  g.Ep = (lay.E + kKt - 1) / kKt * kKt;
  g.Hp = (lay.H + kKt - 1) / kKt * kKt;
  g.Sx = g.Ep / kKt;
  g.Sh = g.Hp / kKt;
  g.S = g.Sx + g.Sh;
  g.MT = g.Hp / 32;
  g.Bp = (B + 7) / 8 * 8;
  int P = 128 / g.Bp;
  if (P > 4) P = 4;
  if (P > n_pert) P = n_pert;
  if (P < 1) P = 1;
  g.P = P;
  g.G = (n_pert + P - 1) / P;
  g.rowsB = 2 * g.Bp * P;
  g.tileB = (uint32_t)g.rowsB * kKt * 2;
  g.n_experts = n_experts;
  g.n_pert = n_pert;
  g.B = B;
  g.T = T;
  return g;
}

bool tc_supported(int B) { return B >= 1 && B <= 128; }

TcSizes tc_sizes(const TcGeom& g) {
  TcSizes z;
  const size_t N = (size_t)g.n_experts, n = (size_t)g.n_pert;
  z.w16 = N * g.MT * g.S * kTileA;
  z.wo16 = N * 2 * g.Sh * kTileA;
  z.op = N * g.S * g.G * g.tileB;
  z.cst = N * n * 2 * g.B * (size_t)g.Hp * sizeof(float);
  z.pm = N * n * 2 * g.B * (size_t)g.T * 2 * sizeof(float);
  z.ply = N * n * 2 * g.B * (size_t)g.T * sizeof(float);
  return z;
}

cudaError_t launch_forward_tc(const Sweep& s, const TcGeom& g, const TcBuffers& tb, int* status,
                              cudaStream_t stream) {
  const size_t smem = kernel_smem_bytes(g);
  cudaError_t e = cudaFuncSetAttribute(gate_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(head_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const TcSizes z = tc_sizes(g);
  TcArgs a;
  a.sw = s;
  a.g = g;
  a.t = 0;
  a.w16 = tb.w16;
  a.wo16 = tb.wo16;
  a.cst = tb.cst;
  a.pm = tb.pm;
  a.ps = tb.ps;
  a.ply = tb.ply;
  a.status = status;

  trace_begin(SOMA_TRACE_PREP, stream);
  prep_tiles_kernel<<<dim3(g.MT * g.S + 2 * g.Sh, g.n_experts), 128, 0, stream>>>(a);
  cudaMemsetAsync(tb.op[0], 0, z.op, stream);
  cudaMemsetAsync(tb.op[1], 0, z.op, stream);
  a.t = 0;
  xpart_kernel<<<dim3(g.Sx * g.G, g.n_experts), 128, 0, stream>>>(a, tb.op[0]);
  trace_end(SOMA_TRACE_PREP, stream);

  const int gate_blocks = g.n_experts * g.MT * g.G;
  const int head_blocks = g.n_experts * 2 * g.G;
  for (int t = 0; t < s.T; ++t) {
    a.t = t;
    a.op_in = tb.op[t & 1];
    a.op_out = tb.op[(t + 1) & 1];
    trace_begin(SOMA_TRACE_GATE, stream);
    gate_tc_kernel<<<gate_blocks, kThreads, smem, stream>>>(a);
    trace_end(SOMA_TRACE_GATE, stream);
    a.op_in = tb.op[(t + 1) & 1];
    trace_begin(SOMA_TRACE_HEAD, stream);
    head_tc_kernel<<<head_blocks, kThreads, smem, stream>>>(a);
    trace_end(SOMA_TRACE_HEAD, stream);
    if (t + 1 < s.T) {
      a.t = t + 1;
      trace_begin(SOMA_TRACE_PREP, stream);
      xpart_kernel<<<dim3(g.Sx * g.G, g.n_experts), 128, 0, stream>>>(a, tb.op[(t + 1) & 1]);
      trace_end(SOMA_TRACE_PREP, stream);
    }
  }
  return cudaGetLastError();
}

cudaError_t launch_reduce_tc(const TcBuffers& tb, int pairs, int n_sign, int B, int T, float eps,
                             float* losses_out, float* coef_out, float* coef_ws, int* status,
                             cudaStream_t stream) {
  trace_begin(SOMA_TRACE_REDUCE, stream);
  reduce_tc_kernel<<<pairs, 256, 0, stream>>>(tb.pm, tb.ps, tb.ply, n_sign, B * T, eps,
                                               losses_out, coef_out, coef_ws, status);
  trace_end(SOMA_TRACE_REDUCE, stream);
  return cudaGetLastError();
}

cudaError_t launch_debug_tc_gemm(const void* A, const void* B, float* D, int N, int K, int* status,
                                 cudaStream_t stream) {
  const size_t smem = (size_t)(128 + N) * K * 2 + 1024;
  cudaError_t e = cudaFuncSetAttribute(debug_tc_gemm_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  debug_tc_gemm_kernel<<<1, 128, smem, stream>>>(static_cast<const __half*>(A),
                                                 static_cast<const __half*>(B), D, N, K, status);
  return cudaGetLastError();
}

}  // namespace soma
