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
// Per timestep t, two launches of one persistent kernel:
//   gate tasks  (expert, 32-unit row tile, group of P probes):
//               D_W[128 x 2BpP] = W_tile x [vbar|dv]^T (shared by the P
//               probes) and D_Z,p[128 x 2Bp] = Z_p x [vbar_p|dv_p]^T, Z_p
//               generated from Philox into shared memory stage by stage;
//               epilogue: gates, cell update, next timestep's operand
//               [hbar|dh] (fp16).
//   head tasks  (expert, 128-row vocabulary half, probe group): the same
//               MMAs over the h part of the operand, then per (sequence,
//               sign) max and sum-exp partials of the half and the target
//               logit; extra blocks of the same launch write the embedding
//               part of the next operand.
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

constexpr int kZWarps = 8;
constexpr int kStages = 3;
constexpr int kLoaders = kStages;  // one issuing thread per ring slot (the copies of
                                   // one thread complete one after another)
constexpr int kEpiWarps = 8;
constexpr int kEpiProbeStep = kEpiWarps / 4;  // warp ew runs probes ew / 4, + kEpiProbeStep, ...
static_assert(kZWarps * 32 == 256, "one Z generator thread per (probe, row): 2 x 128");
static_assert(kEpiWarps == 4 || kEpiWarps == 8, "epilogue warps: 4 lane quarters x 1 or 2 probes");
constexpr int kThreads = (kLoaders + 1 + kZWarps + kEpiWarps) * 32;  // loaders, MMA, Z, epilogue
constexpr int kKt = 64;                 // K per stage (fp16 elements)
constexpr uint32_t kTileA = 128 * kKt * 2;  // one 128-row A tile per stage
constexpr uint32_t kSbo = kKt * 16;     // bytes between 8-row groups
constexpr uint32_t kLbo = 128;          // bytes between core matrices along K
constexpr uint32_t kZCols = 128;        // Z products start 128 columns into a buffer
constexpr uint32_t kTmemCols = 512;     // two accumulator buffers of 256 columns

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

// fp16 pair word J of a run: +-1 for dense probes; for sparse probes the
// magnitude is kept only where the activity bit (same position in `act`) is
// set, so inactive coordinates are +-0.
template <bool SPARSE, int J>
__device__ __forceinline__ uint32_t z_pair(uint32_t raw, uint32_t act) {
  if (!SPARSE) return pm_pair<J>(raw, 0x3C003C00u);
  // activity bits at the sign positions (bits 15 and 31), each spread over
  // its 16-bit half by a byte permute that replicates the top bit of bytes 1
  // and 3: a mask of 1.0 magnitudes where the coordinate is active
  uint32_t m;
  asm("prmt.b32 %0, %1, %2, 0xBB99;" : "=r"(m) : "r"(act << (15 - J)), "r"(0u));
  return ((raw << (15 - J)) & 0x80008000u) | (m & 0x3C003C00u);
}

// Writes 32 elements of a Z tile row in the canonical K-major layout from one
// raw sign word (and, for sparse probes, its activity word); `row` points at
// the first element, consecutive 8-element chunks are 128 bytes apart.
template <bool SPARSE>
__device__ __forceinline__ void store_z_row_at(uint8_t* row, uint32_t raw, uint32_t act) {
  uint4 c0, c1, c2, c3;
  c0.x = z_pair<SPARSE, 0>(raw, act);   c0.y = z_pair<SPARSE, 1>(raw, act);
  c0.z = z_pair<SPARSE, 2>(raw, act);   c0.w = z_pair<SPARSE, 3>(raw, act);
  c1.x = z_pair<SPARSE, 4>(raw, act);   c1.y = z_pair<SPARSE, 5>(raw, act);
  c1.z = z_pair<SPARSE, 6>(raw, act);   c1.w = z_pair<SPARSE, 7>(raw, act);
  c2.x = z_pair<SPARSE, 8>(raw, act);   c2.y = z_pair<SPARSE, 9>(raw, act);
  c2.z = z_pair<SPARSE, 10>(raw, act);  c2.w = z_pair<SPARSE, 11>(raw, act);
  c3.x = z_pair<SPARSE, 12>(raw, act);  c3.y = z_pair<SPARSE, 13>(raw, act);
  c3.z = z_pair<SPARSE, 14>(raw, act);  c3.w = z_pair<SPARSE, 15>(raw, act);
  *reinterpret_cast<uint4*>(row) = c0;
  *reinterpret_cast<uint4*>(row + 128) = c1;
  *reinterpret_cast<uint4*>(row + 256) = c2;
  *reinterpret_cast<uint4*>(row + 384) = c3;
}

// The MMAs of one stage, fully unrolled over K (NP = probes with a Z tile):
// W x operand into [0, rowsB) and Z_p x operand_p into kZCols + 2 Bp p.  The
// descriptors arrive as their low words (start address of the stage's tiles;
// a step along K or to the next probe is an addition), so the issuing thread
// spends a few instructions per MMA and keeps the tensor pipe fed.
template <int NP>
__device__ __forceinline__ void issue_stage(uint32_t d, uint32_t a_lo, uint32_t b_lo, uint32_t z_lo,
                                            uint32_t hi, uint32_t zp_step, uint32_t bp_step,
                                            uint32_t idesc_w, uint32_t idesc_z, uint32_t dz_step,
                                            uint32_t acc0) {
#pragma unroll
  for (int k16 = 0; k16 < kKt / 16; ++k16) {
    const uint32_t ko = (uint32_t)k16 * 16;
    const uint32_t acc = k16 > 0 ? 1u : acc0;
    mma_f16_ss_lohi(d, a_lo + ko, hi, b_lo + ko, hi, idesc_w, acc);
    if (NP >= 1) mma_f16_ss_lohi(d + kZCols, z_lo + ko, hi, b_lo + ko, hi, idesc_z, acc);
    if (NP >= 2)
      mma_f16_ss_lohi(d + kZCols + dz_step, z_lo + ko + zp_step, hi, b_lo + ko + bp_step, hi,
                      idesc_z, acc);
  }
}

// ---------------------------------------------------------------------------
// Persistent warp-specialised kernel.  One CTA per SM walks a static list of
// tasks (blockIdx.x, blockIdx.x + n_ctas, ...; the head launch appends
// n_ctas-independent blocks for the embedding operand, so the stride is
// n_ctas, not the grid size).  Roles:
//   warps 0..2    loaders: warp j bulk-copies the A tile and the operand
//                 group tile of every stage that uses ring slot j (16 KB
//                 copies; the copies of one issuing thread complete one
//                 after another, so each slot has its own issuer);
//   warp 3        MMA issuer: W x operand and Z_p x operand_p per stage into
//                 one of two TMEM accumulator buffers (256 columns each);
//   warps 4..11   Z generators: the +-1 tiles of the stage, from Philox
//                 (one (probe, row) pair per thread);
//   warps 12..19  epilogue: reads a finished accumulator buffer while the
//                 MMAs of the next task fill the other one; warp w reads the
//                 TMEM lanes of quarter w % 4 for probe (w - 12) / 4.
// Barriers: full (the slot's copies landed and its Z tiles are written),
// slot_free (the slot's MMAs are done), acc_full (a buffer's task is
// accumulated), acc_empty (its epilogue has read it), mma_done (all MMAs of
// the CTA completed).  Every wait is bounded (wait_or_abort, mbar_wait).
// ---------------------------------------------------------------------------
constexpr int kMmaWarp = kLoaders;
constexpr int kZWarp0 = kMmaWarp + 1;
constexpr int kEpiWarp0 = kZWarp0 + kZWarps;
constexpr int kAccCols = 256;

struct Ctl {
  uint64_t full[kStages];
  uint64_t slot_free[kStages];
  uint64_t acc_full[2];
  uint64_t acc_empty[2];
  uint64_t mma_done;
  uint32_t tmem_slot;
  volatile int abort;
};

// A wait that times out records SOMA_ERR_TIMEOUT in the status word and sets
// the CTA's abort flag; a wait that is still pending sees the flag within 64
// polls and returns false, so the CTA winds down without issuing further
// copies or MMAs.  A phase that is already complete costs one poll and no
// read of the flag (the flag shares the shared-memory pipe with the
// epilogue's shuffles, and every handoff of the main loop passes here).
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort,
                                              int* status) {
  if (mbar_try_wait(bar, parity)) return true;
  for (uint32_t n = 1; n < (1u << 22); ++n) {
    if ((n & 63u) == 0 && *abort) return false;
    if (mbar_try_wait(bar, parity)) return true;
  }
  *abort = 1;
  atomicCAS(status, 0, kStatusTimeout);
  return false;
}

struct TcArgs {
  Sweep sw;
  TcGeom g;
  int t;
  const uint8_t* w16;    // [N][MT][S] A tiles
  const uint8_t* wo16;   // [N][2][Sh] A tiles
  const uint8_t* op_in;  // [N][S][G] operand group tiles of this timestep
  uint8_t* op_out;       // next timestep's operand
  float* cst;            // [N*n*2][Hp][Bp] cell state
  float* pm;             // [N*n*2][B][T][2] head max partials
  float* ps;             // sum-exp partials
  float* ply;            // [N*n*2][B][T] target logits
  int* status;
};

// One task: (expert, row tile, probe group).  For the gate the row tile is
// 32 hidden units (128 gate rows); for the head it is a 128-row vocabulary
// half.
struct Task {
  int e, m, grp, p_valid;
  const uint8_t* a;  // A tile of stage 0
  const uint8_t* b;  // operand group tile of stage 0
};

template <bool HEAD>
__device__ __forceinline__ Task make_task(const TcArgs& a, int task) {
  const TcGeom& g = a.g;
  Task T;
  T.grp = task % g.G;
  const int rows = HEAD ? 2 : g.MT;
  T.m = (task / g.G) % rows;
  T.e = task / (g.G * rows);
  T.p_valid = min(g.P, a.sw.n_pert - T.grp * g.P);
  if (HEAD) {
    T.a = a.wo16 + (((size_t)T.e * 2 + T.m) * g.Sh) * kTileA;
    T.b = a.op_in + (((size_t)T.e * g.S + g.Sx) * g.G + T.grp) * g.tileB;
  } else {
    T.a = a.w16 + (((size_t)T.e * g.MT + T.m) * g.S) * kTileA;
    T.b = a.op_in + (((size_t)T.e * g.S) * g.G + T.grp) * g.tileB;
  }
  return T;
}

// Flat parameter index of element (row r, k = 0) of the stage-st Z run.
template <bool HEAD>
__device__ __forceinline__ int64_t z_param(const TcArgs& a, const Task& T, int r, int st) {
  const Layout& L = a.sw.lay;
  if (HEAD) return L.w_out + (int64_t)(128 * T.m + r) * a.g.H + (int64_t)kKt * st;
  const int64_t R = (int64_t)tile_gate(r) * a.g.H + 32 * T.m + tile_unit(r);  // W row of tile row r
  return st < a.g.Sx ? L.w_ih + R * a.g.E + (int64_t)kKt * st
                     : L.w_hh + R * a.g.H + (int64_t)kKt * (st - a.g.Sx);
}

// Gate epilogue of one task for one warp: probe p, TMEM lane quarter q4
// (units 8 q4 .. 8 q4 + 7 of the tile).  Thread l runs the cells of unit
// l / 4 for sequences b0 + l % 4 and b0 + 4 + l % 4 of every 8-sequence
// chunk, both signs, in fp32: 16x128b loads give it all four gates of its
// unit (gate-major rows), so no data moves between threads.  Cell state
// layout: [e, i][Hp][Bp][sign].
__device__ void gate_epilogue(const TcArgs& a, const Task& T, uint32_t tacc, const ProbeKey& pk,
                              int q4, int p) {
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  const Layout& L = s.lay;
  const int lane = threadIdx.x & 31;
  const int H = g.H;
  const float eps = s.eps;
  const bool do_z = eps != 0.f;
  const float* th = s.params + (int64_t)T.e * L.P;
  // bias and its probe sign for the row in this lane's TMEM lane, handed to
  // the threads that run that row's unit
  float bias_r = 0.f, dbias_r = 0.f;
  {
    const int Ur = 32 * T.m + tile_unit(32 * q4 + lane);
    if (Ur < H) {
      const int64_t pb = L.b + (int64_t)tile_gate(32 * q4 + lane) * H + Ur;
      bias_r = th[pb];
      if (do_z) {
        const ProbeBits zb = probe_bits(pk, pb, s.sparse);
        dbias_r = eps_z(zb.neg & 1u, zb.act & 1u, eps);
      }
    }
  }
  const int u8 = lane >> 2, bq = lane & 3;
  float bias[4], dbias[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    bias[k] = __shfl_sync(0xffffffffu, bias_r, 8 * k + u8);
    dbias[k] = __shfl_sync(0xffffffffu, dbias_r, 8 * k + u8);
  }
  const int U = 32 * T.m + 8 * q4 + u8;
  const bool unit_ok = U < H;
  // a stage of the next operand holds kKt / 32 of the 32-unit row tiles
  uint8_t* out_tile =
      a.op_out + (((size_t)T.e * g.S + g.Sx + 32 * T.m / kKt) * g.G + T.grp) * g.tileB;
  const int kk = 32 * T.m % kKt + 8 * q4 + u8;
  const int i = T.grp * g.P + p;
  float2* cell = reinterpret_cast<float2*>(a.cst) +
                 (((int64_t)T.e * s.n_pert + i) * g.Hp + U) * (int64_t)g.Bp;
  const uint32_t tq = tacc + ((uint32_t)(32 * q4) << 16);  // gates 0, 1
  const uint32_t tq2 = tq + (16u << 16);                    // gates 2, 3
  for (int b0 = 0; b0 < g.Bp; b0 += 8) {
    float2 cprev[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
    if (unit_ok && a.t > 0) {
      cprev[0] = cell[b0 + bq];
      cprev[1] = cell[b0 + 4 + bq];
    }
    // [seq half][gate]: W vbar, W dv, Z vbar, Z dv
    uint32_t wv[2][4], wd[2][4], zv[2][4], zd[2][4];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const uint32_t cw = (uint32_t)(2 * g.Bp * p + b0 + 4 * h);
      tmem_ld_16x128b(tq + cw, wv[h][0], wv[h][1]);
      tmem_ld_16x128b(tq2 + cw, wv[h][2], wv[h][3]);
      tmem_ld_16x128b(tq + cw + g.Bp, wd[h][0], wd[h][1]);
      tmem_ld_16x128b(tq2 + cw + g.Bp, wd[h][2], wd[h][3]);
      if (do_z) {
        tmem_ld_16x128b(tq + kZCols + cw, zv[h][0], zv[h][1]);
        tmem_ld_16x128b(tq2 + kZCols + cw, zv[h][2], zv[h][3]);
        tmem_ld_16x128b(tq + kZCols + cw + g.Bp, zd[h][0], zd[h][1]);
        tmem_ld_16x128b(tq2 + kZCols + cw + g.Bp, zd[h][2], zd[h][3]);
      }
    }
    tmem_wait_ld();
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      float actp[4], actm[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float zvk = do_z ? __uint_as_float(zv[h][k]) : 0.f;
        const float zdk = do_z ? __uint_as_float(zd[h][k]) : 0.f;
        const float C = fmaf(eps, zdk, __uint_as_float(wv[h][k])) + bias[k];
        const float D = fmaf(eps, zvk, __uint_as_float(wd[h][k])) + dbias[k];
        if (k == 2) {  // g: tanh(x) = 2 sigmoid(2x) - 1
          actp[k] = fmaf(sigm(2.f * (C + D)), 2.f, -1.f);
          actm[k] = fmaf(sigm(2.f * (C - D)), 2.f, -1.f);
        } else {
          actp[k] = sigm(C + D);
          actm[k] = sigm(C - D);
        }
      }
      const float cp = fmaf(actp[1], cprev[h].x, actp[0] * actp[2]);
      const float cm = fmaf(actm[1], cprev[h].y, actm[0] * actm[2]);
      const float hp = actp[3] * fmaf(sigm(2.f * cp), 2.f, -1.f);
      const float hm = actm[3] * fmaf(sigm(2.f * cm), 2.f, -1.f);
      const int b = b0 + 4 * h + bq;
      if (unit_ok) {
        cell[b] = make_float2(cp, cm);
        if (b < s.B) {
          const int row = 2 * g.Bp * p + b;
          *reinterpret_cast<__half*>(out_tile + kmajor_offset(row, kk, kKt)) =
              __float2half_rn(0.5f * (hp + hm));
          *reinterpret_cast<__half*>(out_tile + kmajor_offset(row + g.Bp, kk, kKt)) =
              __float2half_rn(0.5f * (hp - hm));
        }
      }
    }
  }
}

// Head epilogue of one task: logits +- of the 32 vocabulary rows of the
// warp's lane quarter for each probe the warp runs.  16x128b loads give
// thread l four rows (l / 4 + {0, 8, 16, 24}) of sequence b0 + l % 4, so
// the per-(sequence, sign) max and sum-exp over the quarter reduce four rows
// in registers and then across the eight threads of that sequence (three
// shuffle rounds).  The four quarters of the half merge through shared
// memory (`red`, [P][Bp][2][4]); the thread holding the target byte's row
// writes the target logit.
__device__ void head_epilogue(const TcArgs& a, const Task& T, uint32_t tacc, int q4, int ew,
                              float2* red) {
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  const Layout& L = s.lay;
  const int lane = threadIdx.x & 31;
  const float eps = s.eps;
  const bool do_z = eps != 0.f;
  const float* th = s.params + (int64_t)T.e * L.P;
  const int vq = 128 * T.m + 32 * q4;  // first vocabulary row of the quarter
  const float bo_r = th[L.b_out + vq + lane];
  const int t = a.t;
  const int bq = lane & 3, r4 = lane >> 2;
  // rows of this thread: vq + r4 + 8 k, k = 0..3 (k = 2 h + reg)
  float bo[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) bo[k] = __shfl_sync(0xffffffffu, bo_r, r4 + 8 * k);
  const uint32_t tq = tacc + ((uint32_t)(32 * q4) << 16);
  const uint32_t tq2 = tq + (16u << 16);
  for (int p = ew >> 2; p < g.P; p += kEpiProbeStep) {
    if (p >= T.p_valid) continue;
    const int i = T.grp * g.P + p;
    float dbo[4] = {0.f, 0.f, 0.f, 0.f};
    if (do_z) {
      const ProbeKey pk = make_probe_key(s.seed, s.step, (uint32_t)T.e, (uint32_t)i);
      const ProbeBits zb = probe_bits(pk, L.b_out + vq + lane, s.sparse);
      const float dbo_r = eps_z(zb.neg & 1u, zb.act & 1u, eps);
#pragma unroll
      for (int k = 0; k < 4; ++k) dbo[k] = __shfl_sync(0xffffffffu, dbo_r, r4 + 8 * k);
    }
    const int64_t lane_plus = ((int64_t)T.e * s.n_pert + i) * 2;
    for (int b0 = 0; b0 < g.Bp; b0 += 4) {
      // [k]: W vbar, W dv, Z vbar, Z dv of row r4 + 8 k, sequence b0 + bq
      uint32_t wv[4], wd[4], zv[4] = {0u, 0u, 0u, 0u}, zd[4] = {0u, 0u, 0u, 0u};
      const uint32_t cw = (uint32_t)(2 * g.Bp * p + b0);
      tmem_ld_16x128b(tq + cw, wv[0], wv[1]);
      tmem_ld_16x128b(tq2 + cw, wv[2], wv[3]);
      tmem_ld_16x128b(tq + cw + g.Bp, wd[0], wd[1]);
      tmem_ld_16x128b(tq2 + cw + g.Bp, wd[2], wd[3]);
      if (do_z) {
        tmem_ld_16x128b(tq + kZCols + cw, zv[0], zv[1]);
        tmem_ld_16x128b(tq2 + kZCols + cw, zv[2], zv[3]);
        tmem_ld_16x128b(tq + kZCols + cw + g.Bp, zd[0], zd[1]);
        tmem_ld_16x128b(tq2 + kZCols + cw + g.Bp, zd[2], zd[3]);
      }
      tmem_wait_ld();
      float lp[4], lm[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float C = fmaf(eps, __uint_as_float(zd[k]), __uint_as_float(wv[k])) + bo[k];
        const float D = fmaf(eps, __uint_as_float(zv[k]), __uint_as_float(wd[k])) + dbo[k];
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
        red[((p * g.Bp + b) * 2 + 0) * 4 + q4] = make_float2(mp, sp);
        red[((p * g.Bp + b) * 2 + 1) * 4 + q4] = make_float2(mm, sm_);
      }
      if (b < s.B) {
        const int y = s.bytes[seq_offset(s, T.e, i, b) + t + 1] - vq - r4;
        // y = 8 k for the thread that holds the target row
        if (y >= 0 && y < 32 && (y & 7) == 0) {
          const int k = y >> 3;
          const float vp = k == 0 ? lp[0] : k == 1 ? lp[1] : k == 2 ? lp[2] : lp[3];
          const float vm = k == 0 ? lm[0] : k == 1 ? lm[1] : k == 2 ? lm[2] : lm[3];
          a.ply[((lane_plus + 0) * s.B + b) * (int64_t)s.T + t] = vp;
          a.ply[((lane_plus + 1) * s.B + b) * (int64_t)s.T + t] = vm;
        }
      }
    }
  }
  // all epilogue warps: partials of this task are in `red`
  asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
  const int et = threadIdx.x - kEpiWarp0 * 32;
  const int n_red = T.p_valid * g.Bp * 2;
  for (int idx = et; idx < n_red; idx += kEpiWarps * 32) {
    const int sgn = idx & 1;
    const int pb = idx >> 1;
    const int pp = pb / g.Bp, b = pb % g.Bp;
    if (b >= s.B) continue;
    const float2* q = red + (size_t)idx * 4;
    const float M = fmaxf(fmaxf(q[0].x, q[1].x), fmaxf(q[2].x, q[3].x));
    float S = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) S += q[k].y * __expf(q[k].x - M);
    const int i = T.grp * g.P + pp;
    const int64_t ln = ((int64_t)T.e * s.n_pert + i) * 2 + sgn;
    const int64_t o = ((ln * s.B + b) * (int64_t)s.T + t) * 2 + T.m;
    a.pm[o] = M;
    a.ps[o] = S;
  }
  // `red` is reused by the next task
  asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
}

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

__device__ void xpart_block(const TcArgs& a, uint8_t* op, int t, int blk);

// grid: min(tasks, SMs) persistent CTAs (+ for the head, the embedding-part
// blocks of the next timestep's operand), kThreads threads.
template <bool HEAD, bool SPARSE>
__global__ void __launch_bounds__(kThreads, 1) tc_persistent_kernel(const TcArgs a, int n_tasks,
                                                                    int n_ctas) {
  extern __shared__ uint8_t dyn_smem[];
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  if (HEAD && (int)blockIdx.x >= n_ctas) {
    // the embedding part of timestep t + 1's operand (the head reads only
    // the h part of the same buffer)
    if (a.t + 1 < s.T)
      xpart_block(a, const_cast<uint8_t*>(a.op_in), a.t + 1, blockIdx.x - n_ctas);
    return;
  }
  uint8_t* smem = align1024(dyn_smem);
  const StageLayout SL = stage_layout(g);
  Ctl* ctl = reinterpret_cast<Ctl*>(smem + kStages * SL.bytes);
  float2* red = reinterpret_cast<float2*>(smem + kStages * SL.bytes + 1024);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nst = HEAD ? g.Sh : g.S;
  const bool do_z = s.eps != 0.f;
  int* status = a.status;
  volatile int* abort = &ctl->abort;

  if (tid == 0) {
    ctl->abort = 0;
    for (int q = 0; q < kStages; ++q) {
      // the loader's arrival (with the copies' bytes) and, when probes are
      // generated, one arrival per Z warp: the MMA warp waits once per stage
      mbar_init(&ctl->full[q], do_z ? 1 + kZWarps : 1);
      mbar_init(&ctl->slot_free[q], 1);
    }
    for (int q = 0; q < 2; ++q) {
      mbar_init(&ctl->acc_full[q], 1);
      mbar_init(&ctl->acc_empty[q], kEpiWarps);
    }
    mbar_init(&ctl->mma_done, 1);
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(&ctl->tmem_slot, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctl->tmem_slot;

  if (warp < kLoaders) {
    // ---------------------------------------------------------------- loaders
    // the whole warp walks the stages (so that it never sits diverged at the
    // CTA barrier); lanes 0 and 1 issue one copy each (the copies of one
    // thread complete one after another)
    uint32_t gs = 0;
    int last_use = -1;
    for (int task = blockIdx.x; task < n_tasks; task += n_ctas) {
      const Task T = make_task<HEAD>(a, task);
      for (int st = 0; st < nst; ++st, ++gs) {
        const int q = gs % kStages;
        if (q != warp) continue;
        const uint32_t use = gs / kStages;
        if (gs >= kStages && !wait_or_abort(&ctl->slot_free[q], (use - 1) & 1u, abort, status))
          continue;
        uint8_t* slot = smem + q * SL.bytes;
        if (lane == 0) mbar_arrive_expect_tx(&ctl->full[q], kTileA + g.tileB);
        __syncwarp();
        if (lane == 0)
          bulk_g2s(slot + SL.a_off, T.a + (size_t)st * kTileA, kTileA, &ctl->full[q]);
        else if (lane == 1)
          bulk_g2s(slot + SL.b_off, T.b + (size_t)st * g.G * g.tileB, g.tileB, &ctl->full[q]);
        last_use = (int)use;
        __syncwarp();
      }
    }
    // copies still in flight land before the CTA exits.  After an abort the
    // Z warps stop arriving and this wait runs to its bound instead; copies
    // take microseconds, the bound is tenths of a second.
    if (last_use >= 0) mbar_wait(&ctl->full[warp], (uint32_t)last_use & 1u);
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    // the whole warp waits; lane 0 issues the MMAs and commits
    {
      const uint32_t idesc_w = idesc_f16_f32(128, g.rowsB);
      const uint32_t idesc_z = idesc_f16_f32(128, 2 * g.Bp);
      // descriptors of slot 0; slot q is q * SL.bytes further, k16 = 1 is
      // 256 bytes further (two core matrices along K)
      const uint64_t d0 = smem_desc(smem_u32(smem), kLbo, kSbo);
      const uint32_t hi = (uint32_t)(d0 >> 32);
      const uint32_t lo0 = (uint32_t)d0;
      const uint32_t slot_step = SL.bytes >> 4;
      const uint32_t a_lo0 = lo0 + (SL.a_off >> 4), b_lo0 = lo0 + (SL.b_off >> 4);
      const uint32_t z_lo0 = lo0 + (SL.z_off >> 4);
      const uint32_t zp_step = kTileA >> 4;                       // next probe's Z tile
      const uint32_t bp_step = (uint32_t)(2 * g.Bp / 8) * (kSbo >> 4);  // next probe's rows
      const uint32_t dz_step = (uint32_t)(2 * g.Bp);                    // next probe's columns
      uint32_t gs = 0;
      int k = 0;
      for (int task = blockIdx.x; task < n_tasks; task += n_ctas, ++k) {
        const Task T = make_task<HEAD>(a, task);
        const int buf = k & 1;
        if (k >= 2) wait_or_abort(&ctl->acc_empty[buf], (uint32_t)((k >> 1) - 1) & 1u, abort, status);
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(buf * kAccCols);
        const int np = do_z ? T.p_valid : 0;
        for (int st = 0; st < nst; ++st, ++gs) {
          const int q = gs % kStages;
          const uint32_t use = gs / kStages;
          const bool ok = wait_or_abort(&ctl->full[q], use & 1u, abort, status);
          tc_fence_after();
          if (ok && lane == 0) {
            const uint32_t so = (uint32_t)q * slot_step;
            const uint32_t acc0 = st > 0 ? 1u : 0u;
            if (np == 2)
              issue_stage<2>(d, a_lo0 + so, b_lo0 + so, z_lo0 + so, hi, zp_step, bp_step, idesc_w,
                             idesc_z, dz_step, acc0);
            else if (np == 1)
              issue_stage<1>(d, a_lo0 + so, b_lo0 + so, z_lo0 + so, hi, zp_step, bp_step, idesc_w,
                             idesc_z, dz_step, acc0);
            else
              issue_stage<0>(d, a_lo0 + so, b_lo0 + so, z_lo0 + so, hi, zp_step, bp_step, idesc_w,
                             idesc_z, dz_step, acc0);
          }
          if (lane == 0) mma_commit(&ctl->slot_free[q]);
          __syncwarp();
        }
        if (lane == 0) mma_commit(&ctl->acc_full[buf]);
        __syncwarp();
      }
      // every MMA of this CTA completes before its tensor memory is freed
      if (lane == 0) mma_commit(&ctl->mma_done);
      mbar_wait(&ctl->mma_done, 0);
    }
  } else if (warp < kEpiWarp0) {
    // --------------------------------------------------------- Z generators
    // Thread (probe gtid / 128, row gtid % 128).  The raw words of the next
    // stage are drawn before waiting for its slot, so the Philox rounds
    // overlap the wait instead of following it.
    if (do_z) {
      const int gtid = tid - kZWarp0 * 32;
      const int r = gtid & 127, pz = gtid >> 7;
      uint32_t gs = 0;
      for (int task = blockIdx.x; task < n_tasks; task += n_ctas) {
        const Task T = make_task<HEAD>(a, task);
        const bool active = pz < T.p_valid;
        const ProbeKey pk =
            make_probe_key(s.seed, s.step, (uint32_t)T.e, (uint32_t)(T.grp * g.P + pz));
        const ProbeKey pka = activity_key(pk);
        ZSlot cache, cache_a;
        cache.blk = 0xFFFFFFFFu;
        cache_a.blk = 0xFFFFFFFFu;
        const int split = HEAD ? nst : g.Sx;
        const int64_t seg0 = z_param<HEAD>(a, T, r, 0);
        const int64_t seg1 = z_param<HEAD>(a, T, r, split) - (int64_t)kKt * split;
        uint8_t* zrow = smem + SL.z_off + pz * kTileA + kmajor_offset(r, 0, kKt);
        uint32_t raw[kKt / 32] = {}, act[kKt / 32] = {};
        if (active) {
#pragma unroll
          for (int w = 0; w < kKt / 32; ++w) {
            raw[w] = z_run_raw(pk, seg0 + 32 * w, cache);
            if (SPARSE) act[w] = z_run_raw(pka, seg0 + 32 * w, cache_a);
          }
        }
        for (int st = 0; st < nst; ++st, ++gs) {
          const int q = gs % kStages;
          const uint32_t use = gs / kStages;
          // after an abort the generators stop: an arrival on a phase that
          // can no longer complete would overfill it
          if (gs >= kStages && !wait_or_abort(&ctl->slot_free[q], (use - 1) & 1u, abort, status))
            break;
          if (active) {
            uint8_t* zr = zrow + q * SL.bytes;
#pragma unroll
            for (int w = 0; w < kKt / 32; ++w)
              store_z_row_at<SPARSE>(zr + w * 4 * 128, raw[w], act[w]);
          }
          fence_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&ctl->full[q]);
          if (active && st + 1 < nst) {
            const int64_t p1 = (st + 1 < split ? seg0 : seg1) + (int64_t)kKt * (st + 1);
#pragma unroll
            for (int w = 0; w < kKt / 32; ++w) {
              raw[w] = z_run_raw(pk, p1 + 32 * w, cache);
              if (SPARSE) act[w] = z_run_raw(pka, p1 + 32 * w, cache_a);
            }
          }
        }
      }
    }
  } else {
    // --------------------------------------------------------------- epilogue
    const int ew = warp - kEpiWarp0;
    const int q4 = warp & 3;
    int k = 0;
    for (int task = blockIdx.x; task < n_tasks; task += n_ctas, ++k) {
      const Task T = make_task<HEAD>(a, task);
      const int buf = k & 1;
      wait_or_abort(&ctl->acc_full[buf], (uint32_t)(k >> 1) & 1u, abort, status);
      tc_fence_after();
      const uint32_t tacc = tmem + (uint32_t)(buf * kAccCols);
      if (HEAD) {
        head_epilogue(a, T, tacc, q4, ew, red);
      } else {
        for (int p = ew >> 2; p < T.p_valid; p += kEpiProbeStep) {
          const ProbeKey pk =
              make_probe_key(s.seed, s.step, (uint32_t)T.e, (uint32_t)(T.grp * g.P + p));
          gate_epilogue(a, T, tacc, pk, q4, p);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl->acc_empty[buf]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, kTmemCols);
}

// Embedding part of the operand of timestep t: x = Emb[byte_t], dx = eps z_emb.
// Block `blk` of Sx * G * N writes one (expert, stage, group) tile.
__device__ void xpart_block(const TcArgs& a, uint8_t* op, int t, int blk) {
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  const int st = (blk / g.G) % g.Sx, grp = blk % g.G;
  const int e = blk / (g.G * g.Sx);
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
      const int y = s.bytes[seq_offset(s, e, i, b) + t];
      const int64_t p0 = L.emb + (int64_t)y * g.E + k0;
      ProbeBits bits = {0u, 0u};
      if (delta && s.eps != 0.f)
        bits = probe_bits(make_probe_key(s.seed, s.step, (uint32_t)e, (uint32_t)i), p0, s.sparse);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        float x = 0.f;
        if (k0 + j < g.E)
          x = delta ? eps_z((bits.neg >> j) & 1u, (bits.act >> j) & 1u, s.eps) : th[p0 + j];
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

__global__ void xpart_kernel(const TcArgs a, uint8_t* op, int t) {
  xpart_block(a, op, t, blockIdx.x);
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
    const int U = 32 * m + tile_unit(r), gate = tile_gate(r);
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
  // ring slots, the control block (1 KB), the head's reduction buffer
  // [P][Bp][2][4] float2 and alignment slack
  const size_t red = (size_t)g.P * g.Bp * 2 * 4 * sizeof(float2);
  return (size_t)kStages * stage_layout(g).bytes + 1024 + red + 1024;
}

int sm_count() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  if (!cached[dev]) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 1;
    cached[dev] = n;
  }
  return cached[dev];
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
  int P = 64 / g.Bp;  // rowsB = 2 Bp P <= 128 TMEM columns per product
  if (P > 2) P = 2;
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

bool tc_supported(int B) { return B >= 1 && B <= 64; }

TcSizes tc_sizes(const TcGeom& g) {
  TcSizes z;
  const size_t N = (size_t)g.n_experts, n = (size_t)g.n_pert;
  z.w16 = N * g.MT * g.S * kTileA;
  z.wo16 = N * 2 * g.Sh * kTileA;
  z.op = N * g.S * g.G * g.tileB;
  z.cst = N * n * 2 * (size_t)g.Hp * g.Bp * sizeof(float);
  z.pm = N * n * 2 * g.B * (size_t)g.T * 2 * sizeof(float);
  z.ply = N * n * 2 * g.B * (size_t)g.T * sizeof(float);
  return z;
}

cudaError_t launch_forward_tc(const Sweep& s, const TcGeom& g, const TcBuffers& tb, int* status,
                              cudaStream_t stream) {
  const size_t smem = kernel_smem_bytes(g);
  auto gate_kernel = s.sparse ? tc_persistent_kernel<false, true> : tc_persistent_kernel<false, false>;
  auto head_kernel = s.sparse ? tc_persistent_kernel<true, true> : tc_persistent_kernel<true, false>;
  cudaError_t e = cudaFuncSetAttribute(gate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(head_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const TcSizes z = tc_sizes(g);
  TcArgs a;
  a.sw = s;
  a.g = g;
  a.t = 0;
  a.w16 = tb.w16;
  a.wo16 = tb.wo16;
  a.op_in = tb.op[0];
  a.op_out = tb.op[1];
  a.cst = tb.cst;
  a.pm = tb.pm;
  a.ps = tb.ps;
  a.ply = tb.ply;
  a.status = status;

  trace_begin(SOMA_TRACE_PREP, stream);
  prep_tiles_kernel<<<dim3(g.MT * g.S + 2 * g.Sh, g.n_experts), 128, 0, stream>>>(a);
  cudaMemsetAsync(tb.op[0], 0, z.op, stream);
  cudaMemsetAsync(tb.op[1], 0, z.op, stream);
  const int xblocks = g.n_experts * g.Sx * g.G;
  xpart_kernel<<<xblocks, 128, 0, stream>>>(a, tb.op[0], 0);
  trace_end(SOMA_TRACE_PREP, stream);

  const int sms = sm_count();
  const int gate_tasks = g.n_experts * g.MT * g.G;
  const int head_tasks = g.n_experts * 2 * g.G;
  const int gate_ctas = gate_tasks < sms ? gate_tasks : sms;
  const int head_ctas = head_tasks < sms ? head_tasks : sms;
  for (int t = 0; t < s.T; ++t) {
    a.t = t;
    a.op_in = tb.op[t & 1];
    a.op_out = tb.op[(t + 1) & 1];
    trace_begin(SOMA_TRACE_GATE, stream);
    gate_kernel<<<gate_ctas, kThreads, smem, stream>>>(a, gate_tasks, gate_ctas);
    trace_end(SOMA_TRACE_GATE, stream);
    // head of timestep t (h part of the operand of t + 1) and, in the same
    // launch, the embedding part of that operand
    a.op_in = tb.op[(t + 1) & 1];
    trace_begin(SOMA_TRACE_HEAD, stream);
    head_kernel<<<head_ctas + (t + 1 < s.T ? xblocks : 0), kThreads, smem, stream>>>(
        a, head_tasks, head_ctas);
    trace_end(SOMA_TRACE_HEAD, stream);
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
