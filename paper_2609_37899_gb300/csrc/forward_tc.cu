// forward_tc.cu -- tensor-core (tcgen05 / TMEM) forward sweep of the
// perturbed LSTM experts in the mean/difference form.
//
// For one expert e and probe i, the two antithetic copies of the LSTM take
// inputs v+- = [x+-; h+-_{t-1}].  Write vbar = (v+ + v-)/2 and the scaled half
// difference dhat = (v+ - v-)/(2 eps), an O(1) quantity.  With the perturbed
// weights W +- eps Z (Z = z_{e,i} reshaped, entries +-1, or 0 for inactive
// sparse coordinates),
//   (W +- eps Z)(vbar +- eps dhat) = [W vbar + eps^2 Z dhat] +- eps [W dhat + Z vbar]
// exactly, so the gate pre-activations are a+- = C +- eps D with
//   C = W vbar + eps^2 (Z dhat) + b,       D = W dhat + Z vbar + z_b.
// The products are fp16 x fp16 -> fp32 tensor-core GEMMs and eps multiplies
// only in fp32 (epilogue), so no operand ever holds a rounded w +- eps z, and
// the rounding of dhat is relative (2^-11) at any eps: the difference of the
// two copies is never formed by cancelling two rounded numbers, and never
// falls into fp16's subnormal range.  The cell state c+- and the
// activations are fp32 per sign.  The output head uses the same split.
//
// Operand tiles.  P <= 2 probes share one operand group tile; its rows are,
// in blocks of Bp sequences,
//   P = 2:  [eps^2 dhat_0 | vbar_0 | dhat_0 | dhat_1 | vbar_1 | eps^2 dhat_1]
//   P = 1:  [eps^2 dhat_0 | vbar_0 | dhat_0]
// so that every product lands in one accumulator per probe, [C_p | D_p]:
//   W x rows Bp .. (1 + 2P) Bp  -> columns [C_0 | D_0 | D_1 | C_1] (one MMA),
//   Z_0 x rows 0 .. 2 Bp        -> [C_0 | D_0]    (eps^2 dhat_0 -> C, vbar_0 -> D),
//   Z_1 x rows 4 Bp .. 6 Bp     -> [D_1 | C_1]    (vbar_1 -> D, eps^2 dhat_1 -> C).
// The eps^2 dhat rows carry a term of order eps^2 |Z dhat|; their fp16
// rounding (subnormal below |eps^2 dhat| = 6e-5) costs at most 3e-8 per
// element, below the rounding of W vbar that C already carries.
//
// One cooperative launch of one persistent kernel runs the whole sweep, in
// phases t = 0 .. T with two kinds of task:
//   gate tasks  (expert, 32-unit row tile, group of P probes), t < T: the
//               W tile (shared memory) and the P probe tiles Z_p (expanded
//               from a per-sweep table of raw Philox words straight into
//               tensor memory, the A operand of a tcgen05.mma with A in
//               TMEM) against the operand tiles of timestep t; epilogue:
//               gates, cell update, the h part of the operand of t + 1;
//   head tasks  (expert, 128-row vocabulary half, probe group) of timestep
//               t - 1, t >= 1: the same MMAs over the h part of the same
//               operand (h_{t-1}), then per (sequence, sign) max and sum-exp
//               partials of the half and the target logit.
// Per-group phase counters in global memory order the phases without a grid
// barrier.  Before the sweep, one launch writes the weight tiles and the
// probe-word tables, and a second the embedding part of every timestep's
// operand.  A final reduction merges the two halves into per-target NLL and
// the per-(expert, probe) losses and coefficients.
#include <cuda_fp16.h>

#define SOMA_CHECK_FILE 1
#include "checked.cuh"
#include "soma_api.h"
#include "soma_device.cuh"
#include "soma_launch.h"
#include "tc_primitives.cuh"

namespace soma {

using namespace tc;

namespace {

constexpr int kStages = 5;       // ring slots of the shared-memory operands (W and operand tiles)
constexpr int kZSlots = 4;       // ring slots of the TMEM probe tiles (TMEM holds no more)
// Each stage's two copies (W tile, operand tile) are one 2-lane bulk-copy
// instruction of one loader warp.  The copies of one warp complete one after
// another, but more loader warps measured no faster: the copies are not
// what bounds the launch.
constexpr int kMmaWarp = 1;
constexpr int kFetchWarp = 2;    // takes tasks and acquires their phase counters
constexpr int kRelWarp = 3;      // publishes finished tasks on the phase counters
constexpr int kZWarp0 = 4;       // Z generators: a multiple of 4 (TMEM lane quarters)
constexpr int kZWarps = 8;       // (probe, lane quarter)
constexpr int kEpiWarp0 = kZWarp0 + kZWarps;
constexpr int kEpiWarps = 8;     // (probe, lane quarter)
constexpr int kEpiProbeStep = kEpiWarps / 4;  // head: warp group eg runs probes eg, eg + 2, ...
constexpr int kThreads = (kEpiWarp0 + kEpiWarps) * 32;
static_assert(kZWarp0 % 4 == 0 && kEpiWarp0 % 4 == 0, "warp w reads TMEM lane quarter w % 4");
constexpr int kTaskSlots = 4;               // tasks a CTA's fetcher publishes ahead of the others
constexpr int kKt = 64;                     // K per stage (fp16 elements)
constexpr uint32_t kTileA = 128 * kKt * 2;  // one 128-row A tile per stage
constexpr uint32_t kSbo = kKt * 16;         // bytes between 8-row groups
constexpr uint32_t kLbo = 128;              // bytes between core matrices along K
constexpr uint32_t kAccCols = 128;          // one accumulator buffer: 2 Bp P <= 128 columns
constexpr uint32_t kZCol0 = 2 * kAccCols;   // probe tiles: slot q at kZCol0 + 64 q (+ 32 p)
constexpr uint32_t kTmemCols = 512;
static_assert(kZCol0 + kZSlots * 64 <= kTmemCols, "probe tiles fit tensor memory");

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

// Row blocks (units of Bp) of probe p inside an operand group tile and the
// accumulator columns (units of Bp) of its C and D parts; see the header.
__host__ __device__ __forceinline__ int row_mean(int p) { return p == 0 ? 1 : 4; }
__host__ __device__ __forceinline__ int row_dhat(int p) { return p == 0 ? 2 : 3; }
__host__ __device__ __forceinline__ int row_e2(int p) { return p == 0 ? 0 : 5; }
__host__ __device__ __forceinline__ int col_c(int p) { return row_mean(p) - 1; }
__host__ __device__ __forceinline__ int col_d(int p) { return row_dhat(p) - 1; }

// The unperturbed layout: accumulator column block j (and operand row block
// j + 1) holds sequences (4 grp + j) Bp .. + Bp - 1 of the expert's batch.
// "Probe" p of a group then stands for the two blocks col_c(p) (its + lane)
// and col_d(p) (its - lane), and its cell states sit where a probe's two
// signs sit in the perturbed layout.
__host__ __device__ __forceinline__ int inf_seq(const TcGeom& g, int grp, int blk, int b) {
  return (4 * grp + blk) * g.Bp + b;
}

// Probe slots of the cell-state buffer per expert.
__host__ __device__ __forceinline__ int cst_lanes(const TcGeom& g) {
  return g.inf ? 2 * g.G : g.n_pert;
}
template <bool INF>
__device__ __forceinline__ int cst_lanes_of(const TcGeom& g) {
  return INF ? 2 * g.G : g.n_pert;
}

// Shared-memory carve-up of one ring slot.
struct StageLayout {
  uint32_t a_off, b_off, bytes;
};

__host__ __device__ inline StageLayout stage_layout(const TcGeom& g) {
  StageLayout L;
  L.a_off = 0;
  L.b_off = kTileA;
  L.bytes = (L.b_off + g.tileB + 1023u) & ~1023u;
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

// 2^(15 - J): moves raw bits J and J + 16 to the sign bits 15 and 31 of a
// pair word.  Read from the constant bank, so the move is an integer
// multiply-add (the FMA pipe) instead of a shift and a logic op (both on the
// integer pipe, which the rest of the pair-word work already loads).
__constant__ uint32_t kPairShift[16] = {32768u, 16384u, 8192u, 4096u, 2048u, 1024u, 512u, 256u,
                                        128u,   64u,    32u,   16u,   8u,    4u,    2u,   1u};

// fp16 pair word J of a run: +-1 for dense probes; for sparse probes the
// magnitude is kept only where the activity bit (same position in `act`) is
// set, so inactive coordinates are +-0.
template <bool SPARSE, int J>
__device__ __forceinline__ uint32_t z_pair(uint32_t raw, uint32_t act) {
  // dense: the two sign bits isolated, moved into place, ORed with 1.0 | 1.0
  // (an addition: the moved bits and 0x3C003C00 do not overlap)
  if (!SPARSE) return (raw & (0x00010001u << J)) * kPairShift[J] + 0x3C003C00u;
  // activity bits at the sign positions (bits 15 and 31), each spread over
  // its 16-bit half by a byte permute that replicates the top bit of bytes 1
  // and 3: a mask of 1.0 magnitudes where the coordinate is active
  uint32_t m;
  asm("prmt.b32 %0, %1, %2, 0xBB99;" : "=r"(m) : "r"(act << (15 - J)), "r"(0u));
  return ((raw << (15 - J)) & 0x80008000u) | (m & 0x3C003C00u);
}

// The 16 fp16 pair words of one 32-parameter run: word J holds elements 2J
// (low half) and 2J + 1 (high half), i.e. one TMEM column of an A operand.
template <bool SPARSE>
__device__ __forceinline__ void z_run_pairs(uint32_t raw, uint32_t act, uint32_t* o) {
  o[0] = z_pair<SPARSE, 0>(raw, act);    o[1] = z_pair<SPARSE, 1>(raw, act);
  o[2] = z_pair<SPARSE, 2>(raw, act);    o[3] = z_pair<SPARSE, 3>(raw, act);
  o[4] = z_pair<SPARSE, 4>(raw, act);    o[5] = z_pair<SPARSE, 5>(raw, act);
  o[6] = z_pair<SPARSE, 6>(raw, act);    o[7] = z_pair<SPARSE, 7>(raw, act);
  o[8] = z_pair<SPARSE, 8>(raw, act);    o[9] = z_pair<SPARSE, 9>(raw, act);
  o[10] = z_pair<SPARSE, 10>(raw, act);  o[11] = z_pair<SPARSE, 11>(raw, act);
  o[12] = z_pair<SPARSE, 12>(raw, act);  o[13] = z_pair<SPARSE, 13>(raw, act);
  o[14] = z_pair<SPARSE, 14>(raw, act);  o[15] = z_pair<SPARSE, 15>(raw, act);
}

// 32 consecutive 32-bit columns of this thread's TMEM lane <- r[0..31].
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]),
      "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]),
      "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]),
      "r"(r[30]), "r"(r[31])
      : "memory");
}

// The MMAs of one stage, fully unrolled over K (NP = probes with a Z tile):
//   W (shared memory) x operand rows from w_row   -> d, N = 2 Bp P;
//   Z_0 (TMEM, zt)    x operand rows from 0       -> d, N = 2 Bp;
//   Z_1 (TMEM, zt+32) x operand rows from z1_row  -> d + dz1, N = 2 Bp.
// Descriptors arrive as their low words (start address in 16-byte units; a
// step along K is an addition), so the issuing thread spends a few
// instructions per MMA and keeps the tensor pipe fed.
template <int NP>
__device__ __forceinline__ void issue_stage(uint32_t d, uint32_t a_lo, uint32_t b_lo, uint32_t hi,
                                            uint32_t w_row, uint32_t z1_row, uint32_t zt,
                                            uint32_t idesc_w, uint32_t idesc_z, uint32_t dz1,
                                            uint32_t acc0) {
#pragma unroll
  for (int k16 = 0; k16 < kKt / 16; ++k16) {
    const uint32_t ko = (uint32_t)k16 * 16;  // 256 bytes: two core matrices along K
    const uint32_t acc = k16 > 0 ? 1u : acc0;
    mma_f16_ss_lohi(d, a_lo + ko, hi, b_lo + w_row + ko, hi, idesc_w, acc);
    if (NP >= 1) mma_f16_ts_lohi(d, zt + 8u * k16, b_lo + ko, hi, idesc_z, 1u);
    if (NP >= 2)
      mma_f16_ts_lohi(d + dz1, zt + 32u + 8u * k16, b_lo + z1_row + ko, hi, idesc_z, 1u);
  }
}

// ---------------------------------------------------------------------------
// Persistent warp-specialised kernel.  One launch runs every phase of a
// sweep (phase t: the head tasks of timestep t - 1 and the gate tasks of
// timestep t, see make_task); one CTA per SM takes tasks in global order
// (phase by phase, decode_task) from a counter in global memory, so the
// tasks whose inputs are ready first run first wherever an SM is free.  Its
// fetcher publishes each task to the CTA's other roles through a small ring
// of slots.  Phase counters in global memory replace a barrier between
// phases.  Roles:
//   warp 0        loader: lanes 0 and 1 bulk-copy the stage's A tile and
//                 operand group tile in one instruction;
//   warp 1        MMA issuer (the whole warp waits, one elected thread
//                 issues): W x operand (shared memory)
//                 and Z_p x operand (Z_p in tensor memory) per stage into one
//                 of two TMEM accumulator buffers;
//   warp 2        fetcher: takes the next task from the global counter,
//                 acquires its phase counters and publishes it;
//   warp 3        releaser: publishes finished tasks on the phase counters;
//   warps 4..11   Z generators: thread (probe, row) expands the raw probe
//                 words of the sweep's table into the fp16 +-1 row of its
//                 probe tile and stores it into the slot's TMEM columns
//                 (lane = row);
//   warps 12..19  epilogue: reads a finished accumulator buffer while the
//                 MMAs of the next task fill the other one; warp w reads the
//                 TMEM lanes of quarter w % 4 for probe group (w - 12) / 4.
// Barriers: full (the slot's copies landed and its Z tiles are stored: the
// loader's arrival with the copies' bytes and one arrival per Z warp, so the
// issuer waits once per stage), slot_free (the slot's MMAs are done), z_free
// (the MMAs reading a probe-tile slot are done: shared memory holds five
// stages, tensor memory four probe tiles), acc_full (a buffer's task is
// accumulated), acc_empty (its epilogue has read it), mma_done (all MMAs of
// the CTA completed), task_full / task_empty (the task ring).  Every wait is
// bounded (wait_or_abort, mbar_wait, wait_counter, wait_smem_count).
// ---------------------------------------------------------------------------
// One task: (expert, row tile, probe group).  For the gate the row tile is
// 32 hidden units (128 gate rows); for the head it is a 128-row vocabulary
// half.
struct Task {
  bool head;
  int e, m, grp, p_valid, nst;
  const uint8_t* a;  // A tile of stage 0
  const uint8_t* b;  // operand group tile of stage 0 (stages < Sx of a gate task: bx)
  const uint8_t* bx; // gate: the timestep's embedding-part tile of stage 0
};

struct Ctl {
  uint64_t full[kStages];
  uint64_t slot_free[kStages];
  uint64_t z_free[kZSlots];        // the MMAs reading a probe-tile slot are done
  uint64_t acc_full[2];
  uint64_t acc_empty[2];
  uint64_t red_bar;                // the head epilogue's rendezvous
  uint64_t mma_done;
  uint64_t task_full[kTaskSlots];  // the fetcher published the slot's task
  uint64_t task_empty[kTaskSlots]; // every other role has read it
  int task_gid[kTaskSlots];        // global task index, -1: no more tasks
  int task_t[kTaskSlots];          // its phase
  Task task[kTaskSlots];           // and the task, decoded once by the fetcher
  int epi_done;                    // epilogue warps' finished tasks (monotonic)
  uint32_t tmem_slot;
  volatile int abort;
};
static_assert(sizeof(Ctl) <= 1024, "the control block sits in the 1 KB before the head buffer");

// A wait that times out records SOMA_ERR_TIMEOUT in the status word and sets
// the CTA's abort flag; a wait that is still pending sees the flag within 64
// polls and returns false, so the CTA winds down without issuing further
// copies or MMAs.  A phase that is already complete costs one poll and no
// read of the flag.
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

// Ring position of the next stage: shared-memory slot q and the parity of
// its phase, probe-tile slot zq.
struct RingPos {
  uint32_t q, ph, zq;
  __device__ __forceinline__ void next() {
    if (++q == kStages) {
      q = 0;
      ph ^= 1u;
    }
    if (++zq == kZSlots) zq = 0;
  }
};

// The MMAs of one task, issued by one thread: per stage, wait for the
// copies and the probe tiles (one barrier), issue, and release the slot
// with a commit.
// The probe count NP is fixed per task, so the loop carries no dispatch.
template <int NP>
__device__ __forceinline__ bool mma_task(uint64_t* full, uint64_t* slot_free, uint64_t* z_free,
                                         RingPos& rp, int nst, uint32_t d, uint32_t tmem,
                                         uint32_t a_lo0, uint32_t b_lo0, uint32_t slot_step,
                                         uint32_t hi, uint32_t w_row, uint32_t z1_row,
                                         uint32_t idesc_w, uint32_t idesc_z, uint32_t dz1,
                                         volatile int* abort, int* status) {
  for (int st = 0; st < nst; ++st) {
    // the whole warp waits, so the descriptor words stay warp-uniform and
    // one elected thread issues
    const bool ready = wait_or_abort(&full[rp.q], rp.ph, abort, status);
    if (__any_sync(0xffffffffu, !ready)) return false;
    tc_fence_after();
    // the accumulator block, the probe tiles of the slot and the operand
    // windows (rows of 128 bytes per 8-row group step) stay inside their
    // allocations
    if (!SOMA_CHECK((d & 0xFFFFu) + dz1 + (NP >= 2 ? dz1 : 0) <= 2 * kAccCols &&
                        kZCol0 + 64u * rp.zq + 32u * (NP > 0 ? NP : 1) <= kTmemCols &&
                        rp.q < (uint32_t)kStages && rp.zq < (uint32_t)kZSlots,
                    status))
      return false;
    const uint32_t so = rp.q * slot_step;
    if (elect_one()) {
      issue_stage<NP>(d, a_lo0 + so, b_lo0 + so, hi, w_row, z1_row, tmem + kZCol0 + 64u * rp.zq,
                      idesc_w, idesc_z, dz1, st > 0 ? 1u : 0u);
      mma_commit(&slot_free[rp.q]);
      mma_commit(&z_free[rp.zq]);
    }
    __syncwarp();
    rp.next();
  }
  return true;
}

struct TcArgs {
  Sweep sw;
  TcGeom g;
  int gate_tasks, head_tasks;  // per phase
  const uint8_t* w16;    // [N][MT][S] A tiles
  const uint8_t* wo16;   // [N][2][Sh] A tiles
  uint8_t* op[2];        // [N][S][G] operand group tiles; phase t reads op[t % 2] = [x_t | h_{t-1}]
  int* prod;             // [N][G] writes finished into a group's operand (see the phase counters)
  int* hd;               // [N][G] head tasks finished reading a group's operand
  int* next_task;        // the next global task index to hand out
  int total_tasks;       // over all phases
  float* cst;            // [N*n][Hp][Bp] cell state (float2: sign +, -)
  float* pm;             // [N*n*2][B_mem][T][2] head max partials
  float* ps;             // sum-exp partials
  float* ply;            // [N*n*2][B_mem][T] target logits
  const uint2* zb;       // probe-word table (zbits_block), n_zrows rows, then activity words
  size_t n_zrows;
  int* status;
  // extents for the index checks of the checked build (bytes of w16, wo16,
  // each op buffer and the byte batch; floats of cst, pm / ps, ply, params;
  // bytes of the dynamic shared memory)
  const uint8_t* xall;   // [T][N][Sx][G] embedding-part tiles of every timestep
  uint2* xbits;          // [N][n][256][Ep / 32] probe words of the embedding rows
  uint2* zb_out;         // the probe-word table, written before the sweep (a.zb reads it)
  size_t n_w16, n_wo16, n_op, n_xall, n_xbits, n_bytes, n_cst, n_pm, n_ply, n_params;
  uint32_t smem_bytes;
};

// One phase t of the sweep: the gate tasks of timestep t (t < T) and the
// head tasks of timestep t - 1 (t >= 1), both reading the h part of op[t %
// 2]; the gate tasks write h_t into op[(t + 1) % 2].  The embedding part of
// every timestep's operand is written before the sweep (xall).
struct Phase {
  int t_gate, t_head;    // timesteps, -1: none
  int n_gate, n_head;
  const uint8_t* op_in;
  uint8_t* op_out;
};

__device__ __forceinline__ Phase make_phase(const TcArgs& a, int t) {
  Phase ph;
  const int T = a.sw.T;
  ph.t_gate = t < T ? t : -1;
  ph.t_head = t - 1;
  ph.n_gate = t < T ? a.gate_tasks : 0;
  ph.n_head = t >= 1 ? a.head_tasks : 0;
  ph.op_in = a.op[t & 1];
  ph.op_out = a.op[(t + 1) & 1];
  return ph;
}

// Global task index -> (phase, task of the phase): phase 0 has the gate
// tasks only, phases 1 .. T - 1 both kinds, phase T the head tasks only.
__device__ __forceinline__ void decode_task(const TcArgs& a, int gid, int& t, int& task) {
  const int both = a.gate_tasks + a.head_tasks;
  if (gid < a.gate_tasks) {
    t = 0;
    task = gid;
    return;
  }
  gid -= a.gate_tasks;
  const int mid = (a.sw.T - 1) * both;
  if (gid < mid) {
    t = 1 + gid / both;
    task = gid % both;
  } else {
    t = a.sw.T;
    task = gid - mid;
  }
}

// The consumer side of the task ring: waits for the next published task,
// copies it (phase t and the decoded task) and releases the slot (one
// arrival per warp) unless `release` is false.  Returns the global task
// index, -1 at the end, -2 after an abort.
__device__ __forceinline__ int next_task(Ctl* ctl, uint32_t& kt, volatile int* abort, int* status,
                                         int& t, Task& T, bool release = true) {
  const int sl = (int)(kt % kTaskSlots);
  if (!wait_or_abort(&ctl->task_full[sl], (kt / kTaskSlots) & 1u, abort, status)) return -2;
  const int gid = ctl->task_gid[sl];
  if (gid >= 0) {
    t = ctl->task_t[sl];
    T = ctl->task[sl];
  }
  __syncwarp(__activemask());
  if (release && (threadIdx.x & 31) == 0) mbar_arrive(&ctl->task_empty[sl]);
  ++kt;
  return gid;
}

// Waits (bounded) until the shared counter reaches `target`; an acquire at
// CTA scope, so the writes that the counting warps made before their
// release-add are visible to the caller afterwards.
__device__ __forceinline__ bool wait_smem_count(int* ctr, int target, volatile int* abort,
                                                int* status) {
  const uint32_t addr = smem_u32(ctr);
  for (uint32_t n = 0; n < (1u << 22); ++n) {
    int v;
    asm volatile("ld.acquire.cta.shared::cta.b32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    if (v >= target) return true;
    if ((n & 63u) == 63u && *abort) return false;
    __nanosleep(32);
  }
  *abort = 1;
  atomicCAS(status, 0, kStatusTimeout);
  return false;
}

// Phase counters.  A launch may run several phases; tasks of phase t + 1
// start on the groups that phase t has finished, without a grid-wide
// barrier.  Per (expert, group): prod counts the writes finished into the
// group's operand (one per epilogue warp of a gate task), hd the head tasks
// finished (one per epilogue warp).
// Through phase t (inclusive):
__device__ __forceinline__ int prod_target(const TcArgs& a, int t) {
  if (t < 0) return 0;
  const int gate_phases = min(t, a.sw.T - 1) + 1;
  return kEpiWarps * a.g.MT * gate_phases;
}
__device__ __forceinline__ int hd_target(const TcArgs& a, int t) {
  return t < 1 ? 0 : kEpiWarps * 2 * t;
}

// Waits (bounded) until *ctr >= target; lane 0 polls for the warp.  The
// acquire and the cross-proxy fence order the operand data written by other
// CTAs before this warp's later reads, bulk copies included.
__device__ __forceinline__ bool wait_counter(const int* ctr, int target, volatile int* abort,
                                             int* status) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) {
    uint32_t n = 0;
    for (;;) {
      int v;
      asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
      if (v >= target) break;
      if (++n >= (1u << 22) || ((n & 63u) == 0 && *abort)) {
        ok = 0;
        break;
      }
      __nanosleep(64);
    }
    if (!ok && n >= (1u << 22)) {
      *abort = 1;
      atomicCAS(status, 0, kStatusTimeout);
    }
  }
  ok = __shfl_sync(0xffffffffu, ok, 0);
  asm volatile("fence.proxy.async.global;" ::: "memory");
  return ok != 0;
}

// A phase's task list runs group by group ((expert, probe group), in
// order): the group's two head tasks, then its gate tasks (row tiles
// fastest).  The CTAs take tasks in global order (phase by phase, see
// decode_task), so the groups of a phase finish one after another and the
// next phase's tasks of a group become ready in the same order.
template <bool INF>
__device__ __forceinline__ Task make_task(const TcArgs& a, const Phase& ph, int task) {
  const TcGeom& g = a.g;
  Task T;
  const int hb = ph.n_head > 0 ? 2 : 0;
  const int per = hb + (ph.n_gate > 0 ? g.MT : 0);
  const int block = task / per, w = task % per;
  T.head = w < hb;
  T.m = T.head ? w : w - hb;
  T.grp = block % g.G;
  T.e = block / g.G;
  T.p_valid = INF ? g.P : min(g.P, a.sw.n_pert - T.grp * g.P);
  if (T.head) {
    T.nst = g.Sh;
    T.a = a.wo16 + (((size_t)T.e * 2 + T.m) * g.Sh) * kTileA;
    T.b = ph.op_in + (((size_t)T.e * g.S + g.Sx) * g.G + T.grp) * g.tileB;
  } else {
    T.nst = g.S;
    T.a = a.w16 + (((size_t)T.e * g.MT + T.m) * g.S) * kTileA;
    T.b = ph.op_in + (((size_t)T.e * g.S) * g.G + T.grp) * g.tileB;
  }
  T.bx = a.xall +
         ((((size_t)max(ph.t_gate, 0) * g.n_experts + T.e) * g.Sx) * g.G + T.grp) * g.tileB;
  return T;
}

// Flat parameter index of element (row r, k = 0) of the stage-st Z run.
__device__ __forceinline__ int64_t z_param(const TcArgs& a, const Task& T, int r, int st) {
  const Layout& L = a.sw.lay;
  if (T.head) return L.w_out + (int64_t)(128 * T.m + r) * a.g.H + (int64_t)kKt * st;
  const int64_t R = (int64_t)tile_gate(r) * a.g.H + 32 * T.m + tile_unit(r);  // W row of tile row r
  return st < a.g.Sx ? L.w_ih + R * a.g.E + (int64_t)kKt * st
                     : L.w_hh + R * a.g.H + (int64_t)kKt * (st - a.g.Sx);
}

// Probe-word table: for every (expert, probe, tile, stage) the raw words of
// the stage's 64 parameters of each of the 128 tile rows, one uint2 per row
// (runs 0 and 1 of the stage); the activity words of sparse probes follow in
// a second table of the same shape.  Tiles: the MT gate tiles of S stages,
// then the two head tiles of Sh stages.
constexpr int kZRows = 128;

__host__ __device__ __forceinline__ int zbits_stages(const TcGeom& g) {
  return g.MT * g.S + 2 * g.Sh;
}

__host__ __device__ __forceinline__ size_t zbits_row(const TcGeom& g, int e, int probe, bool head,
                                                     int m) {
  const int ts = head ? g.MT * g.S + m * g.Sh : m * g.S;
  return (((size_t)e * g.n_pert + probe) * zbits_stages(g) + ts) * kZRows;
}

// Gate epilogue of one task for one warp of TMEM lane quarter q4 (units
// 8 q4 .. 8 q4 + 7 of the tile).  With P = 2 the warps of group eg = 0, 1 run
// probe eg; with P = 1 both groups run probe 0 and split its 8-sequence
// chunks.  Thread l runs the cells of unit l / 4 for sequences b0 + l % 4 and
// b0 + 4 + l % 4 of each of its chunks, both signs, in fp32: 16x128b loads
// give it all four gates of its unit (gate-major rows), so no data moves
// between threads.  It writes the three operand rows of its (unit,
// sequence) for timestep t + 1: vbar, dhat and eps^2 dhat.  Cell state
// layout: [e, i][Hp][Bp] float2 (+, -).
//
// gate_prepare runs before the accumulator is ready: it loads the bias, its
// probe signs and the previous cell states, so that their latency overlaps
// the task's MMAs.
constexpr int kEpiMaxChunks = 4;  // Bp <= 32 with P = 2; Bp <= 64 split over two groups with P = 1

struct GatePre {
  float bias[4], dbias[4];
  float2 cprev[kEpiMaxChunks][2];
  int p, c0, cstep;
  bool on;
};

template <bool INF>
__device__ __forceinline__ void gate_prepare(const TcArgs& a, const Phase& ph, const Task& T,
                                             int q4, int eg, GatePre& G) {
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  const Layout& L = s.lay;
  const int lane = threadIdx.x & 31;
  const int H = g.H;
  G.p = g.P == 2 ? eg : 0;
  G.c0 = g.P == 2 ? 0 : eg;
  G.cstep = g.P == 2 ? 1 : 2;
  G.on = G.p < T.p_valid;
  if (!G.on) return;
  const int i = T.grp * g.P + G.p;
  const ProbeKey pk = make_probe_key(s.seed, s.step, (uint32_t)T.e, (uint32_t)i);
  const float eps = s.eps;
  const float* th = s.params + (int64_t)T.e * L.P;
  // bias and its probe sign for the row in this lane's TMEM lane, handed to
  // the threads that run that row's unit
  float bias_r = 0.f, dbias_r = 0.f;
  {
    const int Ur = 32 * T.m + tile_unit(32 * q4 + lane);
    const int64_t pb = L.b + (int64_t)tile_gate(32 * q4 + lane) * H + Ur;
    if (Ur < H && SOMA_CHECK((size_t)(T.e * L.P + pb) < a.n_params, a.status)) {
      bias_r = th[pb];
      if (eps != 0.f) {
        const ProbeBits zb = probe_bits(pk, pb, s.sparse);
        dbias_r = eps_z(zb.neg & 1u, zb.act & 1u, eps);
      }
    }
  }
  const int u8 = lane >> 2, bq = lane & 3;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    G.bias[k] = __shfl_sync(0xffffffffu, bias_r, 8 * k + u8);
    G.dbias[k] = __shfl_sync(0xffffffffu, dbias_r, 8 * k + u8);
  }
  const int U = 32 * T.m + 8 * q4 + u8;
  const float2* cell = reinterpret_cast<const float2*>(a.cst) +
                       (((int64_t)T.e * cst_lanes_of<INF>(g) + i) * g.Hp + U) * (int64_t)g.Bp;
  const bool load = U < H && ph.t_gate > 0;
#pragma unroll
  for (int j = 0; j < kEpiMaxChunks; ++j) {
    const int b0 = 8 * (G.c0 + j * G.cstep);
    G.cprev[j][0] = G.cprev[j][1] = make_float2(0.f, 0.f);
    if (load && b0 < g.Bp &&
        SOMA_CHECK((size_t)(cell - reinterpret_cast<const float2*>(a.cst) + b0 + 8) * 2 <= a.n_cst,
                   a.status)) {
      G.cprev[j][0] = cell[b0 + bq];
      G.cprev[j][1] = cell[b0 + 4 + bq];
    }
  }
}

template <bool INF>
__device__ void gate_finish(const TcArgs& a, const Phase& ph, const Task& T, uint32_t tacc,
                            int q4, const GatePre& G) {
  if (!G.on) return;
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  const int lane = threadIdx.x & 31;
  const int H = g.H;
  const float eps = s.eps;
  const float half_inv_eps = eps != 0.f ? 0.5f / eps : 0.f;
  const float half_eps = 0.5f * eps;
  const int p = G.p;
  const int u8 = lane >> 2, bq = lane & 3;
  const int U = 32 * T.m + 8 * q4 + u8;
  const bool unit_ok = U < H;
  // a stage of the next operand holds kKt / 32 of the 32-unit row tiles
  uint8_t* out_tile =
      ph.op_out + (((size_t)T.e * g.S + g.Sx + 32 * T.m / kKt) * g.G + T.grp) * g.tileB;
  const int kk = 32 * T.m % kKt + 8 * q4 + u8;
  const int i = T.grp * g.P + p;
  float2* cell = reinterpret_cast<float2*>(a.cst) +
                 (((int64_t)T.e * cst_lanes_of<INF>(g) + i) * g.Hp + U) * (int64_t)g.Bp;
  const uint32_t tq = tacc + ((uint32_t)(32 * q4) << 16);  // gates 0, 1
  const uint32_t tq2 = tq + (16u << 16);                    // gates 2, 3
  const uint32_t cC = (uint32_t)(col_c(p) * g.Bp), cD = (uint32_t)(col_d(p) * g.Bp);
  const int rM = row_mean(p) * g.Bp, rD = row_dhat(p) * g.Bp, rE = row_e2(p) * g.Bp;
#pragma unroll
  for (int j = 0; j < kEpiMaxChunks; ++j) {
    const int b0 = 8 * (G.c0 + j * G.cstep);
    if (b0 >= g.Bp) break;
    // [seq half][gate]: C (W vbar + eps^2 Z dhat) and D (W dhat + Z vbar)
    uint32_t vc[2][4], vd[2][4];
    if (!SOMA_CHECK(cC + b0 + 8 <= kAccCols && cD + b0 + 8 <= kAccCols, a.status)) break;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const uint32_t cw = (uint32_t)(b0 + 4 * h);
      tmem_ld_16x128b(tq + cC + cw, vc[h][0], vc[h][1]);
      tmem_ld_16x128b(tq2 + cC + cw, vc[h][2], vc[h][3]);
      tmem_ld_16x128b(tq + cD + cw, vd[h][0], vd[h][1]);
      tmem_ld_16x128b(tq2 + cD + cw, vd[h][2], vd[h][3]);
    }
    tmem_wait_ld();
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      float actp[4], actm[4];
      if constexpr (INF) {
        // unperturbed: the + and - lanes are two blocks' own pre-activations
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float ap = __uint_as_float(vc[h][k]) + G.bias[k];
          const float am = __uint_as_float(vd[h][k]) + G.bias[k];
          if (k == 2) {
            actp[k] = fmaf(sigm(2.f * ap), 2.f, -1.f);
            actm[k] = fmaf(sigm(2.f * am), 2.f, -1.f);
          } else {
            actp[k] = sigm(ap);
            actm[k] = sigm(am);
          }
        }
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float C = __uint_as_float(vc[h][k]) + G.bias[k];
          const float D = fmaf(eps, __uint_as_float(vd[h][k]), G.dbias[k]);
          if (k == 2) {  // g: tanh(x) = 2 sigmoid(2x) - 1
            actp[k] = fmaf(sigm(2.f * (C + D)), 2.f, -1.f);
            actm[k] = fmaf(sigm(2.f * (C - D)), 2.f, -1.f);
          } else {
            actp[k] = sigm(C + D);
            actm[k] = sigm(C - D);
          }
        }
      }
      const float cp = fmaf(actp[1], G.cprev[j][h].x, actp[0] * actp[2]);
      const float cm = fmaf(actm[1], G.cprev[j][h].y, actm[0] * actm[2]);
      const float hp = actp[3] * fmaf(sigm(2.f * cp), 2.f, -1.f);
      const float hm = actm[3] * fmaf(sigm(2.f * cm), 2.f, -1.f);
      const int b = b0 + 4 * h + bq;
      const size_t tile_off = (size_t)(out_tile - ph.op_out);
      if (unit_ok &&
          SOMA_CHECK((size_t)(cell - reinterpret_cast<float2*>(a.cst) + b + 1) * 2 <= a.n_cst &&
                         tile_off + g.tileB <= a.n_op && rE + b < g.rowsB && rD + b < g.rowsB &&
                         rM + b < g.rowsB && kk < kKt,
                     a.status)) {
        cell[b] = make_float2(cp, cm);
        if constexpr (INF) {
          // h of the two blocks into their own rows (the W product's rows)
          if (inf_seq(g, T.grp, col_c(p), b) < s.B)
            *reinterpret_cast<__half*>(out_tile + kmajor_offset(rM + b, kk, kKt)) =
                __float2half_rn(hp);
          if (inf_seq(g, T.grp, col_d(p), b) < s.B)
            *reinterpret_cast<__half*>(out_tile + kmajor_offset(rD + b, kk, kKt)) =
                __float2half_rn(hm);
        } else if (b < s.B) {
          const float dh = hp - hm;
          *reinterpret_cast<__half*>(out_tile + kmajor_offset(rM + b, kk, kKt)) =
              __float2half_rn(0.5f * (hp + hm));
          *reinterpret_cast<__half*>(out_tile + kmajor_offset(rD + b, kk, kKt)) =
              __float2half_rn(dh * half_inv_eps);
          *reinterpret_cast<__half*>(out_tile + kmajor_offset(rE + b, kk, kKt)) =
              __float2half_rn(dh * half_eps);
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
// Rendezvous of the epilogue warps around the head's reduction buffer: a
// bounded wait on an mbarrier (count: one arrival per epilogue warp), so a
// warp that has left after an abort makes the others time out instead of
// blocking.  *use counts this warp's rendezvous so far.
__device__ __forceinline__ bool epi_rendezvous(uint64_t* bar, uint32_t* use, volatile int* abort,
                                               int* status) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
  const bool ok = wait_or_abort(bar, *use & 1u, abort, status);
  ++*use;
  __syncwarp();
  return ok;
}

template <bool INF>
__device__ bool head_epilogue(const TcArgs& a, const Phase& ph, const Task& T, uint32_t tacc,
                              int q4, int ew, float2* red, uint64_t* red_bar, uint32_t* red_use,
                              volatile int* abort) {
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  const Layout& L = s.lay;
  const int lane = threadIdx.x & 31;
  const float eps = s.eps;
  const bool do_z = eps != 0.f;
  const float* th = s.params + (int64_t)T.e * L.P;
  const int vq = 128 * T.m + 32 * q4;  // first vocabulary row of the quarter
  const float bo_r =
      SOMA_CHECK((size_t)(T.e * L.P + L.b_out + vq + lane) < a.n_params, a.status)
          ? th[L.b_out + vq + lane]
          : 0.f;
  const int t = ph.t_head;
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
    // perturbed: lanes (e, i, +) and (e, i, -) for sequence b; unperturbed:
    // lane (e, 0, +) for the sequences of blocks col_c(p) and col_d(p)
    const int64_t lane_plus = INF ? (int64_t)T.e * 2 : ((int64_t)T.e * s.n_pert + i) * 2;
    const uint32_t cC = (uint32_t)(col_c(p) * g.Bp), cD = (uint32_t)(col_d(p) * g.Bp);
    for (int b0 = 0; b0 < g.Bp; b0 += 4) {
      // [k]: C and D of row r4 + 8 k, sequence b0 + bq
      uint32_t vc[4], vd[4];
      const uint32_t cw = (uint32_t)b0;
      tmem_ld_16x128b(tq + cC + cw, vc[0], vc[1]);
      tmem_ld_16x128b(tq2 + cC + cw, vc[2], vc[3]);
      tmem_ld_16x128b(tq + cD + cw, vd[0], vd[1]);
      tmem_ld_16x128b(tq2 + cD + cw, vd[2], vd[3]);
      tmem_wait_ld();
      float lp[4], lm[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        if constexpr (INF) {
          lp[k] = __uint_as_float(vc[k]) + bo[k];
          lm[k] = __uint_as_float(vd[k]) + bo[k];
        } else {
          const float C = __uint_as_float(vc[k]) + bo[k];
          const float D = fmaf(eps, __uint_as_float(vd[k]), dbo[k]);
          lp[k] = C + D;
          lm[k] = C - D;
        }
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
      if (r4 == 0 && SOMA_CHECK(((p * g.Bp + b) * 2 + 1) * 4 + q4 < g.P * g.Bp * 8, a.status)) {
        red[((p * g.Bp + b) * 2 + 0) * 4 + q4] = make_float2(mp, sp);
        red[((p * g.Bp + b) * 2 + 1) * 4 + q4] = make_float2(mm, sm_);
      }
      if constexpr (INF) {
        // the target logit of each block's sequence, into lane (e, 0, +)
#pragma unroll
        for (int sg = 0; sg < 2; ++sg) {
          const int q = inf_seq(g, T.grp, sg ? col_d(p) : col_c(p), b);
          if (q >= s.B ||
              !SOMA_CHECK((size_t)(seq_offset(s, T.e, 0, q) + t + 1) < a.n_bytes &&
                              (size_t)((lane_plus * s.B_mem + s.b0 + q) * (int64_t)s.T + t) <
                                  a.n_ply,
                          a.status))
            continue;
          const int y = s.bytes[seq_offset(s, T.e, 0, q) + t + 1] - vq - r4;
          if (y >= 0 && y < 32 && (y & 7) == 0) {
            const int k = y >> 3;
            const float* l = sg ? lm : lp;
            a.ply[(lane_plus * s.B_mem + s.b0 + q) * (int64_t)s.T + t] =
                k == 0 ? l[0] : k == 1 ? l[1] : k == 2 ? l[2] : l[3];
          }
        }
      } else if (b < s.B &&
                 SOMA_CHECK((size_t)(seq_offset(s, T.e, i, b) + t + 1) < a.n_bytes &&
                                (size_t)(((lane_plus + 1) * s.B_mem + s.b0 + b) * (int64_t)s.T +
                                         t) < a.n_ply,
                            a.status)) {
        const int y = s.bytes[seq_offset(s, T.e, i, b) + t + 1] - vq - r4;
        // y = 8 k for the thread that holds the target row
        if (y >= 0 && y < 32 && (y & 7) == 0) {
          const int k = y >> 3;
          const float vp = k == 0 ? lp[0] : k == 1 ? lp[1] : k == 2 ? lp[2] : lp[3];
          const float vm = k == 0 ? lm[0] : k == 1 ? lm[1] : k == 2 ? lm[2] : lm[3];
          a.ply[((lane_plus + 0) * s.B_mem + s.b0 + b) * (int64_t)s.T + t] = vp;
          a.ply[((lane_plus + 1) * s.B_mem + s.b0 + b) * (int64_t)s.T + t] = vm;
        }
      }
    }
  }
  // all epilogue warps: partials of this task are in `red`
  if (!epi_rendezvous(red_bar, red_use, abort, a.status)) return false;
  const int et = threadIdx.x - kEpiWarp0 * 32;
  const int n_red = T.p_valid * g.Bp * 2;
  for (int idx = et; idx < n_red; idx += kEpiWarps * 32) {
    const int sgn = idx & 1;
    const int pb = idx >> 1;
    const int pp = pb / g.Bp, b = pb % g.Bp;
    // the partials' lane and sequence (see the target logits above)
    const int qs = INF ? inf_seq(g, T.grp, sgn ? col_d(pp) : col_c(pp), b) : b;
    if (qs >= s.B) continue;
    const float2* q = red + (size_t)idx * 4;
    const float M = fmaxf(fmaxf(q[0].x, q[1].x), fmaxf(q[2].x, q[3].x));
    float S = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) S += q[k].y * __expf(q[k].x - M);
    const int i = T.grp * g.P + pp;
    const int64_t ln = INF ? (int64_t)T.e * 2 : ((int64_t)T.e * s.n_pert + i) * 2 + sgn;
    const int64_t o = ((ln * s.B_mem + s.b0 + qs) * (int64_t)s.T + t) * 2 + T.m;
    if (!SOMA_CHECK((size_t)o < a.n_pm, a.status)) continue;
    a.pm[o] = M;
    a.ps[o] = S;
  }
  // `red` is reused by the next task
  return epi_rendezvous(red_bar, red_use, abort, a.status);
}

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// grid: one persistent CTA per SM at most (all resident: the launch is
// cooperative), kThreads threads.  The CTAs share the tasks of phases
// 0 .. T through the task counter.
// SPARSE: sparse probes; INF: the unperturbed layout (eps = 0, one sign).
template <bool SPARSE, bool INF>
__global__ void __launch_bounds__(kThreads, 1) tc_persistent_kernel(const TcArgs a) {
  extern __shared__ uint8_t dyn_smem[];
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  uint8_t* smem = align1024(dyn_smem);
  const StageLayout SL = stage_layout(g);
  Ctl* ctl = reinterpret_cast<Ctl*>(smem + kStages * SL.bytes);
  float2* red = reinterpret_cast<float2*>(smem + kStages * SL.bytes + 1024);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool do_z = s.eps != 0.f;
  int* status = a.status;
  volatile int* abort = &ctl->abort;

  if (tid == 0) {
    ctl->abort = 0;
    for (int q = 0; q < kStages; ++q) {
      // the loader's arrival with the copies' bytes and, when probes are
      // generated, one arrival per Z warp
      mbar_init(&ctl->full[q], do_z ? 1 + kZWarps : 1);
      mbar_init(&ctl->slot_free[q], 1);
    }
    for (int q = 0; q < kZSlots; ++q) mbar_init(&ctl->z_free[q], 1);
    for (int q = 0; q < 2; ++q) {
      mbar_init(&ctl->acc_full[q], 1);
      mbar_init(&ctl->acc_empty[q], kEpiWarps);
    }
    mbar_init(&ctl->red_bar, kEpiWarps);
    mbar_init(&ctl->mma_done, 1);
    for (int q = 0; q < kTaskSlots; ++q) {
      mbar_init(&ctl->task_full[q], 1);
      // the loader, the MMA issuer, the Z warps (when probes are
      // generated), the epilogue warps and the releaser read every task
      mbar_init(&ctl->task_empty[q], 3 + (do_z ? kZWarps : 0) + kEpiWarps);
    }
    ctl->epi_done = 0;
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(&ctl->tmem_slot, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctl->tmem_slot;

  if (warp == kFetchWarp) {
    // --------------------------------------------------------------- fetcher
    // Takes the tasks in global order, decodes each, acquires the group's
    // phase counters of phase t - 1 and only then publishes the task to the
    // CTA's other roles, up to kTaskSlots tasks ahead of the slowest of them:
    // the counters' round trips stay off the loader's path.  Copies read
    // what phase t - 1 wrote into the group's operand; a gate task's
    // epilogue also overwrites what phase t - 1 read.
    uint32_t kt = 0;
    for (;;) {
      const int sl = (int)(kt % kTaskSlots);
      if (kt >= kTaskSlots &&
          !wait_or_abort(&ctl->task_empty[sl], ((kt / kTaskSlots) - 1) & 1u, abort, status))
        break;
      int gid = 0;
      if (lane == 0) gid = atomicAdd(a.next_task, 1);
      gid = __shfl_sync(0xffffffffu, gid, 0);
      const bool end = gid >= a.total_tasks;
      int t = 0, task = 0;
      if (!end) decode_task(a, gid, t, task);
      const Phase ph = make_phase(a, t);
      const Task T = make_task<INF>(a, ph, task);
      if (!end && t >= 1) {
        const size_t c = (size_t)T.e * g.G + T.grp;
        if (!SOMA_CHECK(c < (size_t)g.n_experts * g.G, status) ||
            !wait_counter(a.prod + c, prod_target(a, t - 1), abort, status) ||
            (!T.head && !wait_counter(a.hd + c, hd_target(a, t - 1), abort, status)))
          break;
      }
      // the arrival passes the acquire of the counters on (CTA scope)
      if (lane == 0) {
        ctl->task_gid[sl] = end ? -1 : gid;
        ctl->task_t[sl] = t;
        ctl->task[sl] = T;
        mbar_arrive(&ctl->task_full[sl]);
      }
      ++kt;
      if (end) break;
    }
  } else if (warp == 0) {
    // ---------------------------------------------------------------- loader
    // the whole warp walks the stages in order and waits for their slots;
    // lanes 0 and 1 issue the stage's two copies together.
    uint32_t gs = 0, kt = 0;
    bool done = true;
    for (;;) {
      int t;
      Task T;
      const int gid = next_task(ctl, kt, abort, status, t, T);
      if (gid < 0) {
        done = gid == -1;
        break;
      }
      const Phase ph = make_phase(a, t);
      // the operand rows other CTAs wrote (generic proxy) before the
      // fetcher's acquire are read here by bulk copies (async proxy)
      asm volatile("fence.proxy.async.global;" ::: "memory");
      {
        for (int st = 0; st < T.nst; ++st, ++gs) {
          const int q = gs % kStages;
          const uint32_t use = gs / kStages;
          if (gs >= kStages &&
              !wait_or_abort(&ctl->slot_free[q], (use - 1) & 1u, abort, status)) {
            done = false;
            break;
          }
          uint8_t* slot = smem + q * SL.bytes;
          if (lane == 0) mbar_arrive_expect_tx(&ctl->full[q], kTileA + g.tileB);
          __syncwarp();
          if (lane < 2) {
            uint8_t* dst = lane == 0 ? slot + SL.a_off : slot + SL.b_off;
            const bool xs = !T.head && st < g.Sx;  // an embedding-part stage
            const uint8_t* src = lane == 0 ? T.a + (size_t)st * kTileA
                                           : (xs ? T.bx : T.b) + (size_t)st * g.G * g.tileB;
            const uint32_t nb = lane == 0 ? kTileA : g.tileB;
            const uint8_t* gbase =
                lane == 1 ? (xs ? a.xall : ph.op_in) : (T.head ? a.wo16 : a.w16);
            const size_t gsize =
                lane == 1 ? (xs ? a.n_xall : a.n_op) : (T.head ? a.n_wo16 : a.n_w16);
            if (SOMA_CHECK((size_t)(dst - dyn_smem) + nb <= a.smem_bytes &&
                               src >= gbase && (size_t)(src - gbase) + nb <= gsize,
                           status))
              bulk_g2s(dst, src, nb, &ctl->full[q]);
          }
          __syncwarp();
        }
        if (!done) break;
      }
    }
    // The copies of the last stage of each slot land before the CTA exits
    // (earlier phases of a slot completed before its later copies were
    // issued).  After an abort the copies issued so far are not tracked: the
    // slot waits that failed above were bounded, and copies take
    // microseconds against that bound.
    if (done) {
#pragma unroll
      for (int q = 0; q < kStages; ++q) {
        if ((int)gs <= q) continue;
        const uint32_t last = gs - 1 - ((gs - 1 - (uint32_t)q) % kStages);  // last stage of slot q
        mbar_wait(&ctl->full[q], (last / kStages) & 1u);
      }
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    // The whole warp walks the tasks and stages; one elected thread issues.
    {
      const uint32_t idesc_z = idesc_f16_f32(128, 2 * g.Bp);
      // W covers the P probes of the group (2 Bp P columns); a group with
      // one valid probe still multiplies the whole window (the rows of the
      // missing probe are zero)
      const uint32_t idesc_w = idesc_f16_f32(128, 2 * g.Bp * g.P);
      // descriptors of slot 0; slot q is q * SL.bytes further
      const uint64_t d0 = smem_desc(smem_u32(smem), kLbo, kSbo);
      const uint32_t hi = (uint32_t)(d0 >> 32);
      const uint32_t lo0 = (uint32_t)d0;
      const uint32_t slot_step = SL.bytes >> 4;
      const uint32_t a_lo0 = lo0 + (SL.a_off >> 4), b_lo0 = lo0 + (SL.b_off >> 4);
      const uint32_t grp_step = kSbo >> 4;                     // 8 operand rows
      const uint32_t w_row = (uint32_t)(g.Bp / 8) * grp_step;  // the W window starts at row Bp
      const uint32_t z1_row = (uint32_t)(4 * g.Bp / 8) * grp_step;
      const uint32_t dz1 = (uint32_t)(2 * g.Bp);
      RingPos rp = {0u, 0u, 0u};
      uint32_t kt = 0;
      for (int k = 0;; ++k) {
        int t;
        Task T;
        if (next_task(ctl, kt, abort, status, t, T) < 0) break;
        const int buf = k & 1;
        if (k >= 2 &&
            __any_sync(0xffffffffu, !wait_or_abort(&ctl->acc_empty[buf],
                                                   (uint32_t)((k >> 1) - 1) & 1u, abort, status)))
          break;
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)buf * kAccCols;
        const int np = do_z ? T.p_valid : 0;
        bool ok;
        if (np == 2)
          ok = mma_task<2>(ctl->full, ctl->slot_free, ctl->z_free, rp, T.nst, d, tmem, a_lo0, b_lo0,
                           slot_step, hi, w_row, z1_row, idesc_w, idesc_z, dz1, abort, status);
        else if (np == 1)
          ok = mma_task<1>(ctl->full, ctl->slot_free, ctl->z_free, rp, T.nst, d, tmem, a_lo0, b_lo0,
                           slot_step, hi, w_row, z1_row, idesc_w, idesc_z, dz1, abort, status);
        else
          ok = mma_task<0>(ctl->full, ctl->slot_free, ctl->z_free, rp, T.nst, d, tmem, a_lo0, b_lo0,
                           slot_step, hi, w_row, z1_row, idesc_w, idesc_z, dz1, abort, status);
        if (!ok) break;
        if (elect_one()) mma_commit(&ctl->acc_full[buf]);
        __syncwarp();
      }
      // every MMA of this CTA completes before its tensor memory is freed
      if (elect_one()) mma_commit(&ctl->mma_done);
      __syncwarp();
      mbar_wait(&ctl->mma_done, 0);
    }
    __syncwarp();
  } else if (warp == kRelWarp) {
    // --------------------------------------------------------------- releaser
    // Publishes each task's operand writes (gate) or finished reads (head)
    // on the group's phase counter once the CTA's epilogue warps are done
    // with it: one gpu-scope fence and one add per task, off the epilogue
    // warps' path.  The epilogue warps count their finished tasks in shared
    // memory with a CTA-scope release; this warp's acquire of that count,
    // then its fence, order their writes before the add.
    uint32_t kt = 0;
    for (int k = 0;; ++k) {
      int t;
      Task T;
      if (next_task(ctl, kt, abort, status, t, T) < 0) break;
      const size_t c = (size_t)T.e * g.G + T.grp;
      if (!SOMA_CHECK(c < (size_t)g.n_experts * g.G, status) ||
          !wait_smem_count(&ctl->epi_done, kEpiWarps * (k + 1), abort, status))
        break;
      if (lane == 0) {
        __threadfence();
        atomicAdd(T.head ? a.hd + c : a.prod + c, kEpiWarps);
      }
      __syncwarp();
    }
  } else if (warp >= kZWarp0 && warp < kEpiWarp0) {
    // --------------------------------------------------------- Z generators
    // Thread (probe gtid / 128, row gtid % 128 = TMEM lane).  The raw probe
    // words of a stage come from the table zbits_block wrote before the
    // sweep, loaded two stages ahead.  A stage's fp16 row is expanded while
    // the previous stage's slot is still busy; once its slot is free it is
    // stored, and the next stage is expanded while that store completes.
    if (do_z) {
      const int gtid = tid - kZWarp0 * 32;
      const int r = gtid & 127, pz = gtid >> 7;
      const uint32_t trow = tmem + ((uint32_t)(32 * (warp & 3)) << 16) + kZCol0 + 32u * pz;
      uint32_t gs = 0, kt = 0;
      bool alive = true;
      while (alive) {
        int t;
        Task T;
        if (next_task(ctl, kt, abort, status, t, T) < 0) break;
        {
          // The next task's probe words come from DRAM (the table streams
          // through L2 once per phase): when it is already published, its
          // rows are prefetched into L2 now, a task ahead of their loads.
          {
            const int sn = (int)(kt % kTaskSlots);
            if (mbar_test_wait(&ctl->task_full[sn], (kt / kTaskSlots) & 1u) &&
                ctl->task_gid[sn] >= 0) {
              const Task& Tn = ctl->task[sn];
              const size_t rn = zbits_row(g, Tn.e, Tn.grp * g.P + pz, Tn.head, Tn.m) + (size_t)r;
              if (pz < Tn.p_valid && rn + (size_t)kZRows * (Tn.nst - 1) < a.n_zrows) {
                for (int st = 0; st < Tn.nst; ++st) {
                  prefetch_l2(a.zb + rn + (size_t)kZRows * st);
                  if (SPARSE) prefetch_l2(a.zb + a.n_zrows + rn + (size_t)kZRows * st);
                }
              }
            }
          }
          const size_t row0 = zbits_row(g, T.e, T.grp * g.P + pz, T.head, T.m) + (size_t)r;
          // uniform over the warp
          const bool active =
              pz < T.p_valid &&
              SOMA_CHECK(row0 + (size_t)kZRows * (T.nst - 1) < a.n_zrows, status);
          const uint2* zn = a.zb + row0;
          const uint2* za = a.zb + a.n_zrows + row0;
          const uint2 none = make_uint2(0u, 0u);
          // raw words (and activity words) of stages st + 1 and st + 2
          uint2 n1 = none, n2 = none, a1 = none, a2 = none;
          uint32_t zw[kKt / 2];
          if (active) {
            const uint2 n0 = __ldg(zn);
            const uint2 a0 = SPARSE ? __ldg(za) : none;
            if (T.nst > 1) {
              n1 = __ldg(zn + kZRows);
              if (SPARSE) a1 = __ldg(za + kZRows);
            }
            if (T.nst > 2) {
              n2 = __ldg(zn + 2 * kZRows);
              if (SPARSE) a2 = __ldg(za + 2 * kZRows);
            }
            z_run_pairs<SPARSE>(n0.x, a0.x, zw);
            z_run_pairs<SPARSE>(n0.y, a0.y, zw + 16);
          }
          for (int st = 0; st < T.nst; ++st, ++gs) {
            // the stage's shared-memory slot q (its full barrier) and
            // probe-tile slot zq
            const int q = gs % kStages;
            const int zq = gs % kZSlots;
            const uint32_t zuse = gs / kZSlots;
            // after an abort the generators stop: an arrival on a phase that
            // can no longer complete would overfill it
            if (gs >= kZSlots &&
                !wait_or_abort(&ctl->z_free[zq], (zuse - 1) & 1u, abort, status)) {
              alive = false;
              break;
            }
            tc_fence_after();
            if (active &&
                SOMA_CHECK(kZCol0 + 64u * (uint32_t)zq + 32u * pz + 32u <= kTmemCols, status)) {
              tmem_st32(trow + 64u * (uint32_t)zq, zw);
              if (st + 1 < T.nst) {
                z_run_pairs<SPARSE>(n1.x, a1.x, zw);
                z_run_pairs<SPARSE>(n1.y, a1.y, zw + 16);
                n1 = n2;
                a1 = a2;
                if (st + 3 < T.nst) {
                  n2 = __ldg(zn + (size_t)kZRows * (st + 3));
                  if (SPARSE) a2 = __ldg(za + (size_t)kZRows * (st + 3));
                }
              }
              tmem_wait_st();
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&ctl->full[q]);
          }
        }
      }
    }
  } else if (warp >= kEpiWarp0) {
    // --------------------------------------------------------------- epilogue
    // A gate task of phase t overwrites what phase t - 1 read (op[(t + 1) %
    // 2]) and reads the cell states that phase t - 1 wrote, possibly in
    // another CTA: the fetcher published the task only after acquiring the
    // group's counters of phase t - 1.  After each task it
    // counts itself done in shared memory, and the releaser publishes the
    // task on the group's counter.
    const int ew = warp - kEpiWarp0;
    const int q4 = warp & 3;
    int k = 0;
    uint32_t red_use = 0;
    bool alive = true;
    uint32_t kt = 0;
    for (; alive; ++k) {
      int t;
      Task T;
      if (next_task(ctl, kt, abort, status, t, T) < 0) break;
      const Phase ph = make_phase(a, t);
      {
        const int buf = k & 1;
        const size_t c = (size_t)T.e * g.G + T.grp;
        GatePre G;
        if (!SOMA_CHECK(c < (size_t)g.n_experts * g.G, status) ||
            !wait_or_abort(&ctl->acc_full[buf], (uint32_t)(k >> 1) & 1u, abort, status)) {
          alive = false;
          break;
        }
        if (!T.head) gate_prepare<INF>(a, ph, T, q4, ew >> 2, G);
        tc_fence_after();
        const uint32_t tacc = tmem + (uint32_t)buf * kAccCols;
        if (T.head) {
          if (!head_epilogue<INF>(a, ph, T, tacc, q4, ew, red, &ctl->red_bar, &red_use, abort)) {
            alive = false;
            break;
          }
        } else {
          gate_finish<INF>(a, ph, T, tacc, q4, G);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          asm volatile("red.release.cta.shared::cta.add.s32 [%0], 1;" ::"r"(smem_u32(&ctl->epi_done))
                       : "memory");
          mbar_arrive(&ctl->acc_empty[buf]);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, kTmemCols);
}

// Embedding part of the operand of timestep t: per probe p of the group the
// rows vbar = Emb[byte_t], dhat = z_emb[byte_t] (+-1, or 0) and eps^2 dhat.
// Block `blk` of Sx * G * N writes one (expert, stage, group) tile of xall.
template <bool INF>
__device__ void xpart_block(const TcArgs& a, uint8_t* xall, int t, int blk, int first,
                            int stride) {
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  const int st = (blk / g.G) % g.Sx, grp = blk % g.G;
  const int e = blk / (g.G * g.Sx);
  const Layout& L = s.lay;
  const float* th = s.params + (int64_t)e * L.P;
  const float eps2 = s.eps * s.eps;
  uint8_t* tile = xall + ((size_t)t * g.n_experts * g.Sx * g.G + blk) * g.tileB;
  const int chunks = g.rowsB * (kKt / 8);
  static_assert(kKt / 8 == 8, "a core-matrix column is 8 chunks");
  for (int c = first; c < chunks; c += stride) {
    // eight consecutive chunks fill the eight rows of one core matrix (128
    // contiguous bytes of the tile); rowsB is a multiple of 8
    const int row = 8 * (c / 64) + (c & 7), kc = (c >> 3) & 7;
    const int blkr = row / g.Bp, b = row % g.Bp;  // row block 0..3P-1, sequence
    const int p = blkr < 3 ? 0 : 1;
    const bool mean = blkr == row_mean(p), e2 = blkr == row_e2(p);
    const int i = grp * g.P + p;
    __align__(16) __half v[8];
    const int k0 = kKt * st + 8 * kc;
    if constexpr (INF) {
      // row blocks 1..4: the embeddings of four blocks of sequences; 0, 5: zero
      const int q = blkr >= 1 && blkr <= 4 ? inf_seq(g, grp, blkr - 1, b) : s.B;
      float x[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      if (q < s.B && SOMA_CHECK((size_t)seq_offset(s, e, 0, q) + t < a.n_bytes, a.status)) {
        const int y = s.bytes[seq_offset(s, e, 0, q) + t];
        const int64_t p0 = L.emb + (int64_t)y * g.E + k0;
        if (SOMA_CHECK(k0 >= g.E || (size_t)(e * L.P + p0 + min(8, g.E - k0)) <= a.n_params,
                       a.status)) {
#pragma unroll
          for (int j = 0; j < 8; ++j)
            if (k0 + j < g.E) x[j] = th[p0 + j];
        }
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) v[j] = __float2half_rn(x[j]);
    } else if (i < s.n_pert && b < s.B &&
        SOMA_CHECK((size_t)seq_offset(s, e, i, b) + t < a.n_bytes, a.status)) {
      const int y = s.bytes[seq_offset(s, e, i, b) + t];
      const int64_t p0 = L.emb + (int64_t)y * g.E + k0;
      if (!SOMA_CHECK(k0 >= g.E || (size_t)(e * L.P + p0 + min(8, g.E - k0)) <= a.n_params,
                      a.status))
        continue;
      ProbeBits bits = {0u, 0u};
      if (!mean && s.eps != 0.f) {
        // the row's probe words, from the table emb_bits_block wrote
        const size_t wi = (((size_t)e * s.n_pert + i) * 256 + y) * (g.Ep / 32) + k0 / 32;
        if (SOMA_CHECK(wi < a.n_xbits, a.status)) {
          const uint2 w = a.xbits[wi];
          bits.neg = w.x >> (k0 & 31);
          bits.act = w.y >> (k0 & 31);
        }
      }
      const float mag = e2 ? eps2 : 1.f;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        float x = 0.f;
        if (k0 + j < g.E)
          x = mean ? th[p0 + j] : eps_z((bits.neg >> j) & 1u, (bits.act >> j) & 1u, mag);
        v[j] = __float2half_rn(x);
      }
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) v[j] = __float2half_rn(0.f);
    }
    if (SOMA_CHECK((size_t)(tile - xall) + kmajor_offset(row, 8 * kc, kKt) + 16 <= a.n_xall,
                   a.status))
      *reinterpret_cast<uint4*>(tile + kmajor_offset(row, 8 * kc, kKt)) =
          *reinterpret_cast<const uint4*>(v);
  }
}

// The probe words of the embedding rows, once per sweep: (expert e, probe
// i), byte value y, words w of row y (parameters Emb[y][32 w .. 32 w + 31], natural
// order; bits past E belong to the next row and are never used).
// Block b of 2 N n (128 threads): (e, i) = b / 2, byte values y of half b % 2.
__device__ void emb_bits_block(const TcArgs& a, int b) {
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  const int pr = b >> 1;
  const int e = pr / s.n_pert, i = pr % s.n_pert, y = 128 * (b & 1) + (int)threadIdx.x;
  const ProbeKey k = make_probe_key(s.seed, s.step, (uint32_t)e, (uint32_t)i);
  const int words = g.Ep / 32;
  for (int w = 0; w < words; ++w) {
    const size_t wi = (((size_t)e * s.n_pert + i) * 256 + y) * words + w;
    const ProbeBits b = probe_bits(k, s.lay.emb + (int64_t)y * g.E + 32 * w, s.sparse);
    if (SOMA_CHECK(wi < a.n_xbits, a.status)) a.xbits[wi] = make_uint2(b.neg, b.act);
  }
}

// Block b: tile b % (N * Sx * G) of timestep b / (N * Sx * G).
template <bool INF>
__global__ void xpart_kernel(const TcArgs a, uint8_t* xall, int tiles) {
  xpart_block<INF>(a, xall, (int)(blockIdx.x / tiles), (int)(blockIdx.x % tiles), threadIdx.x,
                   blockDim.x);
}

// The probe-word table of one sweep (zbits_row): block b writes the 128 rows
// of (expert, probe, tile stage) b, thread r the raw words of the stage's
// 64 parameters of tile row r (and their activity words for sparse probes).
// Blocks of 128 threads.
template <bool SPARSE>
__device__ void zbits_block(const TcArgs& a, uint2* __restrict__ out, size_t b) {
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  const int TS = zbits_stages(g);
  const int ts = (int)(b % TS), i = (int)((b / TS) % g.n_pert), e = (int)(b / TS / g.n_pert);
  const int r = threadIdx.x;
  Task T;
  T.head = ts >= g.MT * g.S;
  T.e = e;
  const int tj = T.head ? ts - g.MT * g.S : ts;
  const int per = T.head ? g.Sh : g.S;
  T.m = tj / per;
  const int st = tj % per;
  const int64_t p0 = z_param(a, T, r, st);
  const ProbeKey pk = make_probe_key(s.seed, s.step, (uint32_t)e, (uint32_t)i);
  const size_t row = b * kZRows + (size_t)r;
  if (!SOMA_CHECK(row < a.n_zrows, a.status)) return;
  ZSlot c;
  c.blk = 0xFFFFFFFFu;
  uint2 w;
  w.x = z_run_raw(pk, p0, c);
  w.y = z_run_raw(pk, p0 + 32, c);
  out[row] = w;
  if (SPARSE) {
    const ProbeKey pka = activity_key(pk);
    c.blk = 0xFFFFFFFFu;
    w.x = z_run_raw(pka, p0, c);
    w.y = z_run_raw(pka, p0 + 32, c);
    out[a.n_zrows + row] = w;
  }
}

// fp16 A tiles of the gate weights ([x part | h part], gate-major rows) and
// of the head weights: block (tix, e) of (MT * S + 2 * Sh, N), 128 threads,
// thread r writes row r of a tile.
__device__ void prep_tiles_block(const TcArgs& a, int tix, int e) {
  const TcGeom& g = a.g;
  const Sweep& s = a.sw;
  const Layout& L = s.lay;
  const float* th = s.params + (int64_t)e * L.P;
  const int r = threadIdx.x;
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
          if (k < g.E && SOMA_CHECK((size_t)(e * L.P + L.w_ih + R * g.E + k) < a.n_params,
                                    a.status))
            w = th[L.w_ih + R * g.E + k];
        } else {
          const int k = kKt * (st - g.Sx) + kk;
          if (k < g.H && SOMA_CHECK((size_t)(e * L.P + L.w_hh + R * g.H + k) < a.n_params,
                                    a.status))
            w = th[L.w_hh + R * g.H + k];
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
      const bool in =
          k < g.H && SOMA_CHECK((size_t)(e * L.P + L.w_out + (int64_t)vrow * g.H + k) < a.n_params,
                                a.status);
      v[kk] = __float2half_rn(in ? th[L.w_out + (int64_t)vrow * g.H + k] : 0.f);
    }
    tile = const_cast<uint8_t*>(a.wo16) + (((size_t)e * 2 + vh) * g.Sh + st) * kTileA;
  }
  const bool head = tix >= g.MT * g.S;
  const size_t off = (size_t)(tile - (head ? a.wo16 : a.w16));
  if (!SOMA_CHECK(off + kTileA <= (head ? a.n_wo16 : a.n_w16), a.status)) return;
#pragma unroll
  for (int kc = 0; kc < kKt / 8; ++kc)
    *reinterpret_cast<uint4*>(tile + kmajor_offset(r, 8 * kc, kKt)) =
        *reinterpret_cast<const uint4*>(v + 8 * kc);
}

// Everything a sweep needs before its embedding part and its persistent
// launch, in one launch of 128-thread blocks: the fp16 weight tiles
// (n_tiles blocks), the probe-word table (n_zb), the embedding rows' probe
// words (n_eb), then the zeroing of both operand buffers and the phase
// counters (the remaining blocks, grid-stride).
struct PrepJobs {
  int n_tiles, n_zb, n_eb;
  uint4* op0;
  uint4* op1;
  size_t op_vec;  // uint4 per operand buffer
  int* cnt;
  int n_cnt;
};

template <bool SPARSE>
__global__ void __launch_bounds__(128) sweep_prep_kernel(const TcArgs a, const PrepJobs j) {
  int b = (int)blockIdx.x;
  const int per_e = a.g.MT * a.g.S + 2 * a.g.Sh;
  if (b < j.n_tiles) {
    prep_tiles_block(a, b % per_e, b / per_e);
    return;
  }
  b -= j.n_tiles;
  if (b < j.n_zb) {
    zbits_block<SPARSE>(a, a.zb_out, (size_t)b);
    return;
  }
  b -= j.n_zb;
  if (b < j.n_eb) {
    emb_bits_block(a, b);
    return;
  }
  b -= j.n_eb;
  const size_t nz = gridDim.x - (size_t)(j.n_tiles + j.n_zb + j.n_eb);
  const uint4 zero = make_uint4(0u, 0u, 0u, 0u);
  for (size_t v = (size_t)b * blockDim.x + threadIdx.x; v < j.op_vec; v += nz * blockDim.x) {
    j.op0[v] = zero;
    j.op1[v] = zero;
  }
  if (b == 0)
    for (int c = (int)threadIdx.x; c < j.n_cnt; c += blockDim.x) j.cnt[c] = 0;
}

// Per (expert, probe) pair: merge the two vocabulary halves into the NLL of
// every target, then L+, L- (fp64 sums), D = mean(nll+ - nll-) and D / (2 eps).
__global__ void __launch_bounds__(256)
reduce_tc_kernel(const float* __restrict__ pm, const float* __restrict__ ps,
                 const float* __restrict__ ply, int n_sign, int BT, float eps, float* losses_out,
                 float* coef_out, float* coef_ws, int* status, size_t n_ply) {
  __shared__ double red[3][256];
  const int pair = blockIdx.x;
  const int64_t lp = (int64_t)pair * 2, lm = lp + 1;
  double sp = 0.0, sm = 0.0, sd = 0.0;
  for (int j = threadIdx.x; j < BT; j += 256) {
    if (!SOMA_CHECK((size_t)(lm * BT + j) < n_ply, status)) break;
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
    // the difference in fp64: exact for any two fp32 values
    sd += (double)nll[0] - (double)nll[1];
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
// canonical layout (K <= 256, N <= 256, both multiples of 16).  With
// a_in_tmem, A is stored into tensor memory instead (lane = row, column c =
// the k pair 2c, 2c + 1) and the MMA takes it from there, as the probe
// tiles of the forward kernel.
__global__ void __launch_bounds__(128, 1)
debug_tc_gemm_kernel(const __half* A, const __half* B, float* D, int N, int K, int a_in_tmem,
                     int* status) {
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
  if (tid < 32) tmem_alloc(&slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = slot;
  const int warp = tid >> 5, lane = tid & 31;
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
  const uint32_t ta = tmem + 256;  // A in TMEM: columns 256 .. 256 + K / 2
  if (a_in_tmem) {
    // thread = row (lane quarter of its warp), 16 columns (32 k) per store
    const uint32_t trow = ta + ((uint32_t)(32 * warp) << 16);
    const uint32_t* arow = reinterpret_cast<const uint32_t*>(A + (size_t)(32 * warp + lane) * K);
    for (int c0 = 0; c0 < K / 2; c0 += 16) {
      uint32_t r[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) r[j] = arow[c0 + j];
      tmem_st16(trow + c0, r);
    }
    tmem_wait_st();
  }
  fence_async_smem();
  tc_fence_before();
  __syncthreads();
  if (tid == 0) {
    tc_fence_after();
    const uint32_t idesc = idesc_f16_f32(128, N);
    const uint64_t db = smem_desc(smem_u32(sb), 128, K * 16);
    for (int k16 = 0; k16 < K / 16; ++k16) {
      if (a_in_tmem)
        mma_f16_ts_lohi(tmem, ta + 8 * k16, (uint32_t)db + 16 * k16, (uint32_t)(db >> 32), idesc,
                        k16 > 0 ? 1u : 0u);
      else
        mma_f16_ss(tmem, smem_desc(smem_u32(sa) + k16 * 256, 128, K * 16),
                   smem_desc(smem_u32(sb) + k16 * 256, 128, K * 16), idesc, k16 > 0 ? 1u : 0u);
    }
    mma_commit(&bar);
  }
  if (!mbar_wait(&bar, 0) && tid == 0) atomicCAS(status, 0, kStatusTimeout);
  tc_fence_after();
  for (int c0 = 0; c0 < N; c0 += 8) {
    float v[8];
    tmem_ld8(tmem + ((uint32_t)(32 * warp) << 16) + c0, v);
    for (int j = 0; j < 8; ++j) D[(size_t)(32 * warp + lane) * N + c0 + j] = v[j];
  }
  tc_fence_before();
  __syncthreads();
  if (tid < 32) tmem_dealloc(tmem, 512);
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

TcGeom make_tc_geom(const Layout& lay, int n_experts, int n_pert, int B, int T, int B_mem) {
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
  // the accumulator of a group, 2 Bp P columns, fits one 128-column buffer
  int P = g.Bp <= 32 ? 2 : 1;
  if (P > n_pert) P = n_pert;
  if (P < 1) P = 1;
  g.P = P;
  g.G = (n_pert + P - 1) / P;
  g.rowsB = 3 * g.Bp * P;
  g.tileB = (uint32_t)g.rowsB * kKt * 2;
  g.n_experts = n_experts;
  g.n_pert = n_pert;
  g.B = B;
  g.Bm = B_mem;
  g.T = T;
  g.inf = 0;
  return g;
}

TcGeom make_tc_geom_inf(const Layout& lay, int n_experts, int B, int T) {
  TcGeom g = make_tc_geom(lay, n_experts, 1, 32, T, B);
  g.P = 2;
  g.G = (B + kInfGroupSeqs - 1) / kInfGroupSeqs;
  g.rowsB = 3 * g.Bp * g.P;
  g.tileB = (uint32_t)g.rowsB * kKt * 2;
  g.B = B;
  g.inf = 1;
  return g;
}

// The embedding rows' probe words ([N][n][256][Ep / 32] uint2), rounded to 1 KB.
size_t xbits_bytes(const TcGeom& g) {
  const size_t b = (size_t)g.n_experts * g.n_pert * 256 * (g.Ep / 32) * sizeof(uint2);
  return (b + 1023) & ~(size_t)1023;
}

TcSizes tc_sizes(const TcGeom& g) {
  TcSizes z;
  const size_t N = (size_t)g.n_experts, n = (size_t)g.n_pert;
  z.w16 = N * g.MT * g.S * kTileA;
  z.wo16 = N * 2 * g.Sh * kTileA;
  z.op = N * g.S * g.G * g.tileB;
  z.cst = N * (size_t)cst_lanes(g) * 2 * (size_t)g.Hp * g.Bp * sizeof(float);
  z.pm = N * n * 2 * g.Bm * (size_t)g.T * 2 * sizeof(float);
  z.ply = N * n * 2 * g.Bm * (size_t)g.T * sizeof(float);
  // raw words and activity words
  z.zb = 2 * N * n * (size_t)zbits_stages(g) * kZRows * sizeof(uint2);
  // phase counters: prod and hd per (expert, group), then the task counter
  z.cnt = (2 * N * (size_t)g.G + 1) * sizeof(int);
  // the embedding-part tiles, after the embedding rows' probe words
  z.xall = xbits_bytes(g) + (size_t)g.T * N * g.Sx * g.G * g.tileB;
  return z;
}

cudaError_t launch_forward_tc(const Sweep& s, const TcGeom& g, const TcBuffers& tb, int* status,
                              cudaStream_t stream) {
  const size_t smem = kernel_smem_bytes(g);
  auto kernel = g.inf ? tc_persistent_kernel<false, true>
                      : s.sparse ? tc_persistent_kernel<true, false> : tc_persistent_kernel<false, false>;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  const TcSizes z = tc_sizes(g);
  TcArgs a;
  a.sw = s;
  a.g = g;
  a.w16 = tb.w16;
  a.wo16 = tb.wo16;
  a.cst = tb.cst;
  a.pm = tb.pm;
  a.ps = tb.ps;
  a.ply = tb.ply;
  a.zb = tb.zbits;
  a.zb_out = tb.zbits;
  a.n_zrows = (size_t)g.n_experts * g.n_pert * zbits_stages(g) * kZRows;
  a.status = status;
  a.n_w16 = z.w16;
  a.n_wo16 = z.wo16;
  a.n_op = z.op;
  a.xbits = reinterpret_cast<uint2*>(tb.xall);
  a.n_xbits = (size_t)g.n_experts * g.n_pert * 256 * (g.Ep / 32);
  a.xall = tb.xall + xbits_bytes(g);
  a.n_xall = z.xall - xbits_bytes(g);
  a.n_bytes = (size_t)(s.batch_per_probe ? s.n_experts * s.n_pert : s.n_experts) * s.B_mem *
              (size_t)(s.T + 1);
  a.n_cst = z.cst / sizeof(float);
  a.n_pm = z.pm / sizeof(float);
  a.n_ply = z.ply / sizeof(float);
  a.n_params = (size_t)s.n_experts * s.lay.P;
  a.smem_bytes = (uint32_t)smem;
  a.op[0] = tb.op[0];
  a.op[1] = tb.op[1];
  a.prod = tb.cnt;
  a.hd = tb.cnt + (size_t)g.n_experts * g.G;
  a.next_task = tb.cnt + 2 * (size_t)g.n_experts * g.G;
  a.gate_tasks = g.n_experts * g.MT * g.G;
  a.head_tasks = g.n_experts * 2 * g.G;
  a.total_tasks = (a.gate_tasks + a.head_tasks) * s.T;

  // Two launches before the sweep: the weight tiles, the probe-word tables
  // and the zeroed operand buffers and counters; then the embedding part of
  // every timestep's operand (it reads the embedding rows' probe words).
  PrepJobs j;
  j.n_tiles = (g.MT * g.S + 2 * g.Sh) * g.n_experts;
  j.n_zb = s.eps != 0.f ? (int)(a.n_zrows / kZRows) : 0;
  j.n_eb = s.eps != 0.f && !g.inf ? 2 * g.n_experts * s.n_pert : 0;
  j.op0 = reinterpret_cast<uint4*>(tb.op[0]);
  j.op1 = reinterpret_cast<uint4*>(tb.op[1]);
  j.op_vec = z.op / sizeof(uint4);
  j.cnt = tb.cnt;
  j.n_cnt = (int)(z.cnt / sizeof(int));
  const size_t zb_need = (j.op_vec + 1023) / 1024;
  const int zero_blocks = (int)(zb_need < 1 ? 1 : zb_need < 4096 ? zb_need : 4096);
  const unsigned pblocks = (unsigned)(j.n_tiles + j.n_zb + j.n_eb + zero_blocks);
  trace_begin(SOMA_TRACE_PREP, stream);
  if (s.sparse)
    sweep_prep_kernel<true><<<pblocks, 128, 0, stream>>>(a, j);
  else
    sweep_prep_kernel<false><<<pblocks, 128, 0, stream>>>(a, j);
  const int xtiles = g.n_experts * g.Sx * g.G;
  const unsigned xblocks = (unsigned)((size_t)xtiles * s.T);
  uint8_t* xall = tb.xall + xbits_bytes(g);
  if (g.inf)
    xpart_kernel<true><<<xblocks, 128, 0, stream>>>(a, xall, xtiles);
  else
    xpart_kernel<false><<<xblocks, 128, 0, stream>>>(a, xall, xtiles);
  trace_end(SOMA_TRACE_PREP, stream);

  // every phase of the sweep in one cooperative launch: its CTAs wait on
  // each other's phase counters, so all of them must be resident together
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kThreads, smem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorLaunchOutOfResources;
  const int sms = sm_count();
  const int tasks = a.gate_tasks + a.head_tasks;
  const int ctas = tasks < sms ? tasks : sms;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)ctas);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  trace_begin(SOMA_TRACE_GATE, stream);
  e = cudaLaunchKernelEx(&cfg, kernel, a);
  trace_end(SOMA_TRACE_GATE, stream);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_reduce_tc(const TcBuffers& tb, int pairs, int n_sign, int B, int T, float eps,
                             float* losses_out, float* coef_out, float* coef_ws, int* status,
                             cudaStream_t stream) {
  trace_begin(SOMA_TRACE_REDUCE, stream);
  reduce_tc_kernel<<<pairs, 256, 0, stream>>>(tb.pm, tb.ps, tb.ply, n_sign, B * T, eps,
                                               losses_out, coef_out, coef_ws, status,
                                               (size_t)pairs * 2 * B * T);
  trace_end(SOMA_TRACE_REDUCE, stream);
  return cudaGetLastError();
}

cudaError_t launch_debug_tc_gemm(const void* A, const void* B, float* D, int N, int K,
                                 int a_in_tmem, int* status, cudaStream_t stream) {
  const size_t smem = (size_t)(128 + N) * K * 2 + 1024;
  cudaError_t e = cudaFuncSetAttribute(debug_tc_gemm_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  debug_tc_gemm_kernel<<<1, 128, smem, stream>>>(static_cast<const __half*>(A),
                                                 static_cast<const __half*>(B), D, N, K, a_in_tmem,
                                                 status);
  return cudaGetLastError();
}

}  // namespace soma
