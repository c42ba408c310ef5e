// soma_api.cu -- the C ABI of libsoma.so (declared in include/soma_api.h):
// argument validation, workspace carving and the launch sequence of one SPSA
// step (Eq. main-spsa): forward sweep over all (expert, probe, sign) lanes,
// loss reduction into L+, L- and coefficients, Philox-regenerating update.
#include <cmath>
#include <cstdint>
#include <cstring>
#include <vector>

#define SOMA_CHECK_FILE 7
#include "checked.cuh"
#include "soma_api.h"
#include "body_device.cuh"
#include "soma_launch.h"

using namespace soma;

// Per-device status word (see soma_get_status) and, after it, the position of
// the first failed index check of the checked build (soma_debug_check_line).
// Kernels get the address of the pair as their status argument; only
// soma_get_status and soma_debug_check_line read and clear it.
__device__ int g_soma_status[2] = {0, 0};

namespace {

constexpr int kMaxDevices = 64;
constexpr int kMaxPert = 12 * 1024;  // coefficients of one expert staged in shared memory
int* g_status_ptr[kMaxDevices] = {nullptr};

int* status_ptr() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  if (!g_status_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_soma_status) != cudaSuccess) return nullptr;
    g_status_ptr[dev] = static_cast<int*>(p);
  }
  return g_status_ptr[dev];
}

bool dims_ok(const soma_dims& d) {
  return d.vocab == kVocab && d.embed >= 1 && d.embed <= 1024 && d.hidden >= 1 &&
         d.hidden <= 4096;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

constexpr size_t kAlign = 256;
size_t round_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Workspace layout: regions in order, each rounded up to 256 bytes.  The
// checked build puts a 256-byte canary gap before every region and after
// the last; the gaps are filled before a step and checked after it.
#ifdef SOMA_CHECKED
constexpr size_t kGuard = 256;
#else
constexpr size_t kGuard = 0;
#endif
constexpr int kMaxRegions = 12;

struct Regions {
  int n;
  size_t off[kMaxRegions];
  size_t end;
  size_t add(size_t bytes) {
    off[n] = end + kGuard;
    end = off[n] + round_up(bytes);
    return off[n++];
  }
  size_t total() const { return end + kGuard; }
};

#ifdef SOMA_CHECKED
constexpr uint32_t kCanaryWord = 0x5A17C0DEu;

// The canary gaps of a workspace: before each region and after the last.
struct Gaps {
  int n;
  size_t off[kMaxRegions + 1];
};

Gaps gaps_of(const Regions& r) {
  Gaps g;
  g.n = r.n + 1;
  for (int i = 0; i < r.n; ++i) g.off[i] = r.off[i] - kGuard;
  g.off[r.n] = r.end;
  return g;
}

__global__ void canary_fill_kernel(uint32_t* ws, Gaps g) {
  for (int j = threadIdx.x; j < g.n * (int)(kGuard / 4); j += blockDim.x) {
    const int k = j / (int)(kGuard / 4), w = j % (int)(kGuard / 4);
    ws[g.off[k] / 4 + w] = kCanaryWord;
  }
}

// A canary word that changed means a kernel wrote outside its region:
// SOMA_ERR_BOUNDS, position 90000 + the gap index.
__global__ void canary_check_kernel(const uint32_t* ws, Gaps g, int* status) {
  for (int j = threadIdx.x; j < g.n * (int)(kGuard / 4); j += blockDim.x) {
    const int k = j / (int)(kGuard / 4), w = j % (int)(kGuard / 4);
    if (ws[g.off[k] / 4 + w] != kCanaryWord) {
      atomicCAS(status, 0, kStatusBounds);
      atomicCAS(status + 1, 0, 90000 + k);
    }
  }
}
#endif

cudaError_t canary_fill(const Regions& r, void* ws, cudaStream_t st) {
#ifdef SOMA_CHECKED
  canary_fill_kernel<<<1, 256, 0, st>>>(static_cast<uint32_t*>(ws), gaps_of(r));
  return cudaGetLastError();
#else
  (void)r, (void)ws, (void)st;
  return cudaSuccess;
#endif
}

cudaError_t canary_check(const Regions& r, const void* ws, int* status, cudaStream_t st) {
#ifdef SOMA_CHECKED
  canary_check_kernel<<<1, 256, 0, st>>>(static_cast<const uint32_t*>(ws), gaps_of(r), status);
  return cudaGetLastError();
#else
  (void)r, (void)ws, (void)status, (void)st;
  return cudaSuccess;
#endif
}

// Workspace of one sweep with `n_pert` probes and `n_sign` signs.  Small
// experts run on the resident kernel (only the coefficients need scratch);
// every other batch runs on the persistent tensor-core kernel (both signs
// always), in chunks of at most kTcMaxBatch sequences that share the
// operand and cell buffers and write their loss partials into buffers of
// the whole batch.
struct WsPlan {
  bool res;    // the resident small-expert kernel: no scratch but the coefficients
  TcGeom g;    // geometry of the largest chunk
  TcSizes z;   // buffer sizes: the largest chunk's operand and cell buffers
  Regions r;   // w16, wo16, op[0], op[1], cst, pm, ps, ply, zbits, cnt, coef; or coef alone
  size_t total;
};

int chunk_size(int B, int b0) { return B - b0 < kTcMaxBatch ? B - b0 : kTcMaxBatch; }

// A sweep of n_pert probes and n_sign signs.  With n_sign == 1 (eps = 0:
// evaluation and routed inference) the tensor path takes the unperturbed
// layout, every sequence of the batch in one sweep.
WsPlan plan_sweep(const soma_dims& d, int n_experts, int n_pert, int n_sign, int B, int T,
                  bool allow_res = true) {
  WsPlan w;
  std::memset(&w, 0, sizeof(w));
  const Layout lay = make_layout(d.embed, d.hidden);
  const size_t coef = (size_t)n_experts * n_pert * sizeof(float);
  if (allow_res && res_supported(lay, B)) {
    w.res = true;
    w.r.add(coef);
    w.total = w.r.total();
    return w;
  }
  if (n_sign == 1) {
    w.g = make_tc_geom_inf(lay, n_experts, B, T);
    w.z = tc_sizes(w.g);
  } else {
    // the operand and cell buffers of every chunk fit those of the first one
    // or of the last (smaller Bp packs two probes per group)
    w.g = make_tc_geom(lay, n_experts, n_pert, chunk_size(B, 0), T, B);
    w.z = tc_sizes(w.g);
    const int last = chunk_size(B, (B - 1) / kTcMaxBatch * kTcMaxBatch);
    const TcSizes zl = tc_sizes(make_tc_geom(lay, n_experts, n_pert, last, T, B));
    if (zl.op > w.z.op) w.z.op = zl.op;
    if (zl.cst > w.z.cst) w.z.cst = zl.cst;
    if (zl.cnt > w.z.cnt) w.z.cnt = zl.cnt;
    if (zl.xall > w.z.xall) w.z.xall = zl.xall;
  }
  for (size_t bytes :
       {w.z.w16, w.z.wo16, w.z.op, w.z.op, w.z.cst, w.z.pm, w.z.pm, w.z.ply, w.z.zb, w.z.cnt,
        w.z.xall, coef})
    w.r.add(bytes);
  w.total = w.r.total();
  return w;
}

TcBuffers carve_tc(const WsPlan& w, void* ws) {
  uint8_t* p = static_cast<uint8_t*>(ws);
  TcBuffers tb;
  tb.w16 = p + w.r.off[0];
  tb.wo16 = p + w.r.off[1];
  tb.op[0] = p + w.r.off[2];
  tb.op[1] = p + w.r.off[3];
  tb.cst = reinterpret_cast<float*>(p + w.r.off[4]);
  tb.pm = reinterpret_cast<float*>(p + w.r.off[5]);
  tb.ps = reinterpret_cast<float*>(p + w.r.off[6]);
  tb.ply = reinterpret_cast<float*>(p + w.r.off[7]);
  tb.zbits = reinterpret_cast<uint2*>(p + w.r.off[8]);
  tb.cnt = reinterpret_cast<int*>(p + w.r.off[9]);
  tb.xall = p + w.r.off[10];
  return tb;
}

// The tensor-core forward of a whole batch: one sweep per chunk of at most
// kTcMaxBatch sequences (each with its own geometry), all writing the loss
// partials of the batch.
cudaError_t forward_tc_chunks(Sweep s, const Layout& lay, const TcBuffers& tb, int* status,
                              cudaStream_t st) {
  const int B = s.B;
  s.B_mem = B;
  cudaError_t e = cudaSuccess;
  for (int b0 = 0; b0 < B && e == cudaSuccess; b0 += kTcMaxBatch) {
    s.b0 = b0;
    s.B = chunk_size(B, b0);
    const TcGeom g = make_tc_geom(lay, s.n_experts, s.n_pert, s.B, s.T, B);
    e = launch_forward_tc(s, g, tb, status, st);
  }
  return e;
}

// the coefficient scratch is the last region of both layouts
float* coef_scratch(const WsPlan& w, void* ws) {
  return reinterpret_cast<float*>(static_cast<char*>(ws) + w.r.off[w.r.n - 1]);
}

bool sizes_ok(int n_experts, int n_pert, int batch, int seq_len) {
  // lanes index the grid's x dimension and probe/expert indices fit Philox
  // counter words (expert < 2^31 keeps the init domain disjoint)
  if (n_experts < 1 || n_pert < 1 || batch < 1 || seq_len < 1) return false;
  if (n_pert > kMaxPert) return false;
  if ((int64_t)n_experts * n_pert * 2 > (int64_t)INT32_MAX) return false;
  if ((int64_t)batch * (seq_len + 1) > (int64_t)INT32_MAX) return false;
  return true;
}

int cuda_status(cudaError_t e) { return e == cudaSuccess ? SOMA_OK : SOMA_ERR_CUDA; }

}  // namespace

extern "C" {

int64_t soma_param_count(soma_dims d) {
  if (!dims_ok(d)) return -1;
  return make_layout(d.embed, d.hidden).P;
}

size_t soma_workspace_bytes(soma_dims d, int n_experts, int n_pert, int batch, int seq_len) {
  if (!dims_ok(d) || !sizes_ok(n_experts, n_pert, batch, seq_len)) return 0;
  const WsPlan step = plan_sweep(d, n_experts, n_pert, 2, batch, seq_len);
  const WsPlan eval = plan_sweep(d, n_experts, 1, 1, batch, seq_len);
  return step.total > eval.total ? step.total : eval.total;
}

int soma_init_experts(float* params, int n_experts, soma_dims d, uint64_t seed, float std,
                      void* stream) {
  if (!dims_ok(d)) return SOMA_ERR_UNSUPPORTED;
  if (!params || !aligned16(params) || n_experts < 1 || !(std >= 0.f) || !std::isfinite(std))
    return SOMA_ERR_INVALID_ARG;
  const Layout lay = make_layout(d.embed, d.hidden);
  return cuda_status(launch_init(params, lay, n_experts, seed, std, (cudaStream_t)stream));
}

// Forward sweep, reduction and (optionally) the SGD update of one step.
static int spsa_forward(float* params, int n_experts, soma_dims d, int n_pert, int sparse,
                        int batch_per_probe, int summed_loss,
                        float eps, float lr, bool update, uint64_t seed, uint64_t step,
                        const uint8_t* byte_batch, int batch, int seq_len, float* losses_out,
                        float* coef_out, void* workspace, size_t workspace_bytes, void* stream) {
  if (!dims_ok(d)) return SOMA_ERR_UNSUPPORTED;
  if (!params || !byte_batch || !losses_out || !aligned16(params) ||
      !sizes_ok(n_experts, n_pert, batch, seq_len) || !(eps >= 0.f) || !std::isfinite(eps) ||
      !std::isfinite(lr))
    return SOMA_ERR_INVALID_ARG;
  const WsPlan w = plan_sweep(d, n_experts, n_pert, 2, batch, seq_len);
  if (!workspace || !aligned16(workspace) || workspace_bytes < w.total) return SOMA_ERR_WORKSPACE;
  int* status = status_ptr();
  if (!status) return SOMA_ERR_CUDA;
  cudaStream_t st = (cudaStream_t)stream;

  Sweep s;
  s.params = params;
  s.bytes = byte_batch;
  s.lay = make_layout(d.embed, d.hidden);
  s.n_experts = n_experts;
  s.n_pert = n_pert;
  s.n_sign = 2;
  s.B = batch;
  s.T = seq_len;
  s.b0 = 0;
  s.B_mem = batch;
  s.eps = eps;
  s.sparse = sparse;
  s.batch_per_probe = batch_per_probe;
  s.seed = seed;
  s.step = step;
  float* coef_ws = coef_scratch(w, workspace);
  cudaError_t e = canary_fill(w.r, workspace, st);
  if (e != cudaSuccess) {
  } else if (w.res) {
    e = launch_forward_res(s, 2, losses_out, coef_out, coef_ws, status, st);
  } else {
    const TcBuffers tb = carve_tc(w, workspace);
    e = forward_tc_chunks(s, s.lay, tb, status, st);
    if (e == cudaSuccess)
      e = launch_reduce_tc(tb, n_experts * n_pert, 2, batch, seq_len, eps, losses_out, coef_out,
                           coef_ws, status, st);
  }
  if (summed_loss && e == cudaSuccess) e = launch_sum_over_experts(coef_out, n_experts, n_pert, st);
  // eps == 0 makes every coefficient 0 and lr == 0 every step 0: theta stays
  // bit-identical, so the update is not launched at all.
  if (update && e == cudaSuccess && eps != 0.f && lr != 0.f)
    e = launch_spsa_update(params, s.lay, n_experts, n_pert, lr, seed, step, coef_ws, st);
  if (e == cudaSuccess) e = canary_check(w.r, workspace, status, st);
  return cuda_status(e);
}

int soma_spsa_step(float* params, int n_experts, soma_dims d, int n_pert, float eps, float lr,
                   uint64_t seed, uint64_t step, const uint8_t* byte_batch, int batch,
                   int seq_len, float* losses_out, float* coef_out, void* workspace,
                   size_t workspace_bytes, void* stream) {
  return spsa_forward(params, n_experts, d, n_pert, 0, 0, 0, eps, lr, true, seed, step, byte_batch,
                      batch, seq_len, losses_out, coef_out, workspace, workspace_bytes, stream);
}

int soma_spsa_estimate_opts(const float* params, int n_experts, soma_dims d, int n_pert,
                            const soma_estimate_options* opts, float eps, uint64_t seed,
                            uint64_t step, const uint8_t* byte_batch, int batch, int seq_len,
                            float* losses_out, float* coef_out, void* workspace,
                            size_t workspace_bytes, void* stream) {
  if (!dims_ok(d)) return SOMA_ERR_UNSUPPORTED;
  if (!coef_out || !opts ||
      (opts->probe_kind != SOMA_PROBE_DENSE && opts->probe_kind != SOMA_PROBE_SPARSE) ||
      (opts->batch_per_probe != 0 && opts->batch_per_probe != 1) ||
      (opts->summed_loss != 0 && opts->summed_loss != 1))
    return SOMA_ERR_INVALID_ARG;
  // the forward sweep only reads params
  return spsa_forward(const_cast<float*>(params), n_experts, d, n_pert, opts->probe_kind,
                      opts->batch_per_probe, opts->summed_loss, eps, 0.f, false, seed, step,
                      byte_batch, batch, seq_len, losses_out, coef_out, workspace,
                      workspace_bytes, stream);
}

int soma_spsa_estimate(const float* params, int n_experts, soma_dims d, int n_pert,
                       int probe_kind, float eps, uint64_t seed, uint64_t step,
                       const uint8_t* byte_batch, int batch, int seq_len, float* losses_out,
                       float* coef_out, void* workspace, size_t workspace_bytes, void* stream) {
  const soma_estimate_options opts = {probe_kind, 0, 0};
  return soma_spsa_estimate_opts(params, n_experts, d, n_pert, &opts, eps, seed, step,
                                 byte_batch, batch, seq_len, losses_out, coef_out, workspace,
                                 workspace_bytes, stream);
}

int soma_adam_update(float* params, float* m, float* v, int n_experts, soma_dims d, int n_pert,
                     int probe_kind, uint64_t seed, const uint64_t* steps, int n_acc,
                     const float* coef, soma_adam_config cfg, void* stream) {
  if (!dims_ok(d)) return SOMA_ERR_UNSUPPORTED;
  if (!params || !m || !v || !coef || !steps || !aligned16(params) || !aligned16(m) ||
      !aligned16(v) || n_experts < 1 || n_pert < 1 || n_pert > kMaxPert || n_acc < 1 ||
      n_acc > SOMA_MAX_ACCUM || (probe_kind != SOMA_PROBE_DENSE && probe_kind != SOMA_PROBE_SPARSE))
    return SOMA_ERR_INVALID_ARG;
  if (!std::isfinite(cfg.lr) || !(cfg.beta1 >= 0.f && cfg.beta1 < 1.f) ||
      !(cfg.beta2 >= 0.f && cfg.beta2 < 1.f) || !(cfg.delta > 0.f) || !std::isfinite(cfg.delta) ||
      !(cfg.weight_decay >= 0.f) || !std::isfinite(cfg.weight_decay) || cfg.t < 1)
    return SOMA_ERR_INVALID_ARG;
  AdamSteps st;
  st.n_acc = n_acc;
  for (int a = 0; a < n_acc; ++a) st.step[a] = steps[a];
  AdamArgs h;
  h.lr = cfg.lr;
  h.b1 = cfg.beta1;
  h.b2 = cfg.beta2;
  h.delta = cfg.delta;
  h.wd = cfg.weight_decay;
  // bias corrections in double, then rounded once
  h.inv_bc1 = (float)(1.0 / (1.0 - std::pow((double)cfg.beta1, (double)cfg.t)));
  h.inv_bc2 = (float)(1.0 / (1.0 - std::pow((double)cfg.beta2, (double)cfg.t)));
  const Layout lay = make_layout(d.embed, d.hidden);
  return cuda_status(launch_adam_update(params, m, v, lay, n_experts, n_pert, probe_kind, seed, st,
                                        coef, h, (cudaStream_t)stream));
}

int soma_eval_loss(const float* params, int n_experts, soma_dims d, const uint8_t* byte_batch,
                   int batch, int seq_len, float* loss_out, void* workspace,
                   size_t workspace_bytes, void* stream) {
  if (!dims_ok(d)) return SOMA_ERR_UNSUPPORTED;
  if (!params || !byte_batch || !loss_out || !aligned16(params) ||
      !sizes_ok(n_experts, 1, batch, seq_len))
    return SOMA_ERR_INVALID_ARG;
  const WsPlan w = plan_sweep(d, n_experts, 1, 1, batch, seq_len);
  if (!workspace || !aligned16(workspace) || workspace_bytes < w.total) return SOMA_ERR_WORKSPACE;
  int* status = status_ptr();
  if (!status) return SOMA_ERR_CUDA;
  cudaStream_t st = (cudaStream_t)stream;
  Sweep s;
  s.params = params;
  s.bytes = byte_batch;
  s.lay = make_layout(d.embed, d.hidden);
  s.n_experts = n_experts;
  s.n_pert = 1;
  s.n_sign = 1;
  s.B = batch;
  s.T = seq_len;
  s.b0 = 0;
  s.B_mem = batch;
  s.eps = 0.f;
  s.sparse = 0;
  s.batch_per_probe = 0;
  s.seed = 0;
  s.step = 0;
  cudaError_t e = canary_fill(w.r, workspace, st);
  if (e != cudaSuccess) {
  } else if (w.res) {
    e = launch_forward_res(s, 1, loss_out, nullptr, nullptr, status, st);
  } else {
    const TcBuffers tb = carve_tc(w, workspace);
    e = launch_forward_tc(s, w.g, tb, status, st);
    if (e == cudaSuccess)
      e = launch_reduce_tc(tb, n_experts, 1, batch, seq_len, 0.f, loss_out, nullptr, nullptr,
                           status, st);
  }
  if (e == cudaSuccess) e = canary_check(w.r, workspace, status, st);
  return cuda_status(e);
}

int soma_spsa_update(float* params, int n_experts, soma_dims d, int n_pert, float lr,
                     uint64_t seed, uint64_t step, const float* coef, void* stream) {
  if (!dims_ok(d)) return SOMA_ERR_UNSUPPORTED;
  if (!params || !coef || !aligned16(params) || n_experts < 1 || n_pert < 1 ||
      n_pert > kMaxPert || !std::isfinite(lr))
    return SOMA_ERR_INVALID_ARG;
  if (lr == 0.f) return SOMA_OK;
  const Layout lay = make_layout(d.embed, d.hidden);
  return cuda_status(
      launch_spsa_update(params, lay, n_experts, n_pert, lr, seed, step, coef, (cudaStream_t)stream));
}

int soma_checked_build(void) {
#ifdef SOMA_CHECKED
  return 1;
#else
  return 0;
#endif
}

int soma_debug_check_line(void* stream) {
  if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return -1;
  int* p = status_ptr();
  if (!p) return -1;
  int v = 0;
  if (cudaMemcpy(&v, p + 1, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return -1;
  const int zero = 0;
  if (cudaMemcpy(p + 1, &zero, sizeof(int), cudaMemcpyHostToDevice) != cudaSuccess) return -1;
  return v;
}

int soma_get_status(void* stream) {
  if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return SOMA_ERR_CUDA;
  int* p = status_ptr();
  if (!p) return SOMA_ERR_CUDA;
  int v = 0;
  if (cudaMemcpy(&v, p, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return SOMA_ERR_CUDA;
  const int zero = 0;
  if (cudaMemcpy(p, &zero, sizeof(int), cudaMemcpyHostToDevice) != cudaSuccess)
    return SOMA_ERR_CUDA;
  return v;
}

const char* soma_status_string(int code) {
  switch (code) {
    case SOMA_OK: return "ok";
    case SOMA_ERR_INVALID_ARG: return "invalid argument";
    case SOMA_ERR_UNSUPPORTED: return "unsupported dimensions";
    case SOMA_ERR_WORKSPACE: return "workspace missing or too small";
    case SOMA_ERR_CUDA: return "CUDA error";
    case SOMA_ERR_TIMEOUT: return "device-side wait timed out";
    case SOMA_ERR_NONFINITE: return "non-finite loss or coefficient";
    case SOMA_ERR_BOUNDS: return "an index check of the checked build failed";
    default: return "unknown status";
  }
}

int soma_debug_philox(uint64_t seed, const uint32_t* ctr4, uint32_t* out4, int count,
                      void* stream) {
  if (!ctr4 || !out4 || count < 0) return SOMA_ERR_INVALID_ARG;
  if (count == 0) return SOMA_OK;
  return cuda_status(launch_debug_philox(seed, ctr4, out4, count, (cudaStream_t)stream));
}

static int debug_tc_gemm(const uint16_t* a, const uint16_t* b, float* d, int n, int k,
                         int a_in_tmem, void* stream) {
  if (!a || !b || !d || !aligned16(a) || !aligned16(b) || n < 16 || n > 256 || n % 16 ||
      k < 16 || k > 256 || k % 16)
    return SOMA_ERR_INVALID_ARG;
  int* status = status_ptr();
  if (!status) return SOMA_ERR_CUDA;
  return cuda_status(launch_debug_tc_gemm(a, b, d, n, k, a_in_tmem, status, (cudaStream_t)stream));
}

int soma_debug_tc_gemm(const uint16_t* a, const uint16_t* b, float* d, int n, int k,
                       void* stream) {
  return debug_tc_gemm(a, b, d, n, k, 0, stream);
}

int soma_debug_tc_gemm_ts(const uint16_t* a, const uint16_t* b, float* d, int n, int k,
                          void* stream) {
  return debug_tc_gemm(a, b, d, n, k, 1, stream);
}

int soma_debug_check_fail(void* stream) {
  int* status = status_ptr();
  if (!status) return SOMA_ERR_CUDA;
  return cuda_status(launch_debug_check_fail(status, (cudaStream_t)stream));
}

int soma_debug_wait_timeout(uint32_t max_polls, void* stream) {
  if (max_polls < 1 || max_polls > (1u << 22)) return SOMA_ERR_INVALID_ARG;
  int* status = status_ptr();
  if (!status) return SOMA_ERR_CUDA;
  return cuda_status(launch_debug_wait_timeout(max_polls, status, (cudaStream_t)stream));
}

int soma_debug_rademacher(uint64_t seed, uint64_t step, int expert, int pert, int64_t p0,
                          int64_t count, int8_t* z_out, void* stream) {
  if (!z_out || count < 0 || p0 < 0 || expert < 0 || pert < 0) return SOMA_ERR_INVALID_ARG;
  if (count == 0) return SOMA_OK;
  return cuda_status(
      launch_debug_rademacher(seed, step, expert, pert, 0, p0, count, z_out, (cudaStream_t)stream));
}

int soma_debug_probe(uint64_t seed, uint64_t step, int expert, int pert, int probe_kind,
                     int64_t p0, int64_t count, int8_t* z_out, void* stream) {
  if (!z_out || count < 0 || p0 < 0 || expert < 0 || pert < 0 ||
      (probe_kind != SOMA_PROBE_DENSE && probe_kind != SOMA_PROBE_SPARSE))
    return SOMA_ERR_INVALID_ARG;
  if (count == 0) return SOMA_OK;
  return cuda_status(launch_debug_rademacher(seed, step, expert, pert, probe_kind, p0, count, z_out,
                                             (cudaStream_t)stream));
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Routed inference (Sec. 3, Eq. main-mixture)
// ---------------------------------------------------------------------------
namespace {

constexpr int kMaxRoutes = 16;

struct MixPlan {
  int b_max;
  WsPlan sweep;
  size_t gather, route, slot, grouped, nll, total;
  std::vector<int32_t> gather_h, slot_h;
};

// Groups the requests by expert: request r's j-th route lands in slot
// slot_h[r][j] of expert routes[r][j]; gather_h[e][slot] = r.
bool plan_mixture(const soma_dims& d, int N, const int32_t* routes, int R, int k, int T,
                  MixPlan& m) {
  std::vector<int> count((size_t)N, 0);
  m.slot_h.assign((size_t)R * k, 0);
  for (int r = 0; r < R; ++r)
    for (int j = 0; j < k; ++j) {
      const int e = routes[(size_t)r * k + j];
      if (e < 0 || e >= N) return false;
      m.slot_h[(size_t)r * k + j] = count[(size_t)e]++;
    }
  m.b_max = 1;
  for (int e = 0; e < N; ++e) m.b_max = count[(size_t)e] > m.b_max ? count[(size_t)e] : m.b_max;
  m.gather_h.assign((size_t)N * m.b_max, -1);
  for (int r = 0; r < R; ++r)
    for (int j = 0; j < k; ++j)
      m.gather_h[(size_t)routes[(size_t)r * k + j] * m.b_max + m.slot_h[(size_t)r * k + j]] = r;
  // one unperturbed sweep over every expert's group of requests; the
  // mixture reads per-target NLL, which the persistent kernel keeps
  m.sweep = plan_sweep(d, N, 1, 1, m.b_max, T, false);
  m.gather = round_up((size_t)N * m.b_max * sizeof(int32_t));
  m.route = round_up((size_t)R * k * sizeof(int32_t));
  m.slot = m.route;
  m.grouped = round_up((size_t)N * m.b_max * (T + 1));
  m.nll = round_up((size_t)N * m.b_max * T * sizeof(float));
  m.total = m.sweep.total + m.gather + m.route + m.slot + m.grouped + m.nll;
  return true;
}

bool mixture_args_ok(int n_experts, const int32_t* routes, int R, int k, int seq_len, int t0) {
  return n_experts >= 1 && routes && R >= 1 && k >= 1 && k <= kMaxRoutes && seq_len >= 1 &&
         t0 >= 0 && t0 < seq_len && sizes_ok(n_experts, 1, 1, seq_len);
}

}  // namespace

size_t soma_mixture_workspace_bytes(soma_dims d, int n_experts, const int32_t* routes, int R,
                                    int k, int seq_len) {
  if (!dims_ok(d) || !mixture_args_ok(n_experts, routes, R, k, seq_len, 0)) return 0;
  MixPlan m;
  if (!plan_mixture(d, n_experts, routes, R, k, seq_len, m)) return 0;
  return m.total;
}

int soma_mixture_nll(const float* params, int n_experts, soma_dims d, const uint8_t* requests,
                     int R, int seq_len, const int32_t* routes, int k, int t0, float* nll_out,
                     void* workspace, size_t workspace_bytes, void* stream) {
  if (!dims_ok(d)) return SOMA_ERR_UNSUPPORTED;
  if (!params || !requests || !nll_out || !aligned16(params) ||
      !mixture_args_ok(n_experts, routes, R, k, seq_len, t0))
    return SOMA_ERR_INVALID_ARG;
  MixPlan m;
  if (!plan_mixture(d, n_experts, routes, R, k, seq_len, m)) return SOMA_ERR_INVALID_ARG;
  if (!workspace || !aligned16(workspace) || workspace_bytes < m.total) return SOMA_ERR_WORKSPACE;
  int* status = status_ptr();
  if (!status) return SOMA_ERR_CUDA;
  cudaStream_t st = (cudaStream_t)stream;
  char* base = static_cast<char*>(workspace);
  void* sweep_ws = base;
  int32_t* gather = reinterpret_cast<int32_t*>(base + m.sweep.total);
  int32_t* route = reinterpret_cast<int32_t*>(base + m.sweep.total + m.gather);
  int32_t* slot = reinterpret_cast<int32_t*>(base + m.sweep.total + m.gather + m.route);
  uint8_t* grouped =
      reinterpret_cast<uint8_t*>(base + m.sweep.total + m.gather + m.route + m.slot);
  float* nll = reinterpret_cast<float*>(base + m.sweep.total + m.gather + m.route + m.slot +
                                        m.grouped);
  // the routing tables (host, built above) go with the stream's work; the
  // copies from pageable memory return once the data is staged
  cudaError_t e = cudaMemcpyAsync(gather, m.gather_h.data(), m.gather_h.size() * sizeof(int32_t),
                                  cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(route, routes, (size_t)R * k * sizeof(int32_t), cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(slot, m.slot_h.data(), m.slot_h.size() * sizeof(int32_t),
                        cudaMemcpyHostToDevice, st);
  Sweep s;
  s.params = params;
  s.bytes = grouped;
  s.lay = make_layout(d.embed, d.hidden);
  s.n_experts = n_experts;
  s.n_pert = 1;
  s.n_sign = 1;
  s.B = m.b_max;
  s.T = seq_len;
  s.b0 = 0;
  s.B_mem = m.b_max;
  s.eps = 0.f;
  s.sparse = 0;
  s.batch_per_probe = 0;
  s.seed = 0;
  s.step = 0;
  if (e == cudaSuccess)
    e = launch_gather_requests(requests, gather, n_experts, m.b_max, 0, m.b_max, seq_len + 1,
                               grouped, st);
  if (e == cudaSuccess) {
    const TcBuffers tb = carve_tc(m.sweep, sweep_ws);
    e = launch_forward_tc(s, m.sweep.g, tb, status, st);
    if (e == cudaSuccess)
      e = launch_token_nll_tc(tb, n_experts, m.b_max, seq_len, m.b_max, 0, nll, st);
  }
  if (e == cudaSuccess)
    e = launch_mixture(nll, route, slot, R, k, seq_len, t0, m.b_max, nll_out, st);
  return cuda_status(e);
}

// ---- The paper's expert body (body.cu) ------------------------------------

namespace {

bool body_dims_ok(const soma_body_dims& d) {
  return d.vocab == kVocab && d.width == kBodyWidth && d.blocks >= 1 &&
         d.blocks <= kBodyMaxBlocks;
}

// fp64 NLL sums [N * n * n_sign][chunks], then the coefficients [N][n].
struct BodyWs {
  Regions r;  // partial, coef
  size_t total;
};

BodyWs plan_body(int n_experts, int n_pert, int n_sign, int B) {
  BodyWs w;
  std::memset(&w, 0, sizeof(w));
  const int chunks = (B + body_rows_per_cta() - 1) / body_rows_per_cta();
  w.r.add((size_t)n_experts * n_pert * n_sign * chunks * sizeof(double));
  w.r.add((size_t)n_experts * n_pert * sizeof(float));
  w.total = w.r.total();
  return w;
}

bool body_sizes_ok(int n_experts, int n_pert, int batch, int seq_len) {
  if (!sizes_ok(n_experts, n_pert, batch, seq_len)) return false;
  return (batch + body_rows_per_cta() - 1) / body_rows_per_cta() <= 65535;
}

int body_forward(float* params, int n_experts, soma_body_dims d, const float* head, int n_pert,
                 int probe_kind, float eps, float lr, bool update, uint64_t seed, uint64_t step,
                 const uint8_t* byte_batch, int batch, int seq_len, float* losses_out,
                 float* coef_out, void* workspace, size_t workspace_bytes, void* stream) {
  if (!body_dims_ok(d)) return SOMA_ERR_UNSUPPORTED;
  if (!params || !head || !byte_batch || !aligned16(params) || !aligned16(head) ||
      !body_sizes_ok(n_experts, n_pert, batch, seq_len) || !(eps >= 0.f) ||
      !std::isfinite(eps) || !std::isfinite(lr) ||
      (probe_kind != SOMA_PROBE_DENSE && probe_kind != SOMA_PROBE_SPARSE) ||
      (!update && !coef_out))
    return SOMA_ERR_INVALID_ARG;
  const BodyWs w = plan_body(n_experts, n_pert, 2, batch);
  if (!workspace || !aligned16(workspace) || workspace_bytes < w.total) return SOMA_ERR_WORKSPACE;
  int* status = status_ptr();
  if (!status) return SOMA_ERR_CUDA;
  cudaStream_t st = (cudaStream_t)stream;
  double* partial = reinterpret_cast<double*>(static_cast<uint8_t*>(workspace) + w.r.off[0]);
  float* coef_ws = reinterpret_cast<float*>(static_cast<uint8_t*>(workspace) + w.r.off[1]);
  cudaError_t e = canary_fill(w.r, workspace, st);
  if (e == cudaSuccess)
    e = launch_body_tc(params, head, byte_batch, n_experts, d.blocks, n_pert, 2, batch, seq_len,
                       eps, probe_kind, seed, step, partial, status, st);
  if (e == cudaSuccess)
    e = launch_body_reduce(partial, n_experts * n_pert, 2, batch, seq_len, eps, losses_out,
                           coef_out, coef_ws, status, st);
  // eps == 0 or lr == 0 leaves theta bit-identical: no update launch
  if (update && e == cudaSuccess && eps != 0.f && lr != 0.f)
    e = launch_body_sgd(params, n_experts, d.blocks, n_pert, probe_kind, lr, seed, step, coef_ws,
                        st);
  if (e == cudaSuccess) e = canary_check(w.r, workspace, status, st);
  return cuda_status(e);
}

}  // namespace

extern "C" {

int64_t soma_body_param_count(soma_body_dims d) {
  if (!body_dims_ok(d)) return -1;
  return body_param_count(d.width, d.blocks);
}

size_t soma_body_workspace_bytes(soma_body_dims d, int n_experts, int n_pert, int batch,
                                 int seq_len) {
  if (!body_dims_ok(d) || !body_sizes_ok(n_experts, n_pert, batch, seq_len)) return 0;
  return plan_body(n_experts, n_pert, 2, batch).total;  // >= the eval's
}

int soma_body_spsa_estimate(const float* params, int n_experts, soma_body_dims d,
                            const float* head, int n_pert, int probe_kind, float eps,
                            uint64_t seed, uint64_t step, const uint8_t* byte_batch, int batch,
                            int seq_len, float* losses_out, float* coef_out, void* workspace,
                            size_t workspace_bytes, void* stream) {
  // the sweep only reads params
  return body_forward(const_cast<float*>(params), n_experts, d, head, n_pert, probe_kind, eps,
                      0.f, false, seed, step, byte_batch, batch, seq_len, losses_out, coef_out,
                      workspace, workspace_bytes, stream);
}

int soma_body_spsa_step(float* params, int n_experts, soma_body_dims d, const float* head,
                        int n_pert, int probe_kind, float eps, float lr, uint64_t seed,
                        uint64_t step, const uint8_t* byte_batch, int batch, int seq_len,
                        float* losses_out, float* coef_out, void* workspace,
                        size_t workspace_bytes, void* stream) {
  return body_forward(params, n_experts, d, head, n_pert, probe_kind, eps, lr, true, seed, step,
                      byte_batch, batch, seq_len, losses_out, coef_out, workspace,
                      workspace_bytes, stream);
}

int soma_body_eval_loss(const float* params, int n_experts, soma_body_dims d, const float* head,
                        const uint8_t* byte_batch, int batch, int seq_len, float* loss_out,
                        void* workspace, size_t workspace_bytes, void* stream) {
  if (!body_dims_ok(d)) return SOMA_ERR_UNSUPPORTED;
  if (!params || !head || !byte_batch || !loss_out || !aligned16(params) || !aligned16(head) ||
      !body_sizes_ok(n_experts, 1, batch, seq_len))
    return SOMA_ERR_INVALID_ARG;
  const BodyWs w = plan_body(n_experts, 1, 1, batch);
  if (!workspace || !aligned16(workspace) || workspace_bytes < w.total) return SOMA_ERR_WORKSPACE;
  int* status = status_ptr();
  if (!status) return SOMA_ERR_CUDA;
  cudaStream_t st = (cudaStream_t)stream;
  double* partial = reinterpret_cast<double*>(static_cast<uint8_t*>(workspace) + w.r.off[0]);
  cudaError_t e = canary_fill(w.r, workspace, st);
  if (e == cudaSuccess)
    e = launch_body_tc(params, head, byte_batch, n_experts, d.blocks, 1, 1, batch, seq_len, 0.f,
                       0, 0, 0, partial, status, st);
  if (e == cudaSuccess)
    e = launch_body_reduce(partial, n_experts, 1, batch, seq_len, 0.f, loss_out, nullptr,
                           nullptr, status, st);
  if (e == cudaSuccess) e = canary_check(w.r, workspace, status, st);
  return cuda_status(e);
}

int soma_body_adam_update(float* params, float* m, float* v, int n_experts, soma_body_dims d,
                          int n_pert, int probe_kind, uint64_t seed, const uint64_t* steps,
                          int n_acc, const float* coef, soma_adam_config cfg, void* stream) {
  if (!body_dims_ok(d)) return SOMA_ERR_UNSUPPORTED;
  if (!params || !m || !v || !coef || !steps || !aligned16(params) || !aligned16(m) ||
      !aligned16(v) || n_experts < 1 || n_pert < 1 || n_pert > kMaxPert || n_acc < 1 ||
      n_acc > SOMA_MAX_ACCUM || (probe_kind != SOMA_PROBE_DENSE && probe_kind != SOMA_PROBE_SPARSE))
    return SOMA_ERR_INVALID_ARG;
  if (!std::isfinite(cfg.lr) || !(cfg.beta1 >= 0.f && cfg.beta1 < 1.f) ||
      !(cfg.beta2 >= 0.f && cfg.beta2 < 1.f) || !(cfg.delta > 0.f) || !std::isfinite(cfg.delta) ||
      !(cfg.weight_decay >= 0.f) || !std::isfinite(cfg.weight_decay) || cfg.t < 1)
    return SOMA_ERR_INVALID_ARG;
  AdamSteps st;
  st.n_acc = n_acc;
  for (int a = 0; a < n_acc; ++a) st.step[a] = steps[a];
  AdamArgs h;
  h.lr = cfg.lr;
  h.b1 = cfg.beta1;
  h.b2 = cfg.beta2;
  h.delta = cfg.delta;
  h.wd = cfg.weight_decay;
  h.inv_bc1 = (float)(1.0 / (1.0 - std::pow((double)cfg.beta1, (double)cfg.t)));
  h.inv_bc2 = (float)(1.0 / (1.0 - std::pow((double)cfg.beta2, (double)cfg.t)));
  return cuda_status(launch_body_adam(params, m, v, n_experts, d.blocks, n_pert, probe_kind, seed,
                                      st, coef, h, (cudaStream_t)stream));
}

int soma_debug_body_probe(uint64_t seed, uint64_t step, int expert, int pert, soma_body_dims d,
                          int probe_kind, int64_t p0, int64_t count, int8_t* z_out,
                          void* stream) {
  if (!body_dims_ok(d)) return SOMA_ERR_UNSUPPORTED;
  if (!z_out || count < 0 || p0 < 0 || expert < 0 || pert < 0 ||
      (probe_kind != SOMA_PROBE_DENSE && probe_kind != SOMA_PROBE_SPARSE) ||
      p0 + count > ((int64_t)1 << 30))
    return SOMA_ERR_INVALID_ARG;
  if (count == 0) return SOMA_OK;
  return cuda_status(launch_debug_body_probe(seed, step, expert, pert, d.blocks, probe_kind, p0,
                                             count, z_out, (cudaStream_t)stream));
}

}  // extern "C"
