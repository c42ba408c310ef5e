// trace.cu -- optional per-kernel-class timing with CUDA events recorded on
// the launching stream around every kernel of soma_spsa_step / soma_eval_loss
// (soma_trace_enable / soma_trace_read in include/soma_api.h).
#include <mutex>
#include <vector>

#include "soma_api.h"
#include "soma_launch.h"

namespace soma {

namespace {

struct Record {
  int kind;
  cudaEvent_t start, stop;
};

std::mutex g_mu;
bool g_enabled = false;
std::vector<Record> g_pending;
std::vector<cudaEvent_t> g_pool;
Record g_open = {-1, nullptr, nullptr};

cudaEvent_t take_event() {
  if (!g_pool.empty()) {
    cudaEvent_t e = g_pool.back();
    g_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

}  // namespace

void trace_begin(int kind, cudaStream_t stream) {
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_enabled) return;
  g_open.kind = kind;
  g_open.start = take_event();
  g_open.stop = take_event();
  if (g_open.start) cudaEventRecord(g_open.start, stream);
}

void trace_end(int kind, cudaStream_t stream) {
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_enabled || g_open.kind != kind || !g_open.start || !g_open.stop) return;
  cudaEventRecord(g_open.stop, stream);
  g_pending.push_back(g_open);
  g_open.kind = -1;
}

}  // namespace soma

using namespace soma;

extern "C" {

int soma_trace_enable(int enable) {
  std::lock_guard<std::mutex> lk(g_mu);
  g_enabled = enable != 0;
  return SOMA_OK;
}

int soma_trace_read(soma_kernel_times* out, int reset) {
  if (!out) return SOMA_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(g_mu);
  for (int k = 0; k < SOMA_TRACE_KINDS; ++k) {
    out->ms[k] = 0.0;
    out->launches[k] = 0;
  }
  int rc = SOMA_OK;
  for (const Record& r : g_pending) {
    if (cudaEventSynchronize(r.stop) != cudaSuccess) {
      rc = SOMA_ERR_CUDA;
      continue;
    }
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, r.start, r.stop) != cudaSuccess) {
      rc = SOMA_ERR_CUDA;
      continue;
    }
    if (r.kind >= 0 && r.kind < SOMA_TRACE_KINDS) {
      out->ms[r.kind] += ms;
      out->launches[r.kind] += 1;
    }
  }
  if (reset) {
    for (const Record& r : g_pending) {
      g_pool.push_back(r.start);
      g_pool.push_back(r.stop);
    }
    g_pending.clear();
  }
  return rc;
}

}  // extern "C"
