// body_device.cuh -- sizes and the probe law of the paper's expert body
// (Sec. "Model size"; App. E), shared by body.cu and the C ABI.
#pragma once

#include <cstdint>

#include "soma_device.cuh"

namespace soma {

constexpr int kBodyWidth = 32;     // d_t = d_E of the width-32 ensembles
constexpr int kBodyMaxBlocks = 2;  // D
constexpr int kBodyRows = 16;      // sequences of one CTA of the forward sweep

// M_body = 16 D d^2 + (2D + 1) d: per block W_ih, W_hh, W_1 [4d][d] and
// W_2 [d][4d]; then the gains ga_k, gb_k of every block and the final gf.
__host__ __device__ inline int64_t body_param_count(int d, int D) {
  return 16LL * D * d * d + (2LL * D + 1) * d;
}

// First normalisation-gain coordinate: every coordinate from here on is a gain.
__host__ __device__ inline int64_t body_gain_offset(int d, int D) { return 16LL * D * d * d; }

// Sign and activity words of the 32 coordinates 32q .. 32q + 31 in natural
// order (bit j <=> coordinate 32q + j): neg bit set <=> z = -1, act bit
// clear <=> z = 0.  Dense probes are active everywhere.  The sparse law
// (App. E) takes the activity stream on weights and keeps every gain active.
__host__ __device__ __forceinline__ void body_probe_words(const ProbeKey& pk, int q, int sparse,
                                                          int64_t goff, uint32_t& neg,
                                                          uint32_t& act) {
  neg = raw_to_natural(probe_raw_word(pk, (uint32_t)q));
  act = 0xFFFFFFFFu;
  if (sparse) {
    act = raw_to_natural(probe_raw_word(activity_key(pk), (uint32_t)q));
    const int64_t from = goff - 32LL * q;  // offset of the first gain inside the run
    if (from <= 0)
      act = 0xFFFFFFFFu;
    else if (from < 32)
      act |= 0xFFFFFFFFu << from;
  }
}

}  // namespace soma
