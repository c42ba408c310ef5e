// body_device.cuh -- sizes and the probe law of the paper's expert body
// (Sec. "Model size"; App. E), shared by body.cu and the C ABI.
#pragma once

#include <cstdint>

#include "probe_law.cuh"
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

// The body's probe law: sparse on the weights, dense on the gains.
__host__ __device__ __forceinline__ void body_probe_words(const ProbeKey& pk, int q, int sparse,
                                                          int64_t goff, uint32_t& neg,
                                                          uint32_t& act) {
  probe_law_words(pk, q, sparse, goff, neg, act);
}

}  // namespace soma
