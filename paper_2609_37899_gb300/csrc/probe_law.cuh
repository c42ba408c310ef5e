// probe_law.cuh -- the probe of a run of 32 parameters under either probe
// law, shared by the update kernels of both expert models.
#pragma once

#include <cstdint>

#include "soma_device.cuh"

namespace soma {

// Sign and activity words of the 32 coordinates 32q .. 32q + 31 in natural
// order (bit j <=> coordinate 32q + j): neg bit set <=> z = -1, act bit
// clear <=> z = 0.  Dense probes are active everywhere.  Sparse probes (App.
// E) take the activity stream on every coordinate below `dense_from` and keep
// the coordinates from `dense_from` on active: the expert body's
// normalisation gains.  The LSTM expert passes dense_from = P (no gains).
__host__ __device__ __forceinline__ void probe_law_words(const ProbeKey& pk, int q, int sparse,
                                                         int64_t dense_from, uint32_t& neg,
                                                         uint32_t& act) {
  neg = raw_to_natural(probe_raw_word(pk, (uint32_t)q));
  act = 0xFFFFFFFFu;
  if (sparse) {
    act = raw_to_natural(probe_raw_word(activity_key(pk), (uint32_t)q));
    const int64_t from = dense_from - 32LL * q;  // first dense coordinate inside the run
    if (from <= 0)
      act = 0xFFFFFFFFu;
    else if (from < 32)
      act |= 0xFFFFFFFFu << from;
  }
}

// The activity word of run q under the probe law, from its raw activity
// word (sparse probes only): coordinates from dense_from on stay active.
__host__ __device__ __forceinline__ uint32_t probe_law_act(uint32_t act_raw, int64_t q,
                                                           int64_t dense_from) {
  uint32_t act = raw_to_natural(act_raw);
  const int64_t from = dense_from - 32LL * q;  // first dense coordinate inside the run
  if (from <= 0)
    act = 0xFFFFFFFFu;
  else if (from < 32)
    act |= 0xFFFFFFFFu << from;
  return act;
}

}  // namespace soma
