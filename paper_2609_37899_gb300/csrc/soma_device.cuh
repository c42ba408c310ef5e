// soma_device.cuh -- device helpers shared by the libsoma kernels: the
// Philox4x32-10 probe generator, the parameter layout of one expert and the
// argument blocks the host passes to the kernels.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace soma {

constexpr int kVocab = 256;

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of two
// 32x32 -> 64-bit products whose high halves are xor-ed into the other two
// words with the round key; the key advances by the Weyl constants
// (golden ratio, sqrt(3) - 1) after each round.
// ---------------------------------------------------------------------------
__host__ __device__ __forceinline__ uint32_t mul_hi32(uint32_t a, uint32_t b) {
#ifdef __CUDA_ARCH__
  return __umulhi(a, b);
#else
  return (uint32_t)(((uint64_t)a * (uint64_t)b) >> 32);
#endif
}

__host__ __device__ __forceinline__ uint4 philox4x32_10(uint4 ctr, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo_a = 0xD2511F53u * ctr.x;
    const uint32_t hi_a = mul_hi32(0xD2511F53u, ctr.x);
    const uint32_t lo_b = 0xCD9E8D57u * ctr.z;
    const uint32_t hi_b = mul_hi32(0xCD9E8D57u, ctr.z);
    ctr = make_uint4(hi_b ^ ctr.y ^ k0, lo_b, hi_a ^ ctr.w ^ k1, lo_a);
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return ctr;
}

__host__ __device__ __forceinline__ uint32_t word_of(const uint4& w, int j) {
  return j == 0 ? w.x : (j == 1 ? w.y : (j == 2 ? w.z : w.w));
}

// Identity of one probe stream: z_{expert,probe} at update `step`.
struct ProbeKey {
  uint32_t k0, k1;   // seed halves
  uint32_t step;     // low 32 bits of the update counter
  uint32_t expert;   // counter word 3
  uint32_t probe;    // counter word 1
};

__host__ __device__ __forceinline__ ProbeKey make_probe_key(uint64_t seed, uint64_t step,
                                                             uint32_t expert, uint32_t probe) {
  ProbeKey k;
  k.k0 = (uint32_t)(seed & 0xffffffffu);
  k.k1 = (uint32_t)(seed >> 32);
  k.step = (uint32_t)(step & 0xffffffffu);
  k.expert = expert;
  k.probe = probe;
  return k;
}

// The 128 probe bits of parameter block `blk` (parameters 128*blk .. +127).
__host__ __device__ __forceinline__ uint4 probe_block(const ProbeKey& k, uint32_t blk) {
  return philox4x32_10(make_uint4(blk, k.probe, k.step, k.expert), k.k0, k.k1);
}

// Raw probe word of the 32-parameter run w (parameters 32w .. 32w+31): word
// (w & 3) of the Philox block w >> 2.  Inside a run, parameter 32w + o reads
// raw bit (o >> 1) + 16 (o & 1): even offsets take the low half in order, odd
// offsets the high half.
__host__ __device__ __forceinline__ uint32_t probe_raw_word(const ProbeKey& k, uint32_t w) {
  return word_of(probe_block(k, w >> 2), (int)(w & 3));
}

__host__ __device__ __forceinline__ uint32_t spread16(uint32_t x) {
  x &= 0xFFFFu;
  x = (x | (x << 8)) & 0x00FF00FFu;
  x = (x | (x << 4)) & 0x0F0F0F0Fu;
  x = (x | (x << 2)) & 0x33333333u;
  x = (x | (x << 1)) & 0x55555555u;
  return x;
}

// Raw word -> natural order (bit o <=> parameter 32w + o).
__host__ __device__ __forceinline__ uint32_t raw_to_natural(uint32_t raw) {
  return spread16(raw) | (spread16(raw >> 16) << 1);
}

// Bits of z for the 32 consecutive parameters p .. p+31 in natural order:
// bit j set <=> z[p+j] = -1.  One Philox call when p is 32-aligned, at most
// two otherwise.
__host__ __device__ __forceinline__ uint32_t probe_bits32(const ProbeKey& k, int64_t p) {
  const uint32_t w = (uint32_t)(p >> 5);
  const int sh = (int)(p & 31);
  const uint32_t lo = raw_to_natural(probe_raw_word(k, w));
  if (sh == 0) return lo;
  const uint32_t hi = raw_to_natural(probe_raw_word(k, w + 1));
  return (lo >> sh) | (hi << (32 - sh));
}

// Raw bit position of offset o (0..31) inside a run.
__host__ __device__ constexpr int raw_bit(int o) { return (o >> 1) + 16 * (o & 1); }

// Sparse probes (App. E: a coordinate is 0 with probability 1/2, else -1 or
// +1) take a second bit per coordinate: the activity bit, read with the same
// map from the blocks whose counter word 1 is the probe index with its top
// bit set.  z = active ? 1 - 2 * sign bit : 0, so a nonzero sparse
// coordinate equals the dense probe's coordinate.
__host__ __device__ __forceinline__ ProbeKey activity_key(ProbeKey k) {
  k.probe |= 0x80000000u;
  return k;
}

// Sign and activity bits of the 32 parameters p .. p+31 (natural order).
struct ProbeBits {
  uint32_t neg, act;
};

__host__ __device__ __forceinline__ ProbeBits probe_bits(const ProbeKey& k, int64_t p,
                                                         bool sparse) {
  ProbeBits b;
  b.neg = probe_bits32(k, p);
  b.act = sparse ? probe_bits32(activity_key(k), p) : 0xFFFFFFFFu;
  return b;
}

// w + s*eps*z for a z bit: the perturbed parameter in fp32.
__host__ __device__ __forceinline__ float perturb(float w, uint32_t bit, float se) {
  return w + (bit ? -se : se);
}

// The same for a probe coordinate with sign bit `neg` and activity bit `act`.
__host__ __device__ __forceinline__ float perturb(float w, uint32_t neg, uint32_t act, float se) {
  return act ? w + (neg ? -se : se) : w;
}

// eps z of one coordinate.
__host__ __device__ __forceinline__ float eps_z(uint32_t neg, uint32_t act, float eps) {
  return act ? (neg ? -eps : eps) : 0.f;
}

// ---------------------------------------------------------------------------
// Parameter layout of one expert: Emb[V][E], W_ih[4H][E], W_hh[4H][H],
// b[4H], W_out[V][H], b_out[V].
// ---------------------------------------------------------------------------
struct Layout {
  int E, H;
  int64_t emb, w_ih, w_hh, b, w_out, b_out, P;
};

__host__ __device__ inline Layout make_layout(int E, int H) {
  Layout L;
  L.E = E;
  L.H = H;
  L.emb = 0;
  L.w_ih = L.emb + (int64_t)kVocab * E;
  L.w_hh = L.w_ih + 4LL * H * E;
  L.b = L.w_hh + 4LL * H * H;
  L.w_out = L.b + 4LL * H;
  L.b_out = L.w_out + (int64_t)kVocab * H;
  L.P = L.b_out + kVocab;
  return L;
}

// ---------------------------------------------------------------------------
// One forward sweep over (expert, probe, sign) "lanes".  A lane is one
// perturbed copy of one expert: lane = (e * n_pert + i) * n_sign + s, with
// sign +1 for s = 0 and -1 for s = 1.  eval_loss is the sweep with
// n_pert = n_sign = 1 and eps = 0.
// ---------------------------------------------------------------------------
struct Sweep {
  const float* params;     // [N][P]
  const uint8_t* bytes;    // [N][B][T+1]
  Layout lay;
  int n_experts, n_pert, n_sign;
  int B, T;
  float eps;
  int sparse;              // probe kind: 0 dense Rademacher, 1 sparse (App. E)
  int batch_per_probe;     // 0: bytes [N][B_mem][T+1] shared by every probe (Sec. 4);
                           // 1: bytes [N][n_pert][B_mem][T+1], one batch per probe (App. D)
  int b0, B_mem;           // the sweep covers sequences b0 .. b0 + B - 1 of each batch of
                           // B_mem sequences (a batch of more than 64 runs in chunks)
  uint64_t seed, step;
  __host__ __device__ int lanes() const { return n_experts * n_pert * n_sign; }
};

// Offset of the first byte of sequence b (of the sweep) seen by probe i of
// expert e.
__host__ __device__ __forceinline__ int64_t seq_offset(const Sweep& s, int e, int i, int b) {
  const int64_t blk = s.batch_per_probe ? (int64_t)e * s.n_pert + i : (int64_t)e;
  return (blk * s.B_mem + s.b0 + b) * (int64_t)(s.T + 1);
}

__host__ __device__ __forceinline__ void lane_parts(const Sweep& s, int lane, int& e, int& i,
                                                    float& se) {
  const int sgn = lane % s.n_sign;
  const int ei = lane / s.n_sign;
  i = ei % s.n_pert;
  e = ei / s.n_pert;
  se = sgn == 0 ? s.eps : -s.eps;
}

// Device status codes (mirror soma_status).
constexpr int kStatusNonFinite = 6;
constexpr int kStatusTimeout = 5;

}  // namespace soma
