/*
 * soma_api.h -- C ABI of libsoma.so: the SPSA training step of N independent
 * byte-level LSTM experts on one GPU (SOMA, "Scaling Zero-Order Pretraining
 * through Model Sharding").
 *
 * The library computes, for every expert e and probe i = 0..n_pert-1,
 *   L+_{e,i} = L_e(theta_e + eps z_{e,i}),  L-_{e,i} = L_e(theta_e - eps z_{e,i})
 * on one batch shared by every probe and both signs (Sec. 4, Eq. main-spsa),
 * the coefficients c_{e,i} = (L+ - L-) / (2 eps), and the update
 *   theta_e <- theta_e - lr * (1/n_pert) * sum_i c_{e,i} z_{e,i}
 * (Eq. main-spsa inside the plain-SGD form of Eq. localspsa).  L is the mean
 * next-byte cross entropy in nats/byte over all B*T targets (Table
 * experimental-setup, "Evaluation protocol"), with the LSTM state reset to
 * zero for every sequence.  Experts never interact: each has its own batch,
 * probes and loss (Eq. separable-training-objective).
 *
 * Model of one expert (App. C, one LSTM layer instead of the paper's two
 * residual blocks; every parameter is perturbed).  Flat fp32 parameter
 * vector of P = V*E + 4H*E + 4H*H + 4H + V*H + V entries, in this order:
 *   Emb[V][E], W_ih[4H][E], W_hh[4H][H], b[4H], W_out[V][H], b_out[V]
 * row-major, gate blocks of W_ih, W_hh and b in the order i, f, g, o.
 *   x_t = Emb[byte_t];  a = W_ih x_t + W_hh h_{t-1} + b
 *   i,f,o = sigmoid(a_i,a_f,a_o); g = tanh(a_g); c_t = f c_{t-1} + i g;
 *   h_t = o tanh(c_t);  logits = W_out h_t + b_out;
 *   nll_t = logsumexp(logits) - logits[byte_{t+1}].
 *
 * Probes (dense Rademacher, Sec. 5 / App. F): z_{e,i}[p] in {-1,+1} for flat
 * parameter index p, regenerated from Philox4x32-10 (Salmon et al., SC'11):
 *   key = (seed & 0xffffffff, seed >> 32)
 *   counter = (p >> 7, i, step & 0xffffffff, e)
 *   o = p & 31;  bit = bit (o >> 1) + 16 (o & 1) of output word ((p & 127) >> 5)
 *   z = 1 - 2 bit   (even offsets of a 32-parameter run read the low half-word,
 *                    odd offsets the high half-word).
 * Sparse probes (App. E, the paper's training probes; soma_spsa_estimate and
 * soma_adam_update): a second, activity bit per coordinate, read with the same
 * map from the blocks whose counter word 1 is i | 0x80000000;
 *   z = activity ? 1 - 2 bit : 0,
 * so a coordinate is 0 with probability 1/2 and -1 or +1 with probability 1/4.
 * No probe is ever stored.
 *
 * Conventions for every entry point:
 *  - Every buffer is owned by the caller.  Device pointers must point to
 *    memory of the current device and be 16-byte aligned; the library never
 *    allocates or frees.  Scratch memory is the caller's workspace, sized by
 *    soma_workspace_bytes().
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Calls enqueue work on it and return without synchronising.
 *  - Host-side argument errors return a soma_status code before anything is
 *    enqueued.  Errors found on the device (a non-finite loss) are recorded
 *    in a per-device status word read by soma_get_status().
 *  - The library keeps no other state: no handle, no global RNG.  Calls on
 *    different streams may run concurrently if their buffers are disjoint
 *    (they share only the per-device status word).
 */
#ifndef SOMA_API_H
#define SOMA_API_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Model sizes.  vocab must be 256 (one token per byte, App. C). */
typedef struct soma_dims {
  int32_t vocab;  /* V = 256 */
  int32_t embed;  /* E, 1..1024 */
  int32_t hidden; /* H, 1..4096 */
} soma_dims;

typedef enum soma_status {
  SOMA_OK = 0,
  SOMA_ERR_INVALID_ARG = 1, /* null or misaligned pointer, bad count/size/eps/lr */
  SOMA_ERR_UNSUPPORTED = 2, /* dims outside the supported range */
  SOMA_ERR_WORKSPACE = 3,   /* workspace NULL or smaller than soma_workspace_bytes() */
  SOMA_ERR_CUDA = 4,        /* a CUDA launch or runtime call failed */
  SOMA_ERR_TIMEOUT = 5,     /* a bounded device-side wait gave up */
  SOMA_ERR_NONFINITE = 6,   /* a loss or coefficient was NaN or infinite */
  SOMA_ERR_BOUNDS = 7       /* an index check of the checked build failed (never raised
                               by the default build; see soma_checked_build) */
} soma_status;

/* Number of parameters P of one expert (layout above); -1 if d is invalid. */
int64_t soma_param_count(soma_dims d);

/* Bytes of workspace that soma_spsa_step() and soma_eval_loss() need for
 * these sizes (the larger of the two); 0 if the sizes are invalid. */
size_t soma_workspace_bytes(soma_dims d, int n_experts, int n_pert, int batch, int seq_len);

/* Deterministic initialisation of params [n_experts][P] (device, fp32) from
 * Philox4x32-10 in a domain disjoint from the probes (counter word 3 has its
 * top bit set).  std > 0: every parameter ~ N(0, std).  std == 0: Emb ~
 * N(0, 0.1), W_ih and W_hh ~ N(0, 1/sqrt(E+H)), W_out ~ N(0, 1/sqrt(H)),
 * biases 0.  Normals by the Box-Muller transform.  std < 0 is invalid. */
int soma_init_experts(float* params, int n_experts, soma_dims d, uint64_t seed, float std,
                      void* stream);

/* One SPSA step for every expert (Eq. main-spsa).
 *   params      device fp32 [n_experts][P]; updated in place.
 *   n_pert      probes per expert, 1..12288.
 *   eps, lr     probe radius (finite, >= 0) and learning rate (finite).
 *               eps == 0 gives L+ = L- = L(theta), every coefficient 0 and
 *               params unchanged; lr == 0 leaves params bit-unchanged.
 *   seed, step  select the probes (see the header comment); the library
 *               does not advance `step`.
 *   byte_batch  device uint8 [n_experts][batch][seq_len + 1]: expert e's
 *               sequences, shared by all its probes and both signs.
 *   losses_out  device fp32 [n_experts][n_pert][2]: (L+, L-) in nats/byte.
 *   coef_out    device fp32 [n_experts][n_pert] (L+ - L-)/(2 eps), or NULL.
 *   workspace   device scratch of >= soma_workspace_bytes() bytes.
 * Returns SOMA_OK once the work is enqueued. */
int soma_spsa_step(float* params, int n_experts, soma_dims d, int n_pert, float eps, float lr,
                   uint64_t seed, uint64_t step, const uint8_t* byte_batch, int batch,
                   int seq_len, float* losses_out, float* coef_out, void* workspace,
                   size_t workspace_bytes, void* stream);

/* Unperturbed mean loss L(theta_e) in nats/byte for every expert.
 *   params [n_experts][P] and byte_batch [n_experts][batch][seq_len + 1] as
 *   above; loss_out device fp32 [n_experts]. */
int soma_eval_loss(const float* params, int n_experts, soma_dims d, const uint8_t* byte_batch,
                   int batch, int seq_len, float* loss_out, void* workspace,
                   size_t workspace_bytes, void* stream);

/* The update alone, for given coefficients (the last part of Eq. main-spsa):
 *   params[e] -= lr * (1/n_pert) * sum_i coef[e][i] z_{e,i}.
 *   coef: device fp32 [n_experts][n_pert].  No workspace. */
int soma_spsa_update(float* params, int n_experts, soma_dims d, int n_pert, float lr,
                     uint64_t seed, uint64_t step, const float* coef, void* stream);

/* ---- The paper's optimizer step (App. E, Eq. localspsa) ----------------
 * One update averages A accumulation batches, each with its own batch and
 * probes (step counter steps[a]):
 *   ghat  = (1/A) sum_a (1/n_pert) sum_i c_{a,e,i} z^{(a)}_{e,i}
 *   g     = ghat + weight_decay * theta      (coupled decay, before the moments)
 *   m     = beta1 m + (1 - beta1) g,  v = beta2 v + (1 - beta2) g^2
 *   theta = theta - lr * (m / (1 - beta1^t)) / (sqrt(v / (1 - beta2^t)) + delta)
 * A caller runs soma_spsa_estimate once per accumulation batch (writing its
 * coefficients into row a of a [A][n_experts][n_pert] buffer), then
 * soma_adam_update once. */
typedef enum soma_probe_kind {
  SOMA_PROBE_DENSE = 0,  /* Rademacher +-1 (Sec. 5, App. F) */
  SOMA_PROBE_SPARSE = 1  /* 0 w.p. 1/2, -1 or +1 w.p. 1/4 each (App. E) */
} soma_probe_kind;

#define SOMA_MAX_ACCUM 64

typedef struct soma_adam_config {
  float lr;           /* eta_t, finite */
  float beta1;        /* in [0, 1) */
  float beta2;        /* in [0, 1) */
  float delta;        /* delta_Adam > 0 (the paper: 1e-8) */
  float weight_decay; /* lambda >= 0, coupled (the paper: 1e-4) */
  int32_t t;          /* 1-based update count; m = v = 0 before update 1 */
} soma_adam_config;

/* Losses and coefficients of one accumulation batch; params are not changed.
 * Arguments as soma_spsa_step, plus probe_kind (soma_probe_kind); coef_out is
 * required.  Same workspace size as soma_spsa_step. */
int soma_spsa_estimate(const float* params, int n_experts, soma_dims d, int n_pert,
                       int probe_kind, float eps, uint64_t seed, uint64_t step,
                       const uint8_t* byte_batch, int batch, int seq_len, float* losses_out,
                       float* coef_out, void* workspace, size_t workspace_bytes, void* stream);

/* Options of soma_spsa_estimate_opts: the probe kind and the two variants
 * the paper measures its mechanism with (App. D).
 *   batch_per_probe = 0  byte_batch [n_experts][batch][seq_len + 1], one batch
 *                        per expert shared by every probe (Sec. 4);
 *                   = 1  byte_batch [n_experts][n_pert][batch][seq_len + 1],
 *                        an independently drawn batch per probe (both signs
 *                        of a probe share it).
 *   summed_loss     = 0  each expert's own loss (SOMA);
 *                   = 1  the control arm that sums the N experts' losses
 *                        before each finite difference: coef_out[e][i] =
 *                        sum_e' (L+_{e',i} - L-_{e',i}) / (2 eps) for every e
 *                        (losses_out still holds each expert's L+, L-). */
typedef struct soma_estimate_options {
  int32_t probe_kind;
  int32_t batch_per_probe;
  int32_t summed_loss;
} soma_estimate_options;

int soma_spsa_estimate_opts(const float* params, int n_experts, soma_dims d, int n_pert,
                            const soma_estimate_options* opts, float eps, uint64_t seed,
                            uint64_t step, const uint8_t* byte_batch, int batch, int seq_len,
                            float* losses_out, float* coef_out, void* workspace,
                            size_t workspace_bytes, void* stream);

/* The Adam update of Eq. localspsa from the coefficients of n_acc
 * accumulation batches.
 *   params, m, v  device fp32 [n_experts][P]; updated in place (m, v start at
 *                 0 and are owned and kept by the caller between updates).
 *   steps         HOST uint64 [n_acc]: the step counter each batch's probes
 *                 were drawn with; 1 <= n_acc <= SOMA_MAX_ACCUM.
 *   coef          device fp32 [n_acc][n_experts][n_pert].
 * An expert with a non-finite coefficient is left unchanged (params, m, v).
 * No workspace. */
int soma_adam_update(float* params, float* m, float* v, int n_experts, soma_dims d, int n_pert,
                     int probe_kind, uint64_t seed, const uint64_t* steps, int n_acc,
                     const float* coef, soma_adam_config cfg, void* stream);

/* ---- Routed inference (Sec. 3, Eq. main-mixture) ----------------------
 * Request r (teacher-forced, LSTM state reset to zero) is scored by the k
 * experts routes[r][0..k-1]; its prediction averages their probabilities,
 *   p(y | x_<t) = (1/k) sum_j p_{routes[r][j]}(y | x_<t),
 * and nll_out[r][t - t0] = -log p(byte_{t+1} | bytes_<=t) for t0 <= t < seq_len.
 * The routes come from the caller (the paper's router is a fitted tf-idf
 * model); an expert may be listed more than once.  Requests are grouped by
 * expert and each expert runs on its group in sweeps of up to 64 sequences.
 *   params    device fp32 [n_experts][P]
 *   requests  device uint8 [R][seq_len + 1]
 *   routes    HOST int32 [R][k], entries in [0, n_experts); 1 <= k <= 16
 *   nll_out   device fp32 [R][seq_len - t0]; 0 <= t0 < seq_len
 * The workspace size depends on the routing (the largest group), hence the
 * routes argument of soma_mixture_workspace_bytes (0 if invalid). */
size_t soma_mixture_workspace_bytes(soma_dims d, int n_experts, const int32_t* routes, int R,
                                    int k, int seq_len);
int soma_mixture_nll(const float* params, int n_experts, soma_dims d, const uint8_t* requests,
                     int R, int seq_len, const int32_t* routes, int k, int t0, float* nll_out,
                     void* workspace, size_t workspace_bytes, void* stream);

/* Synchronises `stream`, then returns and clears the current device's status
 * word (SOMA_OK if no device-side error was recorded since the last call).
 * Returns SOMA_ERR_CUDA if the synchronisation itself failed. */
int soma_get_status(void* stream);

/* Static, human-readable name of a status code. */
const char* soma_status_string(int code);

/* Tracing.  While enabled, every kernel that soma_spsa_step, soma_eval_loss,
 * soma_spsa_estimate, soma_spsa_update and soma_adam_update launch is bracketed by two CUDA events recorded on the
 * caller's stream; soma_trace_read() waits for the recorded events and sums
 * device time and launch counts per kernel class.  Tracing is process-wide
 * and off by default; events are created on first use and reused. */
enum {
  SOMA_TRACE_GATE = 0,   /* recurrent gate GEMM + fused cell update and head (one launch per sweep) */
  SOMA_TRACE_HEAD = 1,   /* output head + log-softmax + NLL */
  SOMA_TRACE_REDUCE = 2, /* loss and coefficient reduction */
  SOMA_TRACE_UPDATE = 3, /* Philox-regenerating parameter update */
  SOMA_TRACE_PREP = 4,   /* fp16 weight tiles, probe-word tables, embedding operands */
  SOMA_TRACE_KINDS = 5
};
typedef struct soma_kernel_times {
  double ms[SOMA_TRACE_KINDS];       /* summed device time per class */
  int64_t launches[SOMA_TRACE_KINDS];
} soma_kernel_times;
int soma_trace_enable(int enable);
/* reset != 0 also forgets the records that were read. */
int soma_trace_read(soma_kernel_times* out, int reset);

/* Test exports (bit-exactness of the generator the kernels use).
 * soma_debug_philox: out4[j] = Philox4x32-10(ctr4[j], key = seed halves) for
 *   j < count; ctr4 and out4 are device uint32 [count][4].
 * soma_debug_rademacher: z_out[q] = z_{expert,pert}[p0 + q] for q < count,
 *   device int8, using the same bit extraction the kernels use.
 * soma_debug_probe: the same for either probe kind (soma_probe_kind). */
int soma_debug_philox(uint64_t seed, const uint32_t* ctr4, uint32_t* out4, int count,
                      void* stream);
int soma_debug_rademacher(uint64_t seed, uint64_t step, int expert, int pert, int64_t p0,
                          int64_t count, int8_t* z_out, void* stream);
int soma_debug_probe(uint64_t seed, uint64_t step, int expert, int pert, int probe_kind,
                     int64_t p0, int64_t count, int8_t* z_out, void* stream);
/* soma_debug_wait_timeout: one kernel waits on a barrier that nothing
 *   completes.  Its bounded wait gives up after max_polls polls (1 ..
 *   2^22; each poll suspends for at most ~100 ns) and records
 *   SOMA_ERR_TIMEOUT in the status word, which soma_get_status() then
 *   returns; the context stays usable.  This is the path every kernel of the
 *   library takes when one of its waits runs out. */
int soma_debug_wait_timeout(uint32_t max_polls, void* stream);
/* soma_debug_tc_gemm: d[128][n] = a[128][k] * b[n][k]^T (fp16 inputs as
 *   uint16 bit patterns, row-major; fp32 output) through the same shared-
 *   memory descriptors, tcgen05.mma and tensor-memory read-back as the
 *   forward kernels.  16 <= n, k <= 256, both multiples of 16. */
int soma_debug_tc_gemm(const uint16_t* a, const uint16_t* b, float* d, int n, int k,
                       void* stream);

/* soma_debug_tc_gemm_ts: the same product with a staged in tensor memory
 *   (lane = row, each 32-bit column one k pair) and read by tcgen05.mma from
 *   there, the form in which the forward kernels feed their probe tiles Z
 *   (the A operand of the Z products of Sec. 4, Eq. main-spsa, in the
 *   mean/difference form).  Same arguments, limits and errors. */
int soma_debug_tc_gemm_ts(const uint16_t* a, const uint16_t* b, float* d, int n, int k,
                          void* stream);

/* The checked build.  The library built with -DSOMA_CHECKED
 * (libsoma_checked.so, `python -m paper_2609_37899_gb300.build --checked`)
 * guards the shared-memory offsets, tensor-memory columns and global indices
 * of its kernels with index checks, and surrounds every workspace region with
 * 256-byte canary words that it writes before a step and verifies after it.
 * A failed check records SOMA_ERR_BOUNDS in the status word and skips the
 * access (no trap, the context stays usable).  These are test aids with no
 * counterpart in the paper; the default build has none of the checks and no
 * canaries.
 *  - soma_checked_build: 1 in the checked build, 0 otherwise.
 *  - soma_debug_check_line: syncs `stream`, returns and clears the position
 *    of the first failed check (10000 * file id + source line; 90000 + gap
 *    index for a canary), 0 if none; -1 if the synchronisation failed.
 *  - soma_debug_check_fail: enqueues one check whose condition is false and
 *    that guards no access (the checked build's reporting path; a no-op in
 *    the default build). */
int soma_checked_build(void);
int soma_debug_check_line(void* stream);
int soma_debug_check_fail(void* stream);

/* SPSA step without a workspace argument, for callers that cannot allocate
 * device memory (a host runtime that only passes on buffers it was given, or
 * a loop that must not risk an allocation that blocks or fails).  The paper
 * has no counterpart; this is an interface convenience of this library.
 *
 * Same arguments and results as soma_spsa_step() minus the workspace: the
 * scratch is a fixed device array of SOMA_STATIC_WORKSPACE_BYTES inside the
 * library, which every GPU that loads the library keeps until the process
 * exits.  Sizes whose soma_workspace_bytes() exceed that return
 * SOMA_ERR_WORKSPACE before anything is enqueued.  No cudaMalloc, cudaFree
 * or other allocating routine is called (keep tracing off: it creates CUDA
 * events on first use).
 *  - The first call on each device looks up the array's device address with
 *    that device current; make that first call before any stream capture.
 *  - Every call shares the one array and the path writes each scratch word
 *    before it reads it, so nothing needs clearing between calls; two calls
 *    whose work overlaps on the GPU (different streams, or devices sharing
 *    nothing but this rule) race on the array and give wrong results. */
#define SOMA_STATIC_WORKSPACE_BYTES ((size_t)64 << 20)
int soma_spsa_step_static(float* params, int n_experts, soma_dims d, int n_pert, float eps,
                          float lr, uint64_t seed, uint64_t step, const uint8_t* byte_batch,
                          int batch, int seq_len, float* losses_out, float* coef_out,
                          void* stream);

/* ---- The paper's expert body (Sec. "Model size"; App. E) ---------------
 * The width-32 ensembles' expert: D pre-norm residual blocks of width d,
 *   u = LN(x) ga_k;  LSTM_k (bias-free, gates i, f, g, o; state reset per
 *   sequence) on u;  x += h_k;  v = LN(x) gb_k;  x += W_2^k GELU(W_1^k v)
 * (bias-free MLP of width 4d, exact erf GELU), starting from x = E[byte_t],
 * then y = LN(x) gf and logits = E y.  LN(x) = (x - mean) / sqrt(var + 1e-5)
 * with var the mean squared deviation.  E [256][d] is the frozen tied head:
 * shared by every expert, never perturbed.
 * Body parameters of one expert, M_body = 16 D d^2 + (2D + 1) d floats:
 *   per block k: W_ih [4d][d], W_hh [4d][d], W_1 [4d][d], W_2 [d][4d];
 *   then ga_0, gb_0, ..., ga_{D-1}, gb_{D-1}, gf [d] each.
 * Probes (App. E): SOMA_PROBE_DENSE is the dense sign on every coordinate.
 * SOMA_PROBE_SPARSE is the paper's training law: every gain takes the dense
 * sign, every weight the sparse probe (same Philox stream and bit map as
 * above, keyed by the flat body coordinate).
 * Supported: vocab 256, width 32, blocks 1 or 2; else SOMA_ERR_UNSUPPORTED.
 * The forward runs on the tensor cores: one CTA per (expert, probe) pair and
 * chunk of up to 16 sequences, both signs in one mean/difference pass, fp16
 * operands split into hi + lo parts, fp32 accumulation and epilogues, losses
 * summed in fp64. */
typedef struct soma_body_dims {
  int32_t vocab;  /* must be 256 */
  int32_t width;  /* d = d_t = d_E */
  int32_t blocks; /* D */
} soma_body_dims;

/* M_body, or -1 for unsupported dims. */
int64_t soma_body_param_count(soma_body_dims d);

/* Workspace of soma_body_spsa_step / _estimate / _eval_loss (0 for invalid
 * sizes). */
size_t soma_body_workspace_bytes(soma_body_dims d, int n_experts, int n_pert, int batch,
                                 int seq_len);

/* Losses and coefficients of one batch; params are not changed.
 *   params      device fp32 [n_experts][M_body]
 *   head        device fp32 [256][d], the frozen tied matrix E
 *   byte_batch  device uint8 [n_experts][batch][seq_len + 1], shared by every
 *               probe and both signs of an expert
 *   losses_out  device fp32 [n_experts][n_pert][2] (L+, L-) or NULL
 *   coef_out    device fp32 [n_experts][n_pert]: (L+ - L-) / (2 eps)
 * eps == 0 gives L+ == L- == L(theta) and coefficients 0. */
int soma_body_spsa_estimate(const float* params, int n_experts, soma_body_dims d,
                            const float* head, int n_pert, int probe_kind, float eps,
                            uint64_t seed, uint64_t step, const uint8_t* byte_batch, int batch,
                            int seq_len, float* losses_out, float* coef_out, void* workspace,
                            size_t workspace_bytes, void* stream);

/* The estimate, then theta <- theta - lr (1/n_pert) sum_i c_i z_i with the
 * same probes (Eq. main-spsa); coef_out may be NULL. */
int soma_body_spsa_step(float* params, int n_experts, soma_body_dims d, const float* head,
                        int n_pert, int probe_kind, float eps, float lr, uint64_t seed,
                        uint64_t step, const uint8_t* byte_batch, int batch, int seq_len,
                        float* losses_out, float* coef_out, void* workspace,
                        size_t workspace_bytes, void* stream);

/* loss_out device fp32 [n_experts] = L(theta_e) on its batch. */
int soma_body_eval_loss(const float* params, int n_experts, soma_body_dims d, const float* head,
                        const uint8_t* byte_batch, int batch, int seq_len, float* loss_out,
                        void* workspace, size_t workspace_bytes, void* stream);

/* Eq. localspsa on the body coordinates: as soma_adam_update, with the
 * body's probe law. */
int soma_body_adam_update(float* params, float* m, float* v, int n_experts, soma_body_dims d,
                          int n_pert, int probe_kind, uint64_t seed, const uint64_t* steps,
                          int n_acc, const float* coef, soma_adam_config cfg, void* stream);

/* z_out device int8 [count]: body probe coordinates p0 .. p0 + count - 1
 * (p0 + count <= 2^30). */
int soma_debug_body_probe(uint64_t seed, uint64_t step, int expert, int pert, soma_body_dims d,
                          int probe_kind, int64_t p0, int64_t count, int8_t* z_out,
                          void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SOMA_API_H */
