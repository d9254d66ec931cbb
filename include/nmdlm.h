/*
 * nmdlm.h -- C ABI of the GB300 (sm_103a) N-MDLM block-denoise library.
 *
 * The library computes the forward pass of the spiking transformer of
 * Wu, Ruah, Chen, Rajendran, Simeone, "Neuromorphic Diffusion Language Models:
 * Addressing Compute and Memory Bottlenecks via Sparsity and Block Denoising"
 * (arXiv 2607.24841): binary spike blocks of B tokens x T timesteps multiply int8
 * weights (the QBSM class), the integer sums drive integrate-and-fire (IF) neurons
 * (Sec. II-B, Eq. (3)-(4)), and rows of W^T whose input channel is silent are never
 * fetched (Sec. IV-A, assumption (ii)).
 *
 * General conventions
 * -------------------
 *  - Every call returns nmdlm_status; nothing throws across the ABI and nothing
 *    aborts.  nmdlm_status_string() names a status.
 *  - Tensor pointers are DEVICE pointers owned by the caller, unless a parameter
 *    says "host".  `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Calls are asynchronous on that stream.
 *  - Device-side checks (a spike value other than 0/1, a token id out of range, a
 *    bounded wait that ran out) do not fault: kernels record them in an error word
 *    of the context, and nmdlm_ctx_sync_status() reports and clears it.
 *  - The library allocates device memory only in nmdlm_ctx_create() and frees it
 *    only in nmdlm_ctx_destroy().  No other call allocates.
 *  - Bit layouts.  A packed spike row holds channel c at bit (c % 32) of word c / 32
 *    (words(n) = ceil(n / 32)); a row index bt = b * T + t enumerates token b at
 *    timestep t.  A spike block of BT rows and D channels is described by
 *      row_bits    [BT][words(D)]   spike (bt, d) at bit d%32 of word d/32,
 *      col_masks   [D][words(BT)]   spike (bt, d) at bit bt%32 of word bt/32,
 *      active_mask [words(D)]       bit d set iff channel d spikes in some row,
 *      active_idx  [D]              ascending active channels (first *n_active valid).
 *    Bits beyond the last channel / row are zero.
 *  - Weights are stored transposed, W^T [d_in][d_out] int8 row-major, so the weights
 *    of one input channel form one contiguous row; scale [d_out] fp32 turns the
 *    integer sum of output channel o into a current: I = fp32(acc) * scale[o].
 *  - Limits: 1 <= T <= 32, 1 <= BT <= 256, dims >= 1, d_head % 32 == 0.
 */
#ifndef NMDLM_H
#define NMDLM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define NMDLM_ABI_VERSION 2

typedef enum nmdlm_status {
    NMDLM_OK = 0,
    NMDLM_ERR_INVALID_ARG = 1, /* bad pointer/size, or a device-side value check failed */
    NMDLM_ERR_UNSUPPORTED = 2, /* a size outside the documented limits */
    NMDLM_ERR_CUDA = 3,        /* a CUDA runtime call failed (launch, copy, ...) */
    NMDLM_ERR_TIMEOUT = 4,     /* a bounded device wait ran out; the kernel returned early */
    NMDLM_ERR_WORKSPACE = 5    /* the context workspace is too small for the call */
} nmdlm_status;

typedef enum nmdlm_mode {
    NMDLM_MODE_AUTO = 0,   /* library picks; the result never depends on the choice */
    NMDLM_MODE_SPARSE = 1, /* fetch only active rows of W^T (Sec. IV-A assumption (ii)) */
    NMDLM_MODE_DENSE = 2   /* fetch every row of W^T (the plain GEMM of an MDLM) */
} nmdlm_mode;

typedef enum nmdlm_impl {
    NMDLM_IMPL_AUTO = 0, /* tensor-core kernel where it applies, else CUDA cores */
    NMDLM_IMPL_SIMT = 1, /* CUDA-core accumulation (small blocks) */
    NMDLM_IMPL_TC = 2    /* tcgen05 tensor-core kernel */
} nmdlm_impl;

typedef enum nmdlm_if_kind {
    NMDLM_IF_INT = 0, /* threshold on the raw int32 synaptic sum */
    NMDLM_IF_FP32 = 1 /* threshold on the fp32 current (scale, residual, gate applied) */
} nmdlm_if_kind;

typedef enum nmdlm_dtype { NMDLM_I32 = 0, NMDLM_F32 = 1 } nmdlm_dtype;

typedef struct nmdlm_ctx nmdlm_ctx;
typedef struct nmdlm_model nmdlm_model;

const char* nmdlm_status_string(nmdlm_status s);
int nmdlm_abi_version(void);
/* Number of CUDA kernels the library has launched in this process (host-side count;
 * a CUDA graph replay launches again what its capture counted once). */
uint64_t nmdlm_launch_count(void);
/* Message of the last CUDA runtime error behind an NMDLM_ERR_CUDA on this thread. */
const char* nmdlm_last_cuda_error(void);

/* ------------------------------------------------------------- context ---- */
/* Create a context on `device` (made current for the call).  Allocates the
 * workspace (workspace_bytes; 0 = 512 MiB) and the device error word.  *ctx is NULL
 * on failure. */
nmdlm_status nmdlm_ctx_create(nmdlm_ctx** ctx, int device, size_t workspace_bytes);
nmdlm_status nmdlm_ctx_destroy(nmdlm_ctx* ctx);

/* Synchronize `stream`, then read and clear the device error word.  Returns the
 * first recorded device-side error (NMDLM_ERR_INVALID_ARG, NMDLM_ERR_TIMEOUT) or
 * NMDLM_OK. */
nmdlm_status nmdlm_ctx_sync_status(nmdlm_ctx* ctx, void* stream);

/* Kernel family for spiking linears (tests and benchmarks; AUTO by default). */
nmdlm_status nmdlm_ctx_set_impl(nmdlm_ctx* ctx, nmdlm_impl impl);

/* Upper bound, in nanoseconds, of every device-side wait (default 1e9 = 1 s).  A
 * wait that runs out records NMDLM_ERR_TIMEOUT, abandons the kernel's remaining
 * work, waits (with the default bound) for its own asynchronous operations, frees
 * its tensor memory and returns. */
nmdlm_status nmdlm_ctx_set_wait_limit(nmdlm_ctx* ctx, uint64_t ns);

/* Fault-injection check of the bounded-wait mechanism: launches one kernel that
 * waits on a barrier no thread ever completes.  After it, nmdlm_ctx_sync_status()
 * returns NMDLM_ERR_TIMEOUT and the context stays usable. */
nmdlm_status nmdlm_debug_wait_test(nmdlm_ctx* ctx, uint64_t ns, void* stream);

/* Per-kernel timing and algorithmic-byte accounting (off by default).  While
 * enabled, each spiking-linear launch is bracketed by CUDA events on its stream and
 * its device-side counters are accumulated; no CUDA graph capture may be active. */
nmdlm_status nmdlm_ctx_set_profiling(nmdlm_ctx* ctx, int enable);
/* Synchronizes the context's streams seen while profiling and returns, for the
 * spiking-linear kernel: number of launches, total event time (ms), total
 * algorithmic bytes (active W^T rows * d_out + scales + packed spikes in/out), and
 * total active rows fetched.  Resets the accumulators. */
nmdlm_status nmdlm_ctx_profile_read(nmdlm_ctx* ctx, uint64_t* launches, double* total_ms,
                                    double* total_bytes, double* rows_fetched);
/* The same launches one by one (call before nmdlm_ctx_profile_read, which resets them):
 * out [max_launches][6] host doubles {event time (ms), W^T rows fetched, synaptic
 * operations (input spikes * d_out), d_in, d_out, block rows BT}; *n_out launches
 * written.  The measured input sparsity of a launch is 1 - ops / (d_out * BT * d_in),
 * the sigma of Sec. IV-A, and rows / d_in its fetched-row fraction (1 - sigma^{BT} for
 * i.i.d. spikes). */
nmdlm_status nmdlm_ctx_profile_launches(nmdlm_ctx* ctx, int max_launches, double* out,
                                        int* n_out);

/* ------------------------------------------------------------ spikes ---- */
/* A packed spike block (see "Bit layouts").  col_masks and active_mask are what the
 * spiking linear reads; row_bits is what attention reads. */
typedef struct nmdlm_spikes {
    const uint32_t* row_bits;    /* [BT][words(D)] */
    const uint32_t* col_masks;   /* [D][words(BT)] */
    const uint32_t* active_mask; /* [words(D)] */
    const int32_t* active_idx;   /* [D] or NULL */
    const int32_t* n_active;     /* device scalar or NULL */
    int32_t BT, T, D;
} nmdlm_spikes;

/* Pack a uint8 0/1 spike block [BT][D] (row bt = b*T + t) and compact its active
 * channels (Sec. IV-A assumption (ii): channel d is loaded iff some row spikes in
 * it).  Outputs as in "Bit layouts"; any output may be NULL except row_bits.
 * A value other than 0/1 records NMDLM_ERR_INVALID_ARG in the error word. */
nmdlm_status nmdlm_pack_spikes(nmdlm_ctx* ctx, const uint8_t* spikes, int BT, int D,
                               uint32_t* row_bits, uint32_t* col_masks,
                               uint32_t* active_mask, int32_t* active_idx,
                               int32_t* n_active, void* stream);

/* ---------------------------------------------------------------- IF ---- */
/* Integrate-and-fire with soft reset (Sec. II-B, Eq. (3)-(4)), charge-then-fire:
 * H_t = V_{t-1} + I_t, s_t = [H_t >= threshold], V_t = H_t - s_t * threshold,
 * V_0 = 0 unless v_state is given.
 *   current   [B][T][N] int32 (dt = NMDLM_I32, threshold_i) or fp32 (NMDLM_F32,
 *             threshold_f); neuron (b, n) sees current[b][t][n] at step t.
 *   v_state   [B][N] of the same dtype, read as V_0 and overwritten with V_T; or NULL.
 *   spikes_out row bits [B*T][words(N)] (required); col_masks_out [N][words(B*T)]
 *             and active_mask_out [words(N)] optional: together they form the spike
 *             block a spiking linear consumes.
 * B, T or N below 1, or dt neither NMDLM_I32 nor NMDLM_F32, returns
 * NMDLM_ERR_INVALID_ARG; T > 32 or B*T > 256 returns NMDLM_ERR_UNSUPPORTED. */
nmdlm_status nmdlm_if_neuron(nmdlm_ctx* ctx, const void* current, nmdlm_dtype dt, int B,
                             int T, int N, int32_t threshold_i, float threshold_f,
                             void* v_state, uint32_t* spikes_out, uint32_t* col_masks_out,
                             uint32_t* active_mask_out, void* stream);

/* ------------------------------------------------------- spiking linear ---- */
/* IF epilogue fused into the spiking linear (spikes never round-trip as integers).
 * For output channel o, token b, t = 1..T, with acc = the int32 synaptic sum:
 *   NMDLM_IF_INT : H = V + acc, threshold_i on the raw sum.
 *   NMDLM_IF_FP32: I = fp32(acc) * scale[o] (one rounding); I += residual_in[bt][o];
 *                  I = gate(bt, o) ? I : 0 (if gate_bits); H = V + I; threshold_f.
 *   current_out[bt][o] (optional) = I (INT kind: fp32(acc) * scale[o]). */
typedef struct nmdlm_if_epilogue {
    int32_t kind;               /* nmdlm_if_kind */
    int32_t threshold_i;
    float threshold_f;
    const float* residual_in;   /* [BT][d_out] or NULL (FP32 kind only) */
    const uint32_t* gate_bits;  /* row bits [BT][words(d_out)] or NULL (FP32 kind only) */
    float* current_out;         /* [BT][d_out] or NULL */
    uint32_t* spikes_out;       /* row bits [BT][words(d_out)], required */
    uint32_t* col_masks_out;    /* [d_out][words(BT)] or NULL */
    uint32_t* active_mask_out;  /* [words(d_out)] or NULL */
} nmdlm_if_epilogue;

/* QBSM spiking linear (Sec. IV-A): acc[bt][o] = sum_d x[bt][d] * W^T[d][o] over the
 * active channels d of `in` (every other term is zero), exact in int32.
 *   in      spike block with col_masks, active_mask, BT, T, D = d_in.
 *   wT      [d_in][d_out] int8;  scale [d_out] fp32 (needed by an FP32 epilogue or
 *           a current_out).
 *   mode    which rows of W^T are streamed; results identical:
 *           SPARSE the active rows only (row skipping, assumption (ii));
 *           DENSE  every row, in order;
 *           AUTO   the active rows, or every row once at least 1/4 of them are
 *                  active (contiguous rows load as whole tiles; an inactive row only
 *                  multiplies zero spikes).
 *   acc_out [BT][d_out] int32 or NULL;  epi: IF epilogue or NULL (not both NULL).
 *   stats   NULL or device uint64[2] incremented by {active rows of W^T (the rows the
 *           method needs), synaptic operations = spikes * d_out} (Sec. IV-A
 *           assumptions (i)-(ii)).
 * Split-K partial sums are exchanged inside thread-block clusters; the context
 * workspace is not needed by the tensor-core path. */
nmdlm_status nmdlm_spike_linear(nmdlm_ctx* ctx, const nmdlm_spikes* in, const int8_t* wT,
                                const float* scale, int d_in, int d_out, nmdlm_mode mode,
                                int32_t* acc_out, const nmdlm_if_epilogue* epi,
                                uint64_t* stats, void* stream);

/* ------------------------------------------------ ternary bitwise coding ---- */
/* Adaptive quantisation and bitwise ternary coding of activations (Sec. II-C,
 * Conversion).  Row n of a is one activation vector of D values.
 *   Eq. (7): V_th = mean_i |a_i| / K,  ahat = round(a / V_th);
 *   Eq. (8): ahat_i = sum_{t=1}^{T} 2^{t-1} s_{i,t},  s_{i,t} in {-1, 0, 1},
 *            s_{i,t} = sign(ahat_i) * (bit t-1 of |ahat_i|).
 * Precision (the decisions are integers, taken identically by any conforming
 * implementation): |a| summed in fp64, V_th = (mean / K) rounded once to fp32, one
 * fp32 division a / V_th, round() with halves away from zero, |ahat| clamped to
 * 2^T - 1 (T planes hold exactly that).  A row whose V_th is not positive (all zeros,
 * or a NaN in it) and every NaN value quantise to 0.
 *   a          [N][D] fp32 (device).
 *   plus_out, minus_out  uint8 0/1 [N*T][D]: spike row n*T + t-1 carries the +1 and
 *              the -1 spikes of plane t, the layout nmdlm_pack_spikes takes.
 *   ahat_out   [N][D] int32 or NULL;  vth_out [N] fp32 or NULL.
 * K must be finite and > 0 and 1 <= T <= 24, else NMDLM_ERR_INVALID_ARG. */
nmdlm_status nmdlm_ternary_encode(nmdlm_ctx* ctx, const float* a, int N, int D, float K,
                                  int T, uint8_t* plus_out, uint8_t* minus_out,
                                  int32_t* ahat_out, float* vth_out, void* stream);

/* The bit-weighted sum of the modified IF neuron's input currents (Sec. II-C): with
 * I_t[n][o] = acc_plus[n*T + t-1][o] - acc_minus[n*T + t-1][o] (the +1 and -1 planes
 * through nmdlm_spike_linear), y[n][o] = sum_{t=1}^{T} 2^{t-1} I_t[n][o].  The
 * caller guarantees |y| < 2^31 (true whenever 127 * (2^T - 1) * d_in < 2^31).
 *   acc_plus, acc_minus [N*T][d_out] int32;  y_out [N][d_out] int32. */
nmdlm_status nmdlm_ternary_combine(nmdlm_ctx* ctx, const int32_t* acc_plus,
                                   const int32_t* acc_minus, int N, int T, int d_out,
                                   int32_t* y_out, void* stream);

/* The modified IF neuron of Sec. II-C (Eq. (9)-(10)), as this library reads the
 * garbled equations: the neuron integrates its bit-weighted input y (the output of
 * nmdlm_ternary_combine / nmdlm_ternary_linear) at once, V = y, then emits one ternary
 * spike per step from the most significant down: for t = T, ..., 1, s_t = +1 if
 * V >= 2^{t-1} theta, -1 if V <= -2^{t-1} theta, else 0, and V -= 2^{t-1} theta s_t.
 * With theta = 1 and |y| <= 2^T - 1 this re-encodes y exactly in Eq. (8)'s bit planes
 * (sum_t 2^{t-1} s_t = y, V ends at 0); otherwise |V| at the end is below theta unless
 * |y| >= (2^T - 1) theta, where the spikes saturate.
 *   y        [N][d_out] int32 (device).
 *   spikes_out [N][T][d_out] int8 in {-1, 0, 1}: plane t-1 of row n.
 *   v_out    [N][d_out] int32 (V after step 1) or NULL.
 * 1 <= T <= 24 and theta >= 1, else NMDLM_ERR_INVALID_ARG. */
nmdlm_status nmdlm_ternary_if(nmdlm_ctx* ctx, const int32_t* y, int N, int d_out, int T,
                              int theta, int8_t* spikes_out, int32_t* v_out, void* stream);

/* The linear on bitwise ternary spikes, end to end: encode (as above), pack the +1 and
 * -1 planes as one block of 2 N T rows (rows n*2T + t-1 and n*2T + T + t-1), run it
 * through the spiking linear once (the weights stream once for both planes; a row of
 * W^T is fetched when either plane spikes in it, `mode` as in nmdlm_spike_linear) and
 * combine, so y[n][o] = sum_i W^T[i][o] ahat_{n,i} exactly (Eq. (8) substituted into
 * the currents).  Blocks of more than 128 rows (2 N T > 128) run the planes as two
 * launches.
 *   a [N][D] fp32;  wT [D][d_out] int8;  y_out [N][d_out] int32;
 *   ahat_out [N][D] int32 or NULL;  vth_out [N] fp32 or NULL.
 * K and T as for nmdlm_ternary_encode (else NMDLM_ERR_INVALID_ARG); N*T > 256 or
 * 127 * (2^T - 1) * D >= 2^31 returns NMDLM_ERR_UNSUPPORTED.
 * Uses the context workspace (2 N T D bytes of planes, 8 N T d_out bytes of sums, the
 * packed planes). */
nmdlm_status nmdlm_ternary_linear(nmdlm_ctx* ctx, const float* a, int N, int D, float K,
                                  int T, const int8_t* wT, int d_out, nmdlm_mode mode,
                                  int32_t* y_out, int32_t* ahat_out, float* vth_out,
                                  void* stream);

/* ---------------------------------------------------- spike attention ---- */
/* Binary-binary (BBM) spike attention, one timestep and head at a time (the paper
 * names the BBM class and a spiking attention inside each layer, Fig. 1, without an
 * equation; this is the library's reading):
 *   score[i][j] = popcount(q_i AND k_j) over the head's d_head bits,
 *   p = softmax_j(alpha * score), out_i = sum_j p_ij v_j   (fp32),
 *   then IF over t (threshold theta, V_0 = 0) per (token, channel).
 *   q_bits   [B*T][words(H*d_head)] row bits of the block's queries.
 *   k_bits, v_bits [T][L_stride][words(H*d_head)]; keys 0..L_keys-1 are visible to
 *            every query (no causal mask: the block sees its context and itself).
 *   current_out [B*T][H*d_head] fp32 or NULL; spikes_out row bits (required);
 *   col_masks_out / active_mask_out optional (the O projection's input block).
 * d_head % 32 != 0, d_head > 256, T > 32, B*T > 256 or H*d_head > 2^20 returns
 * NMDLM_ERR_UNSUPPORTED, as does a key count whose bits do not fit on chip where the
 * kernel stages them: for d_head 128 (with alpha * 128 <= 18 ln 2) the keys stream
 * through shared memory and any count fits; otherwise one (timestep, head) stages all
 * its K and transposed V bits, L_keys * d_head / 4 bytes (plus B * L_keys bytes of
 * scores when d_head is not 32, 64, 96 or 128), within about 220 KB.
 * Uses the context workspace. */
nmdlm_status nmdlm_spike_attention(nmdlm_ctx* ctx, const uint32_t* q_bits,
                                   const uint32_t* k_bits, const uint32_t* v_bits, int T,
                                   int B, int L_keys, int L_stride, int H, int d_head,
                                   float alpha, float theta, float* current_out,
                                   uint32_t* spikes_out, uint32_t* col_masks_out,
                                   uint32_t* active_mask_out, void* stream);

/* Spike attention without a context and without any device allocation.  The paper
 * has no counterpart: this entry point exists for callers that cannot call cudaMalloc
 * -- for example a host framework whose own allocator owns all device memory, or an
 * embedded runtime with a fixed device-memory budget -- and therefore cannot create an
 * nmdlm_ctx (whose workspace is allocated).  It computes exactly what
 * nmdlm_spike_attention computes (same kernels, same arguments except ctx and
 * current_out) and allocates nothing.
 *   - The fp32 attention currents are staged in a library-owned static device array
 *     of nmdlm_spike_attention_noalloc_max() floats (1,048,576 = 4 MiB); every GPU that
 *     loads the library holds that array until the process exits.  B*T*H*d_head larger
 *     than the maximum returns NMDLM_ERR_UNSUPPORTED without launching anything.
 *   - The first call on a device resolves the array's device address (with that device
 *     current); make that first call before any stream capture.  A cudaDeviceReset
 *     discards the array with the device's memory: after a reset the resolved address
 *     is stale, and this entry point must not be called again in the process.
 *   - Every call shares the one array, which keeps the last call's contents; each call
 *     writes every element it later reads, so nothing needs clearing, but calls that
 *     overlap on the GPU (e.g. on different streams) race on the array and must be
 *     serialized by the caller.
 *   - There is no context error word: device-side checks are not reported. */
nmdlm_status nmdlm_spike_attention_noalloc(const uint32_t* q_bits, const uint32_t* k_bits,
                                           const uint32_t* v_bits, int T, int B, int L_keys,
                                           int L_stride, int H, int d_head, float alpha,
                                           float theta, uint32_t* spikes_out,
                                           uint32_t* col_masks_out, uint32_t* active_mask_out,
                                           void* stream);
/* Capacity, in floats, of the array nmdlm_spike_attention_noalloc stages currents in. */
size_t nmdlm_spike_attention_noalloc_max(void);

/* --------------------------------------------------------------- model ---- */
typedef struct nmdlm_model_desc {
    int32_t n_layers, d_model, n_heads, d_head, d_mlp;
    int32_t gated;   /* 0: up -> IF -> down; 1: the up current passes only where the gate
                        population spiked (gate IF on its own projection) */
    int32_t vocab;   /* logits rows; token id `vocab` is the mask token */
    int32_t T;       /* spike timesteps per token */
    float theta;     /* threshold of every fp32 IF population */
    int32_t B, S;    /* block size and denoising steps per block, B % S == 0 */
    int32_t max_ctx; /* positions held by the K/V caches and the position table */
    int32_t n_enc_layers; /* 0: every layer serves the context pass and the denoising
                             steps.  > 0: the encoder-decoder split of Sec. III-A,
                             Eq. (5)-(6): n_enc_layers encoder layers run on the context
                             pass only, then the n_layers decoder layers on the steps */
} nmdlm_model_desc;

typedef struct nmdlm_linear_w {
    const int8_t* wT;   /* [d_in][d_out] */
    const float* scale; /* [d_out] */
} nmdlm_linear_w;

typedef struct nmdlm_layer_w {
    nmdlm_linear_w q, k, v, o; /* [D][D] each */
    nmdlm_linear_w gate;       /* [D][F], gated models only */
    nmdlm_linear_w up;         /* [D][F] */
    nmdlm_linear_w down;       /* [F][D] */
} nmdlm_layer_w;

/* Record a model.  `layers` is a HOST array of n_enc_layers + n_layers entries (the
 * encoder layers first) whose device pointers stay owned by the caller and must
 * outlive the model.  tok_emb
 * [vocab+1][D] fp32 (row vocab = mask token), pos_emb [max_ctx][D] fp32, head
 * W^T [D][vocab] int8 + scale [vocab].  Allocates no device memory. */
nmdlm_status nmdlm_model_create(nmdlm_ctx* ctx, const nmdlm_model_desc* desc,
                                const nmdlm_layer_w* layers, const float* tok_emb,
                                const float* pos_emb, nmdlm_linear_w head,
                                nmdlm_model** model);
nmdlm_status nmdlm_model_destroy(nmdlm_model* model);
/* Workspace bytes the model's step needs (host query). */
size_t nmdlm_model_workspace_bytes(const nmdlm_model_desc* desc);

/* One layer on a block (Fig. 1): Q/K/V spiking linears with IF epilogues (K and V
 * written into the caches at positions ctx_len..ctx_len+B-1), spike attention over
 * keys 0..ctx_len+B-1, output projection with residual current and IF, MLP (plain or
 * gated) and down projection with residual current and IF.  Optional trace outputs
 * receive intermediates (NULL skips them). */
typedef struct nmdlm_layer_io {
    const uint32_t* x_bits;        /* [BT][words(D)] input spikes */
    const uint32_t* x_col_masks;   /* [D][words(BT)] */
    const uint32_t* x_active_mask; /* [words(D)] */
    const float* u_in;             /* [BT][D] residual current stream */
    uint32_t* k_cache;             /* this layer's [T][max_ctx][words(D)] */
    uint32_t* v_cache;
    int32_t ctx_len;
    uint32_t* x_bits_out;          /* [BT][words(D)] */
    uint32_t* x_col_masks_out;     /* [D][words(BT)] */
    uint32_t* x_active_mask_out;   /* [words(D)] */
    float* u_out;                  /* [BT][D] */
    /* trace (optional) */
    uint32_t* q_bits;              /* [BT][words(D)] */
    float* attn_current;           /* [BT][D] */
    uint32_t* attn_bits;           /* [BT][words(D)] */
    float* u1;                     /* [BT][D] residual after the output projection */
    uint32_t* x1_bits;             /* [BT][words(D)] */
    uint32_t* g_bits;              /* [BT][words(F)] gate spikes (gated) */
    uint32_t* h_bits;              /* [BT][words(F)] spikes entering the down projection */
    /* teacher forcing (parity checks): when attn_bits_in is set, the layer runs Q/K/V
     * (and writes the caches) but skips its attention and attention IF and feeds these
     * spikes to the output projection; all three must then be given. */
    const uint32_t* attn_bits_in;        /* [BT][words(D)] */
    const uint32_t* attn_col_masks_in;   /* [D][words(BT)] */
    const uint32_t* attn_active_mask_in; /* [words(D)] */
} nmdlm_layer_io;

/* `layer` indexes the model's whole layer array (encoder layers first). */
nmdlm_status nmdlm_layer_forward(nmdlm_ctx* ctx, const nmdlm_model* model, int layer,
                                 const nmdlm_layer_io* io, void* stream);

/* Block state of the generation loop (Sec. III-A; Eq. (2)). */
typedef struct nmdlm_block_state {
    int32_t* tokens;   /* device [B]; masked positions hold the mask id (vocab) */
    int32_t* mask;     /* device [B]; 1 = still masked */
    uint32_t* k_cache; /* device [n_enc_layers + n_layers][T][max_ctx][words(D)] */
    uint32_t* v_cache;
    int32_t ctx_len;   /* host: committed context positions */
    int32_t step;      /* host: denoising steps already taken in this block */
} nmdlm_block_state;

/* One denoising step s = step+1 of Sec. III-A (Eq. (6)): embed the block (mask
 * embedding at masked positions, positions ctx_len+b), run every layer (the block's
 * K/V go to cache positions ctx_len..ctx_len+B-1 without committing them), decode
 * rate-coded logits, and unmask the B/S most confident masked positions (greedy by
 * max-probability; ties to the lowest token id, then the lowest position).
 *   unmasked_out [B/S] int32 or NULL: positions unmasked, in selection order.
 *   logits_out [B][vocab] fp32 or NULL.
 * Errors: step == S (block finished), ctx_len + B > max_ctx. */
nmdlm_status nmdlm_block_denoise_step(nmdlm_ctx* ctx, const nmdlm_model* model,
                                      nmdlm_block_state* st, int32_t* unmasked_out,
                                      float* logits_out, void* stream);

/* Context pass over the finished block (Eq. (2): the block joins x^{<b}): runs every
 * layer on the clean tokens, writing their K/V spikes at ctx_len..ctx_len+B-1, then
 * ctx_len += B, step = 0, and every position is re-masked for the next block.  With
 * n_enc_layers > 0 it runs the encoder layers instead (Eq. (5): h^b, the last encoder
 * layer's output spikes for the block), and each decoder layer's K and V spikes of h^b
 * (its own K/V projections and IF) go to that decoder layer's cache positions; a
 * denoising step then runs only the decoder layers (Eq. (6)). */
nmdlm_status nmdlm_block_commit(nmdlm_ctx* ctx, const nmdlm_model* model,
                                nmdlm_block_state* st, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* NMDLM_H */
