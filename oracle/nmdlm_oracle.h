/*
 * nmdlm_oracle.h -- CPU oracle for the N-MDLM spiking block-denoise forward pass.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, __graft_entry__.smoke() and the
 * CPU-baseline leg of bench.py may load this library.  It shares no code, header,
 * table or helper with the CUDA library under paper_2607_24841_gb300/.
 *
 * Conventions (all arrays dense, row-major, caller-owned host memory):
 *   spikes      uint8 0/1, layout [B][T][N]  (row index bt = b*T + t)
 *   weights     int8  W^T, layout [d_in][d_out] (row d holds every output's
 *               weight for input channel d)
 *   scales      fp32 [d_out]
 *   K/V cache   uint8 0/1, layout [T][L][D]  (timestep, key position, channel)
 *
 * Every function is a plain restatement of a definition in the paper
 * (Wu, Ruah, Chen, Rajendran, Simeone: "Neuromorphic Diffusion Language Models",
 * arXiv 2607.24841); each cites the passage it follows.
 */
#ifndef NMDLM_ORACLE_H
#define NMDLM_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* IF update order.  ORC_IF_CHARGE_THEN_FIRE is the reading used everywhere:
 * H_t = V_{t-1} + I_t, s_t = [H_t >= th], V_t = H_t - s_t*th, V_0 = 0.
 * ORC_IF_FIRE_THEN_CHARGE is the literal order printed in Eq. (3)-(4): the spike
 * at t is decided on V_t before I_t is added.  Only tests use it. */
enum { ORC_IF_CHARGE_THEN_FIRE = 0, ORC_IF_FIRE_THEN_CHARGE = 1 };

/* IF threshold kinds of the linear epilogue. */
enum { ORC_EPI_INT = 0, ORC_EPI_F32 = 1 };

int orc_version(void);

/* Host threads for the loops marked "parallel" in nmdlm_oracle.c (OpenMP; 1 when the
 * oracle is built without it).  Each output element is computed by one thread in the
 * written order, so results never depend on the thread count. */
void orc_set_threads(int n);
int orc_get_threads(void);

/* Sec. II-B, Eq. (3)-(4): integrate-and-fire with soft reset, integer currents.
 * current [B][T][N] int64, spikes out [B][T][N], v_final [B][N] (nullable). */
void orc_if_int(const int64_t* current, int B, int T, int N, int64_t theta,
                int order, uint8_t* spikes, int64_t* v_final);

/* Same neuron with fp32 currents and membrane.  margin [B][N] (nullable) receives
 * min_t |H_t - theta| evaluated in fp64 on the fp32 membrane values. */
void orc_if_f32(const float* current, int B, int T, int N, float theta,
                uint8_t* spikes, float* v_final, double* margin);

/* Sec. IV-A assumption (ii): channel d of the BT x D spike block is active iff
 * some row bt has x_{bt,d} = 1.  Produces the packed forms the CUDA path uses:
 *   row_bits   [BT][ceil(D/32)]   bit (d%32) of word d/32 is x_{bt,d}
 *   col_masks  [D][ceil(BT/32)]   bit (bt%32) of word bt/32 is x_{bt,d}
 *   active_mask[ceil(D/32)]       bit d%32 of word d/32 set iff d active
 *   active_idx [D]                ascending active channels, first *n_active valid
 * Any output pointer may be NULL. */
void orc_pack(const uint8_t* spikes, int BT, int D, uint32_t* row_bits,
              uint32_t* col_masks, uint32_t* active_mask, int32_t* active_idx,
              int32_t* n_active);

/* Sec. IV-A: Y = X W^T with X in {0,1}^{BT x d_in}.  acc [BT][d_out] int64. */
void orc_qbsm(const uint8_t* spikes, const int8_t* wT, int BT, int d_in, int d_out,
              int64_t* acc);

/* The same sum at n sampled output positions (bt_idx[i], o_idx[i]). */
void orc_qbsm_at(const uint8_t* spikes, const int8_t* wT, int BT, int d_in, int d_out,
                 int n, const int32_t* bt_idx, const int32_t* o_idx, int64_t* acc);

/* Sec. IV-A event counts: rows of W^T loaded under assumption (ii) and synaptic
 * operations (one accumulate per spike per output channel) under assumption (i). */
void orc_qbsm_counts(const uint8_t* spikes, int BT, int d_in, int d_out,
                     int64_t* rows_fetched, int64_t* sops);

/* IF epilogue of a spiking linear layer.  For each output channel o and token b,
 * over t = 1..T:
 *   ORC_EPI_INT: H = V + acc (int64), threshold theta_i on the raw sum;
 *                current_out (nullable) = fp32(acc) * scale[o].
 *   ORC_EPI_F32: I = fp32(acc) * scale[o]; I = I + residual[bt][o] (if given);
 *                I = gate[bt][o] ? I : 0 (if given); fp32 IF with theta_f;
 *                current_out (nullable) = I.
 * acc [BT][d_out], residual [BT][d_out] fp32, gate [BT][d_out] uint8,
 * spikes [BT][d_out], margin [B][d_out] (nullable, F32 only). */
void orc_if_epilogue(const int64_t* acc, int B, int T, int d_out, const float* scale,
                     const float* residual, const uint8_t* gate, int kind,
                     int64_t theta_i, float theta_f, float* current_out,
                     uint8_t* spikes, double* margin);

/* Binary-binary spike attention for one block.  For every timestep t and head h:
 *   score[i][j] = sum_c q[i,t,h*dh+c] * k[t,j,h*dh+c]     (0/1 dot = popcount of AND)
 *   p[i][j]     = softmax_j(alpha * score[i][j])          (fp64)
 *   out[i,t,h*dh+c] = sum_j p[i][j] * v[t,j,h*dh+c]        (fp64, rounded to fp32)
 * q [B][T][D]; k, v [T][L][D] with keys 0..L-1 all visible (no causal mask);
 * out [B][T][D] fp32. */
void orc_attention(const uint8_t* q, const uint8_t* k, const uint8_t* v, int B, int T,
                   int L, int H, int dh, double alpha, float* out);

/* ---------------------------------------------------------------- model ---- */
/* n_enc = 0: every layer serves both the context pass and the denoising steps.
 * n_enc > 0 (the encoder-decoder split of Sec. III-A, Eq. (5)-(6)): the layer array
 * holds n_enc encoder layers followed by n_layers decoder layers, and the caches hold
 * n_enc + n_layers layers (see orc_block_step). */
typedef struct {
    int n_layers, D, H, dh, F, gated, V, T, B, S, Lmax;
    float theta;
    int n_enc;
} orc_model;

typedef struct { const int8_t* w; const float* scale; } orc_lin;

typedef struct {
    orc_lin q, k, v, o, gate, up, down;   /* gate unused when !gated */
} orc_layer_w;

/* Per-layer intermediates (every pointer nullable). */
typedef struct {
    uint8_t* q;          /* [BT][D] */
    float* attn_cur;     /* [BT][D]   attention output current */
    uint8_t* attn;       /* [BT][D]   attention output spikes */
    double* attn_margin; /* [B][D]    IF margin of the attention spikes */
    float* u1;           /* [BT][D]   residual current after the output projection */
    uint8_t* x1;         /* [BT][D] */
    uint8_t* g;          /* [BT][F]   gate spikes (gated MLP) */
    uint8_t* h;          /* [BT][F]   hidden spikes entering the down projection */
} orc_layer_trace;

/* One spiking transformer layer on a block (Fig. 1; Sec. III-A).
 * x_in, u_in: input spikes [BT][D] and the residual current stream [BT][D].
 * k_cache/v_cache [T][Lmax][D]: positions 0..ctx-1 are the context; the block's
 * own K/V spikes are written to positions ctx..ctx+B-1 and attended to as well.
 * x_out, u_out: output spikes and residual current. */
void orc_layer(const orc_model* m, const orc_layer_w* w, const uint8_t* x_in,
               const float* u_in, uint8_t* k_cache, uint8_t* v_cache, int ctx,
               uint8_t* x_out, float* u_out, orc_layer_trace* trace);

/* Token + position embedding currents, constant over T:
 * u0[b][t][d] = tok_emb[tokens[b]][d] + pos_emb[pos0+b][d]  (fp32 add). */
void orc_embed(const float* tok_emb, const float* pos_emb, const int32_t* tokens,
               int B, int T, int D, int pos0, float* u0);

/* Rate-decoded logits head: logit[b][v] = (fp32(sum_t acc[b*T+t][v]) * scale[v]) / T. */
void orc_head(const uint8_t* x, const int8_t* wT, const float* scale, int B, int T,
              int D, int V, float* logits);

/* Unmasking of Sec. III-A: among still-masked positions pick the k most confident
 * (confidence = max softmax probability, fp64; token = argmax, lowest id on ties;
 * positions ranked by confidence, lowest position on ties).  Updates tokens/mask in
 * place.  conf/tok [B] (nullable) receive every position's confidence and argmax;
 * chosen [k] (nullable) the selected positions in selection order.  Returns the
 * number of positions unmasked. */
int orc_unmask(const float* logits, int B, int V, int k, int32_t* tokens,
               uint8_t* mask, double* conf, int32_t* tok, int32_t* chosen);

/* One denoising step (commit = 0) or one context pass over the now-clean block
 * (commit = 1) of Sec. III-A.  tokens/mask [B] in/out; caches [n_enc + n_layers][T]
 * [Lmax][D].  logits [B][V] (nullable, step only); chosen [B/S] (nullable).  Returns
 * the number of unmasked positions (0 for a commit pass).
 * With n_enc > 0 (Eq. (5)-(6)): the context pass runs the encoder layers over the clean
 * block (their own caches, block-causal: the block sees the committed context and
 * itself) and h, the last encoder layer's output spikes, becomes the decoder's context:
 * each decoder layer's K and V spikes of h (its own K/V projections and IF) are written
 * at the block's positions of that decoder layer's cache.  A denoising step runs only
 * the decoder layers, whose attention sees those context K/V and the block's own. */
int orc_block_step(const orc_model* m, const orc_layer_w* layers, const float* tok_emb,
                   const float* pos_emb, orc_lin head, int32_t* tokens, uint8_t* mask,
                   uint8_t* k_cache, uint8_t* v_cache, int ctx, int commit,
                   float* logits, int32_t* chosen);

/* orc_block_step that also reports, in *attn_margin (nullable), the smallest distance
 * min |H - theta| over every attention IF membrane of every layer in the pass: where it
 * is tiny, an fp32 implementation that sums the softmax mixture in another order may
 * legitimately decide that spike the other way. */
int orc_block_step_margin(const orc_model* m, const orc_layer_w* layers,
                          const float* tok_emb, const float* pos_emb, orc_lin head,
                          int32_t* tokens, uint8_t* mask, uint8_t* k_cache, uint8_t* v_cache,
                          int ctx, int commit, float* logits, int32_t* chosen,
                          double* attn_margin);

/* Sec. II-C (Conversion), Eq. (7): adaptive step V_th(a) = mean_i |a_i| / K and
 * ahat = round(a / V_th); Eq. (8): ahat_i = sum_{t=1}^{T} 2^{t-1} s_{i,t} with ternary
 * s_{i,t} in {-1, 0, 1}.  One row n of a [N][D] is one activation vector a.
 * Readings: the mean is summed in fp64 and V_th = (mean / K) rounded once to fp32;
 * the quotient a_i / V_th is one fp32 division and round() takes halves away from
 * zero; a row with V_th = 0 (all zeros) quantises to 0; NaN quantises to 0;
 * |ahat_i| is clamped to 2^T - 1 (T planes hold exactly that; the printed
 * T = floor(log2 max|ahat|) is one plane short of max|ahat| itself, see
 * orc_ternary_planes_needed); s_{i,t} = sign(ahat_i) * (bit t-1 of |ahat_i|).
 *   s    [N][T][D] int8 (row n*T + t-1);  ahat [N][D] int32 (nullable);
 *   vth  [N] fp32 (nullable).  1 <= T <= 30. */
/* Eq. (7)'s sum of |a| over one activation row, taken exactly and rounded once to
 * fp64 (nearest, ties to even); NaN if the row holds a NaN, +Inf if it holds an
 * infinity.  The mean and the step follow from it in fp64, so V_th does not depend on
 * any order of summation. */
double orc_abs_sum_exact(const float* row, int D);

void orc_ternary_encode(const float* a, int N, int D, float K, int T, int8_t* s,
                        int32_t* ahat, float* vth);

/* Planes T for which sum_{t=1}^{T} 2^{t-1} s_t reaches m = max|ahat|: the bit
 * length of m (floor(log2 m) + 1 for m >= 1, 0 for m = 0). */
int orc_ternary_planes_needed(int64_t m);

/* Sec. II-C: the modified IF neuron's input current I_t[o] = sum_i W^T[i][o] s_{i,t}
 * for ternary s, and its bit-weighted sum y[o] = sum_t 2^{t-1} I_t[o], which by
 * Eq. (8) equals sum_i W^T[i][o] ahat_i.
 *   s [N][T][D] int8;  wT [D][d_out] int8;  I [N][T][d_out] int64 (nullable);
 *   y [N][d_out] int64. */
void orc_ternary_linear(const int8_t* s, const int8_t* wT, int N, int T, int D, int d_out,
                        int64_t* I, int64_t* y);

/* The modified IF neuron of Sec. II-C, Eq. (9)-(10), on the bit-weighted currents of
 * the linear on ternary spikes.  The printed indices are garbled (2^t I_t against the
 * 2^{t-1} weights of Eq. (8), I_t against s_t); reading:
 *   input  V = sum_{t=1}^{T} 2^{t-1} I_t      (= y = w^T ahat by Eq. (8)),
 *   output for t = T down to 1 (most significant step first):
 *          s_t = +1 if V >= 2^{t-1} theta, -1 if V <= -2^{t-1} theta, else 0,
 *          V  -= 2^{t-1} theta s_t             (Eq. (9)'s reset, Eq. (10)'s thresholds).
 * For |y| < 2^T theta the residual satisfies |V_T| < theta and theta sum_t 2^{t-1} s_t
 * = y - V_T (Eq. (11)'s approximation); with theta = 1 the spikes are Eq. (8)'s bitwise
 * coding of y.  y [N][d_out] int64, theta >= 1; s_out [N][T][d_out] in {-1, 0, 1} (plane
 * t-1 carries weight 2^{t-1}); v_final [N][d_out] (nullable). */
void orc_ternary_if(const int64_t* y, int N, int d_out, int T, int64_t theta, int8_t* s_out,
                    int64_t* v_final);

#ifdef __cplusplus
}
#endif
#endif
