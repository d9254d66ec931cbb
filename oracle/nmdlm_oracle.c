/*
 * nmdlm_oracle.c -- CPU oracle for the N-MDLM spiking block-denoise forward pass.
 *
 * TEST INFRASTRUCTURE ONLY.  Plain, slow loops that restate the paper's
 * definitions (Wu et al., "Neuromorphic Diffusion Language Models", arXiv
 * 2607.24841) so that a reader can check them by eye.  No packing, no skipping,
 * no blocking, no shared code with the CUDA library.
 *
 * Precision: synaptic sums in int64 (checked to fit int32); IF membranes in fp32,
 * the precision in which the CUDA path takes the same spike decision; softmax and
 * the attention mixture in fp64.  Compiled with -ffp-contract=off so every fp32
 * expression below is rounded once per operation, in the order written.
 *
 * Readings taken where the paper is silent (each one is also stated at its use):
 *   - IF order: charge-then-fire (H = V + I, fire on H, reset by subtraction),
 *     V_0 = 0, membranes reset for every layer, token and denoising step.
 *   - spikes are binary {0,1}; channel d of the spike block skips row d of W^T.
 *   - a per-output-channel fp32 scale turns the integer sum into a current.
 *   - residual currents are added before the IF that follows the output and
 *     down projections; there is no normalisation layer.
 *   - attention: per timestep and head, AND/popcount scores, softmax with
 *     alpha = 1/sqrt(dh) over every context and block key, mixture of V spikes,
 *     IF with the model threshold.
 *   - gated MLP: the down projection's input current is gate_spike * I_up.
 *   - logits are rate-decoded: fp32(sum_t acc_t) * scale / T.
 *   - unmasking is greedy by max-probability, ties to the lowest id / position.
 * The paper gives no layer equations: the composition of a layer (and of a denoising
 * step and the encoder-decoder context pass) from these readings is pinned by layers
 * worked by hand (tests/golden/layer_worked.json), each building block by its own
 * oracle tests.
 */
#include "nmdlm_oracle.h"

#include <assert.h>
#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

int orc_version(void) { return 2; }

/* Host threads for the loops below marked "parallel": each output element is still
 * computed by one thread in the order written, so the results do not depend on it. */
void orc_set_threads(int n) {
#ifdef _OPENMP
    omp_set_num_threads(n > 0 ? n : 1);
#else
    (void)n;
#endif
}

int orc_get_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

static size_t idx3(int a, int b, int c, int nb, int nc) {
    return ((size_t)a * (size_t)nb + (size_t)b) * (size_t)nc + (size_t)c;
}

/* ------------------------------------------------------------------ IF ---- */
/* Sec. II-B, Eq. (3): s_t = 1 iff the membrane reaches V_th (ties fire).
 * Eq. (4): V_{t+1} = V_t + I_t - s_t V_th (soft reset by subtraction).
 * Reading (charge-then-fire): the spike at t is decided on H_t = V_{t-1} + I_t,
 * so the current of step t can already produce the spike of step t. */
void orc_if_int(const int64_t* current, int B, int T, int N, int64_t theta, int order,
                uint8_t* spikes, int64_t* v_final) {
    for (int b = 0; b < B; ++b) {
        for (int n = 0; n < N; ++n) {
            int64_t v = 0;
            for (int t = 0; t < T; ++t) {
                int64_t i_t = current[idx3(b, t, n, T, N)];
                uint8_t s;
                if (order == ORC_IF_FIRE_THEN_CHARGE) {
                    s = (v >= theta) ? 1 : 0;          /* Eq. (3) on V_t */
                    v = v + i_t - (int64_t)s * theta;  /* Eq. (4) */
                } else {
                    int64_t h = v + i_t;
                    s = (h >= theta) ? 1 : 0;
                    v = h - (int64_t)s * theta;
                }
                spikes[idx3(b, t, n, T, N)] = s;
            }
            if (v_final) v_final[(size_t)b * N + n] = v;
        }
    }
}

void orc_if_f32(const float* current, int B, int T, int N, float theta, uint8_t* spikes,
                float* v_final, double* margin) {
    for (int b = 0; b < B; ++b) {
        for (int n = 0; n < N; ++n) {
            float v = 0.0f;
            double mg = INFINITY;
            for (int t = 0; t < T; ++t) {
                float h = v + current[idx3(b, t, n, T, N)];
                uint8_t s = (h >= theta) ? 1 : 0;
                double d = fabs((double)h - (double)theta);
                if (d < mg) mg = d;
                v = s ? (h - theta) : h;
                spikes[idx3(b, t, n, T, N)] = s;
            }
            if (v_final) v_final[(size_t)b * N + n] = v;
            if (margin) margin[(size_t)b * N + n] = mg;
        }
    }
}

/* ---------------------------------------------------------------- pack ---- */
/* Sec. IV-A, assumption (ii): the d-th input channel is loaded only if at least
 * one of the BT rows carries x_{t,d} = 1. */
void orc_pack(const uint8_t* spikes, int BT, int D, uint32_t* row_bits,
              uint32_t* col_masks, uint32_t* active_mask, int32_t* active_idx,
              int32_t* n_active) {
    int dw = (D + 31) / 32, bw = (BT + 31) / 32;
    if (row_bits) memset(row_bits, 0, sizeof(uint32_t) * (size_t)BT * dw);
    if (col_masks) memset(col_masks, 0, sizeof(uint32_t) * (size_t)D * bw);
    if (active_mask) memset(active_mask, 0, sizeof(uint32_t) * (size_t)dw);
    int count = 0;
    for (int d = 0; d < D; ++d) {
        int any = 0;
        for (int bt = 0; bt < BT; ++bt) {
            if (spikes[(size_t)bt * D + d]) {
                any = 1;
                if (row_bits) row_bits[(size_t)bt * dw + d / 32] |= 1u << (d % 32);
                if (col_masks) col_masks[(size_t)d * bw + bt / 32] |= 1u << (bt % 32);
            }
        }
        if (any) {
            if (active_mask) active_mask[d / 32] |= 1u << (d % 32);
            if (active_idx) active_idx[count] = d;
            ++count;
        }
    }
    if (n_active) *n_active = count;
}

/* ---------------------------------------------------------------- QBSM ---- */
/* Sec. IV-A: Y = X W^T, X in {0,1}^{BT x D} the spike trains of B tokens over T
 * steps.  Written as the dense sum; sparsity only removes zero terms from it. */
void orc_qbsm(const uint8_t* spikes, const int8_t* wT, int BT, int d_in, int d_out,
              int64_t* acc) {
#pragma omp parallel for schedule(dynamic, 1) /* parallel: one row bt per thread */
    for (int bt = 0; bt < BT; ++bt) {
        int64_t* row = acc + (size_t)bt * d_out;
        for (int o = 0; o < d_out; ++o) row[o] = 0;
        for (int d = 0; d < d_in; ++d) {
            int64_t x = spikes[(size_t)bt * d_in + d];
            const int8_t* w = wT + (size_t)d * d_out;
            for (int o = 0; o < d_out; ++o) row[o] += x * (int64_t)w[o];
        }
        for (int o = 0; o < d_out; ++o) assert(row[o] <= INT32_MAX && row[o] >= INT32_MIN);
    }
}

void orc_qbsm_at(const uint8_t* spikes, const int8_t* wT, int BT, int d_in, int d_out,
                 int n, const int32_t* bt_idx, const int32_t* o_idx, int64_t* acc) {
    (void)BT;
#pragma omp parallel for schedule(static) /* parallel: one sampled sum per thread */
    for (int i = 0; i < n; ++i) {
        int64_t s = 0;
        for (int d = 0; d < d_in; ++d)
            s += (int64_t)spikes[(size_t)bt_idx[i] * d_in + d] *
                 (int64_t)wT[(size_t)d * d_out + o_idx[i]];
        acc[i] = s;
    }
}

/* Sec. IV-A: (i) only spikes x = 1 cost synaptic operations, one per output
 * channel; (ii) row d of W^T is fetched iff channel d carries a spike. */
void orc_qbsm_counts(const uint8_t* spikes, int BT, int d_in, int d_out,
                     int64_t* rows_fetched, int64_t* sops) {
    int64_t rows = 0, nnz = 0;
    for (int d = 0; d < d_in; ++d) {
        int any = 0;
        for (int bt = 0; bt < BT; ++bt) {
            if (spikes[(size_t)bt * d_in + d]) { any = 1; ++nnz; }
        }
        rows += any;
    }
    if (rows_fetched) *rows_fetched = rows;
    if (sops) *sops = nnz * (int64_t)d_out;
}

/* ------------------------------------------------------------ epilogue ---- */
/* The integer sums become currents of the next IF population (Sec. II-B: the
 * synaptic current is the weighted sum of incoming spikes).  Readings: a
 * per-channel fp32 scale, a residual current added before the IF, an optional
 * gate spike that passes or blocks the current. */
void orc_if_epilogue(const int64_t* acc, int B, int T, int d_out, const float* scale,
                     const float* residual, const uint8_t* gate, int kind,
                     int64_t theta_i, float theta_f, float* current_out,
                     uint8_t* spikes, double* margin) {
    size_t n = (size_t)B * T * d_out;
    if (kind == ORC_EPI_INT) {
        orc_if_int(acc, B, T, d_out, theta_i, ORC_IF_CHARGE_THEN_FIRE, spikes, NULL);
        if (current_out && scale)
            for (size_t i = 0; i < n; ++i)
                current_out[i] = (float)acc[i] * scale[i % (size_t)d_out];
        return;
    }
    float* cur = (float*)malloc(sizeof(float) * n);
    for (size_t i = 0; i < n; ++i) {
        float c = (float)acc[i] * scale[i % (size_t)d_out];
        if (residual) c = c + residual[i];
        if (gate) c = gate[i] ? c : 0.0f;
        cur[i] = c;
    }
    orc_if_f32(cur, B, T, d_out, theta_f, spikes, NULL, margin);
    if (current_out) memcpy(current_out, cur, sizeof(float) * n);
    free(cur);
}

/* ----------------------------------------------------------- attention ---- */
/* Binary-binary multiplication (BBM) between spike tensors, Spikformer-style
 * attention inside each layer (Fig. 1).  The paper gives no equation; reading:
 * softmax attention over AND/popcount scores, then a mixture of V spikes. */
void orc_attention(const uint8_t* q, const uint8_t* k, const uint8_t* v, int B, int T,
                   int L, int H, int dh, double alpha, float* out) {
    int D = H * dh;
#pragma omp parallel for schedule(dynamic, 1) /* parallel: one (timestep, head) per thread */
    for (int th = 0; th < T * H; ++th) {
        int t = th / H, h = th % H;
        double* score = (double*)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
        for (int i = 0; i < B; ++i) {
            const uint8_t* qi = q + idx3(i, t, h * dh, T, D);
            double mx = -INFINITY;
            for (int j = 0; j < L; ++j) {
                const uint8_t* kj = k + idx3(t, j, h * dh, L, D);
                int dot = 0;
                for (int c = 0; c < dh; ++c) dot += qi[c] * kj[c];
                score[j] = alpha * (double)dot;
                if (score[j] > mx) mx = score[j];
            }
            double z = 0.0;
            for (int j = 0; j < L; ++j) {
                score[j] = exp(score[j] - mx);
                z += score[j];
            }
            for (int c = 0; c < dh; ++c) {
                double o = 0.0;
                for (int j = 0; j < L; ++j)
                    o += (score[j] / z) * (double)v[idx3(t, j, h * dh + c, L, D)];
                out[idx3(i, t, h * dh + c, T, D)] = (float)o;
            }
        }
        free(score);
    }
}

/* --------------------------------------------------------------- layer ---- */
static void lin_if(const orc_lin* w, const uint8_t* x, int B, int T, int d_in, int d_out,
                   const float* residual, const uint8_t* gate, float theta,
                   float* current_out, uint8_t* spikes) {
    int64_t* acc = (int64_t*)malloc(sizeof(int64_t) * (size_t)B * T * d_out);
    orc_qbsm(x, w->w, B * T, d_in, d_out, acc);
    orc_if_epilogue(acc, B, T, d_out, w->scale, residual, gate, ORC_EPI_F32, 0, theta,
                    current_out, spikes, NULL);
    free(acc);
}

/* Fig. 1: each neuromorphic transformer layer is attention + MLP with IF neurons.
 * Sec. III-A: the block's tokens attend to the context representation (here the
 * K/V spikes of the committed context) and to the block itself. */
void orc_layer(const orc_model* m, const orc_layer_w* w, const uint8_t* x_in,
               const float* u_in, uint8_t* k_cache, uint8_t* v_cache, int ctx,
               uint8_t* x_out, float* u_out, orc_layer_trace* trace) {
    int B = m->B, T = m->T, D = m->D, F = m->F, BT = B * T, L = ctx + B;
    size_t nd = (size_t)BT * D, nf = (size_t)BT * F;
    uint8_t* q = (uint8_t*)malloc(nd);
    uint8_t* kb = (uint8_t*)malloc(nd);
    uint8_t* vb = (uint8_t*)malloc(nd);
    lin_if(&w->q, x_in, B, T, D, D, NULL, NULL, m->theta, NULL, q);
    lin_if(&w->k, x_in, B, T, D, D, NULL, NULL, m->theta, NULL, kb);
    lin_if(&w->v, x_in, B, T, D, D, NULL, NULL, m->theta, NULL, vb);
    /* the block's K/V spikes join the keys at positions ctx..ctx+B-1 */
    for (int b = 0; b < B; ++b)
        for (int t = 0; t < T; ++t)
            for (int d = 0; d < D; ++d) {
                k_cache[idx3(t, ctx + b, d, m->Lmax, D)] = kb[idx3(b, t, d, T, D)];
                v_cache[idx3(t, ctx + b, d, m->Lmax, D)] = vb[idx3(b, t, d, T, D)];
            }
    /* gather keys 0..L-1 into dense [T][L][D] arrays */
    uint8_t* kk = (uint8_t*)malloc((size_t)T * L * D);
    uint8_t* vv = (uint8_t*)malloc((size_t)T * L * D);
    for (int t = 0; t < T; ++t)
        for (int j = 0; j < L; ++j) {
            memcpy(kk + idx3(t, j, 0, L, D), k_cache + idx3(t, j, 0, m->Lmax, D), D);
            memcpy(vv + idx3(t, j, 0, L, D), v_cache + idx3(t, j, 0, m->Lmax, D), D);
        }
    float* acur = (float*)malloc(sizeof(float) * nd);
    orc_attention(q, kk, vv, B, T, L, m->H, m->dh, 1.0 / sqrt((double)m->dh), acur);
    uint8_t* a = (uint8_t*)malloc(nd);
    double* amargin = trace && trace->attn_margin ? trace->attn_margin : NULL;
    orc_if_f32(acur, B, T, D, m->theta, a, NULL, amargin);

    float* u1 = (float*)malloc(sizeof(float) * nd);
    uint8_t* x1 = (uint8_t*)malloc(nd);
    lin_if(&w->o, a, B, T, D, D, u_in, NULL, m->theta, u1, x1);

    uint8_t* hs = (uint8_t*)malloc(nf);
    uint8_t* g = NULL;
    if (m->gated) {
        g = (uint8_t*)malloc(nf);
        lin_if(&w->gate, x1, B, T, D, F, NULL, NULL, m->theta, NULL, g);
        lin_if(&w->up, x1, B, T, D, F, NULL, g, m->theta, NULL, hs);
    } else {
        lin_if(&w->up, x1, B, T, D, F, NULL, NULL, m->theta, NULL, hs);
    }
    lin_if(&w->down, hs, B, T, F, D, u1, NULL, m->theta, u_out, x_out);

    if (trace) {
        if (trace->q) memcpy(trace->q, q, nd);
        if (trace->attn_cur) memcpy(trace->attn_cur, acur, sizeof(float) * nd);
        if (trace->attn) memcpy(trace->attn, a, nd);
        if (trace->u1) memcpy(trace->u1, u1, sizeof(float) * nd);
        if (trace->x1) memcpy(trace->x1, x1, nd);
        if (trace->g && g) memcpy(trace->g, g, nf);
        if (trace->h) memcpy(trace->h, hs, nf);
    }
    free(q); free(kb); free(vb); free(kk); free(vv); free(acur); free(a);
    free(u1); free(x1); free(hs); free(g);
}

/* ----------------------------------------------------- embed, head, unmask ---- */
/* Sec. III-A: the block starts from the embedding of the special mask token at
 * every position; tokens already unmasked contribute their own embedding. */
void orc_embed(const float* tok_emb, const float* pos_emb, const int32_t* tokens, int B,
               int T, int D, int pos0, float* u0) {
    for (int b = 0; b < B; ++b)
        for (int t = 0; t < T; ++t)
            for (int d = 0; d < D; ++d)
                u0[idx3(b, t, d, T, D)] = tok_emb[(size_t)tokens[b] * D + d] +
                                          pos_emb[(size_t)(pos0 + b) * D + d];
}

void orc_head(const uint8_t* x, const int8_t* wT, const float* scale, int B, int T, int D,
              int V, float* logits) {
    int64_t* acc = (int64_t*)malloc(sizeof(int64_t) * (size_t)B * T * V);
    orc_qbsm(x, wT, B * T, D, V, acc);
    for (int b = 0; b < B; ++b)
        for (int v = 0; v < V; ++v) {
            int64_t s = 0;
            for (int t = 0; t < T; ++t) s += acc[idx3(b, t, v, T, V)];
            logits[(size_t)b * V + v] = ((float)s * scale[v]) / (float)T;
        }
    free(acc);
}

/* Sec. III-A: at each denoising step B/S of the still-masked positions are
 * unmasked.  The selection rule is deferred by the paper to block diffusion;
 * reading: greedy by confidence. */
int orc_unmask(const float* logits, int B, int V, int k, int32_t* tokens, uint8_t* mask,
               double* conf, int32_t* tok, int32_t* chosen) {
    double* cf = (double*)malloc(sizeof(double) * (size_t)B);
    int32_t* am = (int32_t*)malloc(sizeof(int32_t) * (size_t)B);
    for (int b = 0; b < B; ++b) {
        const float* l = logits + (size_t)b * V;
        int best = 0;
        for (int v = 1; v < V; ++v)
            if (l[v] > l[best]) best = v;
        double z = 0.0;
        for (int v = 0; v < V; ++v) z += exp((double)l[v] - (double)l[best]);
        cf[b] = 1.0 / z;  /* the largest softmax probability */
        am[b] = best;
        if (conf) conf[b] = cf[b];
        if (tok) tok[b] = best;
    }
    int done = 0;
    for (int r = 0; r < k; ++r) {
        int pick = -1;
        for (int b = 0; b < B; ++b) {
            if (!mask[b]) continue;
            if (pick < 0 || cf[b] > cf[pick]) pick = b;
        }
        if (pick < 0) break;
        tokens[pick] = am[pick];
        mask[pick] = 0;
        if (chosen) chosen[r] = pick;
        ++done;
    }
    free(cf); free(am);
    return done;
}

/* ---------------------------------------------------------------- step ---- */
/* Sec. III-A, Eq. (6): z_{s+1} = f_dec(z_s, h^b) with B/S more tokens unmasked.
 * commit = 1 runs the same layers over the finished block so that its K/V spikes
 * become context for the next block (Eq. (2): p(x^b | x^{<b})). */
int orc_block_step(const orc_model* m, const orc_layer_w* layers, const float* tok_emb,
                   const float* pos_emb, orc_lin head, int32_t* tokens, uint8_t* mask,
                   uint8_t* k_cache, uint8_t* v_cache, int ctx, int commit,
                   float* logits, int32_t* chosen) {
    return orc_block_step_margin(m, layers, tok_emb, pos_emb, head, tokens, mask, k_cache,
                                 v_cache, ctx, commit, logits, chosen, NULL);
}

int orc_block_step_margin(const orc_model* m, const orc_layer_w* layers,
                          const float* tok_emb, const float* pos_emb, orc_lin head,
                          int32_t* tokens, uint8_t* mask, uint8_t* k_cache, uint8_t* v_cache,
                          int ctx, int commit, float* logits, int32_t* chosen,
                          double* attn_margin) {
    int B = m->B, T = m->T, D = m->D;
    size_t nd = (size_t)B * T * D, layer_cache = (size_t)T * m->Lmax * D;
    float* u = (float*)malloc(sizeof(float) * nd);
    float* u2 = (float*)malloc(sizeof(float) * nd);
    uint8_t* x = (uint8_t*)malloc(nd);
    uint8_t* x2 = (uint8_t*)malloc(nd);
    orc_embed(tok_emb, pos_emb, tokens, B, T, D, ctx, u);
    orc_if_f32(u, B, T, D, m->theta, x, NULL, NULL);
    double* margin = (double*)malloc(sizeof(double) * (size_t)B * D);
    orc_layer_trace tr;
    memset(&tr, 0, sizeof(tr));
    tr.attn_margin = margin;
    double min_margin = INFINITY;
    /* Sec. III-A: the shared-layer model runs every layer in both passes; the
     * encoder-decoder model runs its encoders on the context pass and its decoders on
     * the denoising steps */
    int first = 0, count = m->n_layers;
    if (m->n_enc > 0 && commit) count = m->n_enc;
    if (m->n_enc > 0 && !commit) first = m->n_enc;
    for (int l = first; l < first + count; ++l) {
        orc_layer(m, &layers[l], x, u, k_cache + l * layer_cache, v_cache + l * layer_cache,
                  ctx, x2, u2, &tr);
        for (size_t i = 0; i < (size_t)B * D; ++i)
            if (margin[i] < min_margin) min_margin = margin[i];
        uint8_t* tx = x; x = x2; x2 = tx;
        float* tu = u; u = u2; u2 = tu;
    }
    if (m->n_enc > 0 && commit) {
        /* Eq. (5): h = the encoder's output for the block; each decoder layer's context
         * K/V at the block's positions are its own K/V projections of h, through IF */
        uint8_t* kb = (uint8_t*)malloc(nd);
        uint8_t* vb = (uint8_t*)malloc(nd);
        for (int l = 0; l < m->n_layers; ++l) {
            const orc_layer_w* w = &layers[m->n_enc + l];
            lin_if(&w->k, x, B, T, D, D, NULL, NULL, m->theta, NULL, kb);
            lin_if(&w->v, x, B, T, D, D, NULL, NULL, m->theta, NULL, vb);
            uint8_t* kc = k_cache + (size_t)(m->n_enc + l) * layer_cache;
            uint8_t* vc = v_cache + (size_t)(m->n_enc + l) * layer_cache;
            for (int b = 0; b < B; ++b)
                for (int t = 0; t < T; ++t)
                    for (int d = 0; d < D; ++d) {
                        kc[idx3(t, ctx + b, d, m->Lmax, D)] = kb[idx3(b, t, d, T, D)];
                        vc[idx3(t, ctx + b, d, m->Lmax, D)] = vb[idx3(b, t, d, T, D)];
                    }
        }
        free(kb);
        free(vb);
    }
    int done = 0;
    if (!commit) {
        float* lg = logits ? logits : (float*)malloc(sizeof(float) * (size_t)B * m->V);
        orc_head(x, head.w, head.scale, B, T, D, m->V, lg);
        done = orc_unmask(lg, B, m->V, B / m->S, tokens, mask, NULL, NULL, chosen);
        if (!logits) free(lg);
    }
    if (attn_margin) *attn_margin = min_margin;
    free(u); free(u2); free(x); free(x2); free(margin);
    return done;
}

/* ------------------------------------------------- ternary bitwise coding ---- */
/* Sec. II-C (Conversion), Eq. (7)-(8); readings in nmdlm_oracle.h. */
int orc_ternary_planes_needed(int64_t m) {
    int n = 0;
    while (m > 0) {
        ++n;
        m >>= 1;
    }
    return n;
}

/* Sum of |a_i| over one activation row, exact, then rounded once to fp64 (nearest,
 * ties to even).  Every finite fp32 magnitude is an integer m < 2^24 times 2^(e - 149)
 * with 0 <= e <= 253, so the sum is an integer multiple of 2^-149 below 2^308; it is
 * accumulated in ten 32-bit limbs (held in 64-bit words so carries wait until the end).
 * A NaN gives NaN and an infinity +Inf, as an fp64 running sum would. */
double orc_abs_sum_exact(const float* row, int D) {
    uint64_t limb[11];
    int nan = 0, inf = 0;
    memset(limb, 0, sizeof(limb));
    for (int i = 0; i < D; ++i) {
        float x = fabsf(row[i]);
        uint32_t bits;
        memcpy(&bits, &x, sizeof(bits));
        uint32_t ex = bits >> 23, man = bits & 0x7FFFFFu;
        if (ex == 255) {
            if (man) nan = 1; else inf = 1;
            continue;
        }
        uint64_t m = ex ? (uint64_t)(man | 0x800000u) : (uint64_t)man;
        int sh = ex ? (int)ex - 1 : 0; /* value = m * 2^sh * 2^-149 */
        uint64_t part = m << (sh % 32);   /* < 2^55: spans limbs sh/32 and sh/32 + 1 */
        limb[sh / 32] += part & 0xFFFFFFFFu;
        limb[sh / 32 + 1] += part >> 32;
    }
    if (nan) return NAN;
    if (inf) return INFINITY;
    for (int j = 0; j < 10; ++j) {
        limb[j + 1] += limb[j] >> 32;
        limb[j] &= 0xFFFFFFFFu;
    }
    int top = -1; /* highest set bit of the integer */
    for (int j = 10; j >= 0 && top < 0; --j)
        if (limb[j]) {
            int b = 31;
            while (!((limb[j] >> b) & 1u)) --b;
            top = 32 * j + b;
        }
    if (top < 0) return 0.0;
    /* the 53 bits from `top` down, the next bit, and whether any lower bit is set */
    uint64_t mant = 0;
    int lsb = top - 52; /* bit position of the last kept bit (may be negative) */
    for (int b = top; b >= lsb && b >= 0; --b)
        mant = (mant << 1) | ((limb[b / 32] >> (b % 32)) & 1u);
    if (lsb < 0) return ldexp((double)mant, -149); /* fewer than 54 significant bits: exact */
    int round = lsb > 0 ? (int)((limb[(lsb - 1) / 32] >> ((lsb - 1) % 32)) & 1u) : 0;
    int sticky = 0;
    for (int b = lsb - 2; b >= 0 && !sticky; --b)
        if ((limb[b / 32] >> (b % 32)) & 1u) sticky = 1;
    if (round && (sticky || (mant & 1u))) mant += 1;
    return ldexp((double)mant, lsb - 149);
}

void orc_ternary_encode(const float* a, int N, int D, float K, int T, int8_t* s,
                        int32_t* ahat, float* vth) {
    assert(T >= 1 && T <= 30 && K > 0.0f);
    const int64_t cap = ((int64_t)1 << T) - 1;
    for (int n = 0; n < N; ++n) {
        const float* row = a + (size_t)n * D;
        /* Eq. (7): V_th(a) = mean(|a|) / K; the sum of |a| taken exactly (reading: the
         * quantisation decides integers, so its step must not depend on an order of
         * summation), then mean and step in fp64, rounded once to fp32 */
        const double sum = orc_abs_sum_exact(row, D);
        const double mean = sum / (double)D;
        const float v = (float)(mean / (double)K);
        if (vth) vth[n] = v;
        for (int i = 0; i < D; ++i) {
            int64_t q = 0;
            if (v > 0.0f) {
                const float x = row[i] / v; /* one fp32 division */
                if (x == x) {               /* NaN quantises to 0 */
                    const float r = roundf(x);   /* halves away from zero */
                    if (r >= (float)cap) q = cap;
                    else if (r <= -(float)cap) q = -cap;
                    else q = (int64_t)r;
                }
            }
            if (ahat) ahat[(size_t)n * D + i] = (int32_t)q;
            /* Eq. (8): q = sum_t 2^{t-1} s_t with s_t = sign(q) * bit (t-1) of |q| */
            const int64_t mag = q < 0 ? -q : q;
            const int sg = q < 0 ? -1 : 1;
            for (int t = 0; t < T; ++t)
                s[idx3(n, t, i, T, D)] = (int8_t)(((mag >> t) & 1) ? sg : 0);
        }
    }
}

void orc_ternary_linear(const int8_t* s, const int8_t* wT, int N, int T, int D, int d_out,
                        int64_t* I, int64_t* y) {
    for (int n = 0; n < N; ++n) {
        for (int o = 0; o < d_out; ++o) {
            int64_t total = 0;
            for (int t = 0; t < T; ++t) {
                int64_t cur = 0; /* I_t[o] = sum_i W^T[i][o] s_{i,t} */
                for (int i = 0; i < D; ++i)
                    cur += (int64_t)wT[(size_t)i * d_out + o] * s[idx3(n, t, i, T, D)];
                if (I) I[idx3(n, t, o, T, d_out)] = cur;
                total += cur * ((int64_t)1 << t); /* weight 2^{t-1}, t counted from 1 */
            }
            y[(size_t)n * d_out + o] = total;
        }
    }
}

/* Sec. II-C, Eq. (9)-(10) as read in nmdlm_oracle.h: integrate the bit-weighted input
 * (given as y), then emit ternary spikes from the most significant step down. */
void orc_ternary_if(const int64_t* y, int N, int d_out, int T, int64_t theta, int8_t* s_out,
                    int64_t* v_final) {
    assert(T >= 1 && T <= 30 && theta >= 1);
    for (int n = 0; n < N; ++n)
        for (int o = 0; o < d_out; ++o) {
            int64_t v = y[(size_t)n * d_out + o];
            for (int t = T; t >= 1; --t) {
                const int64_t thr = ((int64_t)1 << (t - 1)) * theta;
                int8_t s = 0;
                if (v >= thr) s = 1;
                else if (v <= -thr) s = -1;
                v -= thr * s;
                s_out[idx3(n, t - 1, o, T, d_out)] = s;
            }
            if (v_final) v_final[(size_t)n * d_out + o] = v;
        }
}
