/*
 * CPU oracle for the Hierarchical Sparse Attention (HSA) hot path.
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product path may load, link or call
 * this file: only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline
 * leg (and `bench.py --impl reference`) use it, through oracle/__init__.py. It
 * shares no code with the CUDA library.
 *
 * Plain, slow, obviously correct loops that follow the paper's statement of
 * the operator (arXiv 2504.16795):
 *   - chunk summary  K̄_i = mean of the S keys of chunk i       (§3.1 "Chunk
 *     Selection"; Appendix A, Eq. 3: q·K̄ equals the mean of the token logits)
 *   - selection score s_{t,i} = c_sel * q̂_t · K̄_i over causally visible chunks,
 *     top-k by rank                                            (§3.1 "Chunk Selection")
 *   - selected indices ordered by decreasing chunk index (I')  (§3.1.1 "Chunk Weights")
 *   - chunk weights w = softmax over the selected scores        (§4.1 "Ablation
 *     Studies", the "w/o s.b." variant: softmax instead of stick-breaking),
 *     or, with `stick`, the paper's default stick-breaking weights over I'
 *     (§3.1.1 "Chunk Weights"): w_k = sigmoid(s_k) * prod_{i<k} (1 - sigmoid(s_i))
 *   - token-level attention inside every selected chunk and the weighted sum
 *     over chunks                                              (§3.1.1 "Hierarchical
 *     Attention"; Algorithm 1); plain softmax inside a chunk, or with
 *     `softmax1` the softmax-off-by-one of §3.1.2 "Kernel Design" (a zero logit
 *     joins the denominator, so a token may give a chunk little weight)
 *   - gradients into q, K, V (Algorithms 2 and 3) and, through w, into the
 *     selection scores, K̄ and K (Appendix A: the scores receive gradients
 *     because w takes part in the forward pass)
 *
 * Readings where the paper leaves a convention open:
 *   - token t (0-indexed) sees only completed chunks before its own: i < t / S;
 *   - fewer than k visible chunks: all are selected, the rest padded with -1;
 *     zero visible chunks give O = 0 and no gradient;
 *   - the group score sums the G query heads of the group: q̂_t = sum_h q_{t,h}
 *     (K̂ is K̄ repeated over the heads), scaled by c_sel = 1/sqrt(G*d) unless
 *     the caller gives another scale;
 *   - inner attention uses plain softmax with scale c_att = 1/sqrt(d);
 *   - equal scores rank the lower chunk index first.
 *
 * Precision. Everything is fp64 (inputs are widened exactly from bf16), except
 * that when `f32` is set the chunk summaries and the selection scores are
 * computed in fp32 with the summation order the definition gives (token order
 * for the mean, head order for q̂, dimension order with a fused multiply-add
 * chain for the dot product). That is the precision in which the CUDA kernels
 * take the top-k decision, so the integer result is compared exactly.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
    double s;
    int64_t i;
} scored_t;

/* rank order of §3.1: larger score first, equal scores by lower chunk index */
static int rank_order(const void* pa, const void* pb) {
    const scored_t* a = (const scored_t*)pa;
    const scored_t* b = (const scored_t*)pb;
    if (a->s > b->s) return -1;
    if (a->s < b->s) return 1;
    return (a->i < b->i) ? -1 : (a->i > b->i) ? 1 : 0;
}

/* I' of §3.1.1: decreasing chunk index */
static int chunk_index_descending(const void* pa, const void* pb) {
    const scored_t* a = (const scored_t*)pa;
    const scored_t* b = (const scored_t*)pb;
    return (a->i > b->i) ? -1 : (a->i < b->i) ? 1 : 0;
}

static inline int64_t at4(int64_t i0, int64_t i1, int64_t i2, int64_t i3, int64_t n1, int64_t n2, int64_t n3) {
    return ((i0 * n1 + i1) * n2 + i2) * n3 + i3;
}

int hsa_oracle_version(void) { return 1; }

#ifdef _OPENMP
#include <omp.h>
int hsa_oracle_threads(void) { return omp_get_max_threads(); }
#else
int hsa_oracle_threads(void) { return 1; }
#endif

/* ------------------------------------------------------------------ chunk mean pool
 * K [B, L, Hkv, d] -> kbar [B, L/S, Hkv, d]; kbar_i = (1/S) sum_{s<S} K_{iS+s}.
 */
void hsa_oracle_pool(const double* K, int B, int L, int Hkv, int d, int S, int f32, double* kbar) {
    const int Nc = L / S;
#pragma omp parallel for collapse(2) schedule(static)
    for (int b = 0; b < B; ++b)
        for (int i = 0; i < Nc; ++i)
            for (int g = 0; g < Hkv; ++g)
                for (int e = 0; e < d; ++e) {
                    double out;
                    if (f32) {
                        float acc = 0.0f;
                        for (int s = 0; s < S; ++s) acc = acc + (float)K[at4(b, (int64_t)i * S + s, g, e, L, Hkv, d)];
                        out = (double)(acc / (float)S);
                    } else {
                        double acc = 0.0;
                        for (int s = 0; s < S; ++s) acc += K[at4(b, (int64_t)i * S + s, g, e, L, Hkv, d)];
                        out = acc / (double)S;
                    }
                    kbar[at4(b, i, g, e, Nc, Hkv, d)] = out;
                }
}

/* One selection row: scores over chunks 0..nvis-1 for the group vector q̂,
 * ranked, cut to k_eff, reordered by decreasing index. */
static void select_row(const double* qhat, const double* kbar_g, int64_t kbar_stride, int64_t nvis, int d,
                       int topk, double scale_sel, int f32, scored_t* work, int32_t* idx_out,
                       double* s_out, double* gap_out) {
    for (int64_t i = 0; i < nvis; ++i) {
        const double* kb = kbar_g + i * kbar_stride;
        double s;
        if (f32) {
            float acc = 0.0f;
            for (int e = 0; e < d; ++e) acc = fmaf((float)qhat[e], (float)kb[e], acc);
            s = (double)(acc * (float)scale_sel);
        } else {
            double acc = 0.0;
            for (int e = 0; e < d; ++e) acc += qhat[e] * kb[e];
            s = acc * scale_sel;
        }
        work[i].s = s;
        work[i].i = i;
    }
    qsort(work, (size_t)nvis, sizeof(scored_t), rank_order);
    const int64_t keff = nvis < topk ? nvis : topk;
    if (gap_out) *gap_out = (keff > 0 && nvis > keff) ? work[keff - 1].s - work[keff].s : INFINITY;
    qsort(work, (size_t)keff, sizeof(scored_t), chunk_index_descending);
    for (int j = 0; j < topk; ++j) {
        if (j < keff) {
            idx_out[j] = (int32_t)work[j].i;
            s_out[j] = work[j].s;
        } else {
            idx_out[j] = -1;
            s_out[j] = -INFINITY;
        }
    }
}

/* group vector q̂_t of §3.1 for the heads [g*G, (g+1)*G) */
static void group_query(const double* q_row, int G, int g, int d, int f32, double* qhat) {
    for (int e = 0; e < d; ++e) {
        if (f32) {
            float acc = 0.0f;
            for (int hh = 0; hh < G; ++hh) acc = acc + (float)q_row[(int64_t)(g * G + hh) * d + e];
            qhat[e] = (double)acc;
        } else {
            double acc = 0.0;
            for (int hh = 0; hh < G; ++hh) acc += q_row[(int64_t)(g * G + hh) * d + e];
            qhat[e] = acc;
        }
    }
}

/* ------------------------------------------------------------------ chunk selection
 * q [B, L, Hq, d], kbar [B, L/S, Hkv, d] -> idx [B, L, Hkv, topk] int32,
 * s_sel [B, L, Hkv, topk]; gap (optional) [B, L, Hkv] = k-th minus (k+1)-th score.
 * token_mask (optional, [B, L]): only rows whose mask byte is nonzero are computed.
 */
void hsa_oracle_select(const double* q, const double* kbar, int B, int L, int Hq, int Hkv, int d, int S,
                       int topk, double scale_sel, int f32, const uint8_t* token_mask, int32_t* idx, double* s_sel,
                       double* gap) {
    const int Nc = L / S, G = Hq / Hkv;
#pragma omp parallel
    {
        scored_t* work = (scored_t*)malloc(sizeof(scored_t) * (size_t)(Nc > 0 ? Nc : 1));
        double* qhat = (double*)malloc(sizeof(double) * (size_t)d);
#pragma omp for collapse(2) schedule(dynamic, 16)
        for (int b = 0; b < B; ++b)
            for (int t = 0; t < L; ++t) {
                if (token_mask && !token_mask[(int64_t)b * L + t]) continue;
                const int64_t nvis = (t / S) < Nc ? (t / S) : Nc;
                const double* q_row = q + at4(b, t, 0, 0, L, Hq, d);
                for (int g = 0; g < Hkv; ++g) {
                    group_query(q_row, G, g, d, f32, qhat);
                    const int64_t o = at4(b, t, g, 0, L, Hkv, topk);
                    select_row(qhat, kbar + at4(b, 0, g, 0, Nc, Hkv, d), (int64_t)Hkv * d, nvis, d, topk, scale_sel,
                               f32, work, idx + o, s_sel + o, gap ? gap + at4(b, t, g, 0, L, Hkv, 1) : NULL);
                }
            }
        free(work);
        free(qhat);
    }
}

/* number of leading valid indices of one selection row */
static int count_selected(const int32_t* I, int topk) {
    int k = 0;
    while (k < topk && I[k] >= 0) ++k;
    return k;
}

static double sigmoid(double x) { return 1.0 / (1.0 + exp(-x)); }

/* chunk weights over the k_eff selected scores, slots in I' order (decreasing
 * chunk index): softmax, or (stick) stick-breaking — slot k takes the fraction
 * sigmoid(s_k) of what the slots before it left of a unit stick */
static void chunk_weights(const double* s, int keff, int topk, int stick, double* w) {
    if (stick) {
        double rest = 1.0;
        for (int j = 0; j < topk; ++j) {
            if (j < keff) {
                const double beta = sigmoid(s[j]);
                w[j] = beta * rest;
                rest *= 1.0 - beta;
            } else {
                w[j] = 0.0;
            }
        }
        return;
    }
    double m = -INFINITY, z = 0.0;
    for (int j = 0; j < keff; ++j) m = s[j] > m ? s[j] : m;
    for (int j = 0; j < keff; ++j) z += exp(s[j] - m);
    for (int j = 0; j < topk; ++j) w[j] = j < keff ? exp(s[j] - m) / z : 0.0;
}

/* token-level attention of one query head over one chunk: P (S) and O_j (d);
 * softmax1: the denominator also holds exp(0) (softmax-off-by-one) */
static void chunk_attention(const double* qh, const double* Kc, const double* Vc, int64_t row_stride, int d, int S,
                            double scale_attn, int softmax1, double* P, double* Oj) {
    double m = -INFINITY, z = 0.0;
    for (int s = 0; s < S; ++s) {
        double a = 0.0;
        for (int e = 0; e < d; ++e) a += qh[e] * Kc[(int64_t)s * row_stride + e];
        P[s] = scale_attn * a;
        m = P[s] > m ? P[s] : m;
    }
    for (int s = 0; s < S; ++s) {
        P[s] = exp(P[s] - m);
        z += P[s];
    }
    if (softmax1) z += exp(-m);
    for (int s = 0; s < S; ++s) P[s] /= z;
    for (int e = 0; e < d; ++e) {
        double acc = 0.0;
        for (int s = 0; s < S; ++s) acc += P[s] * Vc[(int64_t)s * row_stride + e];
        Oj[e] = acc;
    }
}

/* ------------------------------------------------------------------ forward
 * O [B, L, Hq, d] = sum_j w_j Attn(q_t, K_{I_j}, V_{I_j}); w [B, L, Hkv, topk].
 * token_mask (optional, [B, L]): only those tokens are computed.
 */
void hsa_oracle_forward(const double* q, const double* K, const double* V, const int32_t* idx,
                        const double* s_sel, int B, int L, int Hq, int Hkv, int d, int S, int topk,
                        double scale_attn, int softmax1, int stick, const uint8_t* token_mask, double* O, double* w) {
    const int G = Hq / Hkv;
#pragma omp parallel
    {
        double* P = (double*)malloc(sizeof(double) * (size_t)S);
        double* Oj = (double*)malloc(sizeof(double) * (size_t)d);
#pragma omp for collapse(2) schedule(dynamic, 16)
        for (int b = 0; b < B; ++b)
            for (int t = 0; t < L; ++t)
                for (int g = 0; g < Hkv; ++g) {
                    if (token_mask && !token_mask[(int64_t)b * L + t]) continue;
                    const int64_t o = at4(b, t, g, 0, L, Hkv, topk);
                    const int keff = count_selected(idx + o, topk);
                    chunk_weights(s_sel + o, keff, topk, stick, w + o);
                    for (int hh = 0; hh < G; ++hh) {
                        const int h = g * G + hh;
                        const double* qh = q + at4(b, t, h, 0, L, Hq, d);
                        double* Oh = O + at4(b, t, h, 0, L, Hq, d);
                        for (int e = 0; e < d; ++e) Oh[e] = 0.0;
                        for (int j = 0; j < keff; ++j) {
                            const int64_t i = idx[o + j];
                            const double* Kc = K + at4(b, i * S, g, 0, L, Hkv, d);
                            const double* Vc = V + at4(b, i * S, g, 0, L, Hkv, d);
                            chunk_attention(qh, Kc, Vc, (int64_t)Hkv * d, d, S, scale_attn, softmax1, P, Oj);
                            for (int e = 0; e < d; ++e) Oh[e] += w[o + j] * Oj[e];
                        }
                    }
                }
        free(P);
        free(Oj);
    }
}

/* ------------------------------------------------------------------ backward
 * Given dO = dℒ/dO, returns dq [B,L,Hq,d], dK, dV [B,L,Hkv,d]; optionally
 * dkbar [B,L/S,Hkv,d] (gradient reaching the chunk summaries) and
 * ds [B,L,Hkv,topk] (gradient reaching the selected scores).
 *
 * Chain (per token t, group g, selected slot j, head h, chunk row s):
 *   D_{h,j}  = dO_h · O_{h,j}                       (Algorithm 2: rowsum(O' ∘ ∇O'))
 *   dw_j     = sum_h D_{h,j}                          (Algorithm 2: ∇w = rowsum(D'))
 *   dP_s     = w_j dO_h · V_s ;  sum_s P_s dP_s = w_j D_{h,j}
 *   da_s     = P_s (dP_s - w_j D_{h,j})               (Algorithm 2/3: ∇S = wP∘(∇P - D'))
 *   dq_h    += c_att sum_s da_s K_s ; dK_s += c_att da_s q_h ; dV_s += w_j P_s dO_h
 *   ds_j     = w_j (dw_j - sum_j' w_j' dw_j')        (softmax over the selected scores)
 *   ds_j     = (1 - b_j) w_j dw_j - b_j sum_{k>j} w_k dw_k,  b = sigmoid(s)
 *                                                     (stick-breaking: w_k = b_k prod_{i<k} (1 - b_i))
 *   dq_h    += c_sel sum_j ds_j K̄_{I_j} (every head of the group) ; dK̄_{I_j} += c_sel ds_j q̂
 *   dK_{iS+s} += dK̄_i / S                             (mean pool)
 * token_mask (optional, [B, L]): only those tokens are processed, so dq rows
 * of other tokens stay 0 and dK, dV, dK̄ collect the masked tokens'
 * contributions only (exact for a chunk whose selecting tokens are all in
 * the mask).
 */
void hsa_oracle_backward(const double* q, const double* K, const double* V, const double* kbar,
                         const int32_t* idx, const double* s_sel, const double* dO, int B, int L, int Hq,
                         int Hkv, int d, int S, int topk, double scale_sel, double scale_attn, int softmax1,
                         int stick, const uint8_t* token_mask, double* dq, double* dK, double* dV, double* dkbar,
                         double* ds) {
    const int G = Hq / Hkv, Nc = L / S;
#pragma omp parallel for collapse(2) schedule(dynamic, 1)
    for (int b = 0; b < B; ++b)
        for (int g = 0; g < Hkv; ++g) {
            double* P = (double*)malloc(sizeof(double) * (size_t)G * topk * S);
            double* Oj = (double*)malloc(sizeof(double) * (size_t)G * topk * d);
            double* D = (double*)malloc(sizeof(double) * (size_t)G * topk);
            double* w = (double*)malloc(sizeof(double) * (size_t)topk);
            double* dw = (double*)malloc(sizeof(double) * (size_t)topk);
            double* dsl = (double*)malloc(sizeof(double) * (size_t)topk);
            double* qhat = (double*)malloc(sizeof(double) * (size_t)d);
            double* dkb = (double*)calloc((size_t)(Nc > 0 ? Nc : 1) * d, sizeof(double));
            for (int t = 0; t < L; ++t)
                for (int e = 0; e < d; ++e) {
                    dK[at4(b, t, g, e, L, Hkv, d)] = 0.0;
                    dV[at4(b, t, g, e, L, Hkv, d)] = 0.0;
                }
            for (int t = 0; t < L; ++t) {
                if (token_mask && !token_mask[(int64_t)b * L + t]) continue;
                const int64_t o = at4(b, t, g, 0, L, Hkv, topk);
                const int32_t* I = idx + o;
                const int keff = count_selected(I, topk);
                for (int hh = 0; hh < G; ++hh)
                    for (int e = 0; e < d; ++e) dq[at4(b, t, g * G + hh, e, L, Hq, d)] = 0.0;
                if (ds)
                    for (int j = 0; j < topk; ++j) ds[o + j] = 0.0;
                if (keff == 0) continue;
                chunk_weights(s_sel + o, keff, topk, stick, w);
                /* recompute the forward quantities of Algorithm 1 */
                for (int j = 0; j < keff; ++j) dw[j] = 0.0;
                for (int hh = 0; hh < G; ++hh) {
                    const double* qh = q + at4(b, t, g * G + hh, 0, L, Hq, d);
                    const double* dOh = dO + at4(b, t, g * G + hh, 0, L, Hq, d);
                    for (int j = 0; j < keff; ++j) {
                        const int64_t i = I[j];
                        double* Pj = P + ((size_t)hh * topk + j) * S;
                        double* Ojh = Oj + ((size_t)hh * topk + j) * d;
                        chunk_attention(qh, K + at4(b, i * S, g, 0, L, Hkv, d), V + at4(b, i * S, g, 0, L, Hkv, d),
                                        (int64_t)Hkv * d, d, S, scale_attn, softmax1, Pj, Ojh);
                        double acc = 0.0;
                        for (int e = 0; e < d; ++e) acc += dOh[e] * Ojh[e];
                        D[hh * topk + j] = acc;
                        dw[j] += acc;
                    }
                }
                if (stick) {
                    double later = 0.0; /* sum_{k>j} w_k dw_k */
                    for (int j = keff - 1; j >= 0; --j) {
                        const double beta = sigmoid(s_sel[o + j]);
                        dsl[j] = (1.0 - beta) * w[j] * dw[j] - beta * later;
                        later += w[j] * dw[j];
                    }
                } else {
                    double wdw = 0.0;
                    for (int j = 0; j < keff; ++j) wdw += w[j] * dw[j];
                    for (int j = 0; j < keff; ++j) dsl[j] = w[j] * (dw[j] - wdw);
                }
                group_query(q + at4(b, t, 0, 0, L, Hq, d), G, g, d, 0, qhat);
                for (int hh = 0; hh < G; ++hh) {
                    const int h = g * G + hh;
                    const double* qh = q + at4(b, t, h, 0, L, Hq, d);
                    const double* dOh = dO + at4(b, t, h, 0, L, Hq, d);
                    double* dqh = dq + at4(b, t, h, 0, L, Hq, d);
                    for (int j = 0; j < keff; ++j) {
                        const int64_t i = I[j];
                        const double* Pj = P + ((size_t)hh * topk + j) * S;
                        const double Dhj = D[hh * topk + j];
                        for (int s = 0; s < S; ++s) {
                            const int64_t row = at4(b, i * S + s, g, 0, L, Hkv, d);
                            double dOV = 0.0;
                            for (int e = 0; e < d; ++e) dOV += dOh[e] * V[row + e];
                            const double dP = w[j] * dOV;
                            const double da = Pj[s] * (dP - w[j] * Dhj);
                            for (int e = 0; e < d; ++e) {
                                dqh[e] += scale_attn * da * K[row + e];
                                dK[row + e] += scale_attn * da * qh[e];
                                dV[row + e] += w[j] * Pj[s] * dOh[e];
                            }
                        }
                        for (int e = 0; e < d; ++e)
                            dqh[e] += scale_sel * dsl[j] * kbar[at4(b, i, g, e, Nc, Hkv, d)];
                    }
                }
                for (int j = 0; j < keff; ++j) {
                    const int64_t i = I[j];
                    for (int e = 0; e < d; ++e) dkb[(size_t)i * d + e] += scale_sel * dsl[j] * qhat[e];
                    if (ds) ds[o + j] = dsl[j];
                }
            }
            for (int i = 0; i < Nc; ++i)
                for (int e = 0; e < d; ++e) {
                    const double share = dkb[(size_t)i * d + e] / (double)S;
                    for (int s = 0; s < S; ++s) dK[at4(b, (int64_t)i * S + s, g, e, L, Hkv, d)] += share;
                    if (dkbar) dkbar[at4(b, i, g, e, Nc, Hkv, d)] = dkb[(size_t)i * d + e];
                }
            free(P);
            free(Oj);
            free(D);
            free(w);
            free(dw);
            free(dsl);
            free(qhat);
            free(dkb);
        }
}

/* ------------------------------------------------------------------ selection backward
 * The selection chain alone, for a given score gradient ds [B,L,Hkv,topk]
 * (Appendix A: the scores s = c_sel q̂·K̄ receive gradient through the chunk
 * weights; several layers sharing one selection add their ds first):
 *   dq_h    = c_sel sum_j ds_j K̄_{I_j}         (every head h of the group)
 *   dK̄_i    = c_sel sum_{(t,j): I_j = i} ds_j q̂_t
 *   dK_{iS+s} = dK̄_i / S                       (mean pool); other rows 0
 */
void hsa_oracle_select_backward(const double* q, const double* kbar, const int32_t* idx, const double* ds, int B,
                                int L, int Hq, int Hkv, int d, int S, int topk, double scale_sel, double* dq,
                                double* dK, double* dkbar) {
    const int G = Hq / Hkv, Nc = L / S;
    for (int64_t u = 0; u < (int64_t)B * L * Hq * d; ++u) dq[u] = 0.0;
    for (int64_t u = 0; u < (int64_t)B * L * Hkv * d; ++u) dK[u] = 0.0;
    for (int64_t u = 0; u < (int64_t)B * Nc * Hkv * d; ++u) dkbar[u] = 0.0;
    double* qhat = (double*)malloc(sizeof(double) * (size_t)d);
    for (int b = 0; b < B; ++b)
        for (int t = 0; t < L; ++t)
            for (int g = 0; g < Hkv; ++g) {
                const int64_t o = at4(b, t, g, 0, L, Hkv, topk);
                const int keff = count_selected(idx + o, topk);
                if (keff == 0) continue;
                group_query(q + at4(b, t, 0, 0, L, Hq, d), G, g, d, 0, qhat);
                for (int j = 0; j < keff; ++j) {
                    const int64_t i = idx[o + j];
                    for (int hh = 0; hh < G; ++hh)
                        for (int e = 0; e < d; ++e)
                            dq[at4(b, t, g * G + hh, e, L, Hq, d)] += scale_sel * ds[o + j] * kbar[at4(b, i, g, e, Nc, Hkv, d)];
                    for (int e = 0; e < d; ++e) dkbar[at4(b, i, g, e, Nc, Hkv, d)] += scale_sel * ds[o + j] * qhat[e];
                }
            }
    for (int b = 0; b < B; ++b)
        for (int i = 0; i < Nc; ++i)
            for (int g = 0; g < Hkv; ++g)
                for (int e = 0; e < d; ++e)
                    for (int s = 0; s < S; ++s)
                        dK[at4(b, (int64_t)i * S + s, g, e, L, Hkv, d)] = dkbar[at4(b, i, g, e, Nc, Hkv, d)] / (double)S;
    free(qhat);
}

/* ------------------------------------------------------------------ decode
 * One query token per batch row sitting right after a memory of Nc complete
 * chunks (§3.2 "Inference": only the chunk summaries are scanned, then the k
 * selected chunks are fetched). All Nc chunks are visible.
 *   q [Bq, Hq, d], kbar [Nc, Hkv, d] -> idx, s_sel [Bq, Hkv, topk], gap [Bq, Hkv]
 */
void hsa_oracle_decode_select(const double* q, const double* kbar, int64_t Nc, int Bq, int Hq, int Hkv, int d,
                              int topk, double scale_sel, int f32, int32_t* idx, double* s_sel, double* gap) {
    const int G = Hq / Hkv;
#pragma omp parallel
    {
        scored_t* work = (scored_t*)malloc(sizeof(scored_t) * (size_t)(Nc > 0 ? Nc : 1));
        double* qhat = (double*)malloc(sizeof(double) * (size_t)d);
#pragma omp for collapse(2) schedule(dynamic, 1)
        for (int b = 0; b < Bq; ++b)
            for (int g = 0; g < Hkv; ++g) {
                group_query(q + (int64_t)b * Hq * d, G, g, d, f32, qhat);
                const int64_t o = ((int64_t)b * Hkv + g) * topk;
                select_row(qhat, kbar + (int64_t)g * d, (int64_t)Hkv * d, Nc, d, topk, scale_sel, f32, work,
                           idx + o, s_sel + o, gap ? gap + (int64_t)b * Hkv + g : NULL);
            }
        free(work);
        free(qhat);
    }
}

/* Attention of the decode queries over their selected chunks.
 * Ksel, Vsel [Bq, Hkv, topk, S, d] hold the rows of chunk idx[b, g, j] (any
 * content where idx = -1). -> w [Bq, Hkv, topk], O [Bq, Hq, d]. */
void hsa_oracle_decode_attend(const double* q, const double* Ksel, const double* Vsel, const int32_t* idx,
                              const double* s_sel, int Bq, int Hq, int Hkv, int d, int S, int topk,
                              double scale_attn, int softmax1, int stick, double* w, double* O) {
    const int G = Hq / Hkv;
#pragma omp parallel
    {
        double* P = (double*)malloc(sizeof(double) * (size_t)S);
        double* Oj = (double*)malloc(sizeof(double) * (size_t)d);
#pragma omp for collapse(2) schedule(dynamic, 1)
        for (int b = 0; b < Bq; ++b)
            for (int g = 0; g < Hkv; ++g) {
                const int64_t o = ((int64_t)b * Hkv + g) * topk;
                const int keff = count_selected(idx + o, topk);
                chunk_weights(s_sel + o, keff, topk, stick, w + o);
                for (int hh = 0; hh < G; ++hh) {
                    const int h = g * G + hh;
                    const double* qh = q + ((int64_t)b * Hq + h) * d;
                    double* Oh = O + ((int64_t)b * Hq + h) * d;
                    for (int e = 0; e < d; ++e) Oh[e] = 0.0;
                    for (int j = 0; j < keff; ++j) {
                        const int64_t base = ((o + j) * S) * (int64_t)d;
                        chunk_attention(qh, Ksel + base, Vsel + base, d, d, S, scale_attn, softmax1, P, Oj);
                        for (int e = 0; e < d; ++e) Oh[e] += w[o + j] * Oj[e];
                    }
                }
            }
        free(P);
        free(Oj);
    }
}
