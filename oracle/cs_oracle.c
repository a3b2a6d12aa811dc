/*
 * cs_oracle.c -- plain, slow, fp64 CPU oracle for the draft-and-verify step.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference leg of bench.py may load this library.  It shares
 * no code, header, table or helper with the CUDA path; the two only see the
 * same seeded inputs.
 *
 * What it computes.  In the paper's cache-miss branch (Sec. 3.4) the target
 * LLM generates while the small model drafts tokens for it, and the target
 * verifies them with the standard speculative-sampling draft-and-verify step
 * (also named in Sec. 2 and App. A.4).  The paper gives no formula of its
 * own and defers the rule to the two speculative-sampling works it cites;
 * the rule below is that standard one:
 *
 *   1. Verify attention: for each request b, query head h and draft row
 *      i in [0, k], softmax over keys j <= L_b-(k+1)+i of q.K_j*scale, times V.
 *      Plain definition written out: scores, max, exp, sum, weighted sum.
 *   2. Speculative acceptance (temperature T > 0): p_i = softmax(z_t,i / T),
 *      q_i = softmax(z_d,i / T); accept x_i iff u_i < p_i(x_i)/q_i(x_i);
 *      a = first rejected position (k if none); on rejection draw from
 *      max(0, p_a - q_a) normalised, else draw the bonus token from p_k;
 *      the draw is the inverse CDF in ascending token id with uniform u_k.
 *   3. Greedy (T == 0): g_i = argmax z_t,i (lowest id on ties); accept x_i
 *      iff x_i == g_i; emit g_a.
 *   4. Draft-side sampling (the drafter's per-position step before the
 *      verify pass): x = inverse CDF of softmax(z / T) at u, ascending token
 *      id, the computed total as the normaliser; T == 0 takes the argmax.
 *   6. Semantic routing (Sec. 3.1): the score of request x against group G_i
 *      is the cosine similarity of its embedding with the group's centroid;
 *      i* = argmax_i (lowest i on ties); a score below tau sends x to the
 *      cache-miss branch (group -1).
 *   5. Paged KV cache: the k+1 verify positions' K/V rows go to key
 *      positions L_b-(k+1) .. L_b-1 of their request (slot pos % ps of page
 *      page_table[b][pos / ps]); after the acceptance step the context keeps
 *      L_b - k + a rows (the prefix, the verify input token and the a
 *      accepted drafts).
 *   7. Token-tree verification (Sec. 2's multi-candidate variants): the
 *      attention of section 1 with each node seeing the prefix and its own
 *      ancestors; the walk that tests the children of each node in turn
 *      against the running residual (multi-candidate speculative
 *      sampling); the commit that moves the accepted path's K/V rows next
 *      to the root.
 *
 * Every floating-point step is fp64; inputs (bf16 bit patterns or fp32) are
 * widened exactly.  Loops run in the order the definition states (ascending
 * key index, ascending token id); OpenMP only splits independent requests /
 * heads across threads and never changes any sum's order.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_OK 0
#define ORC_BAD_ARG 1
#define ORC_NO_MEM 2

/* bf16 is the upper 16 bits of an IEEE binary32; widening is exact. */
static double bf16_bits_to_double(uint16_t bits) {
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Element `idx` of a logit row stored as fp32 (dtype 0) or bf16 (dtype 1). */
static double logit_at(const void* row, int32_t dtype, int64_t idx) {
    if (dtype == 0) return (double)((const float*)row)[idx];
    return bf16_bits_to_double(((const uint16_t*)row)[idx]);
}

int oracle_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oracle_set_threads(int n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* ------------------------------------------------------------------------
 * 1. Verify attention over a paged KV cache.
 *
 * q        [B, k+1, Hq, D]   bf16 bits
 * k_pages  [P, Hkv, ps, D]   bf16 bits
 * v_pages  [P, Hkv, ps, D]   bf16 bits
 * page_table [B, max_pages]  int32; key j of request b lives in page
 *                            page_table[b][j / ps] at slot j % ps
 * ctx_lens [B]               int32; L_b counts the k+1 verify positions and
 *                            is clamped to [0, max_pages*ps]
 * out      [B, k+1, Hq, D]   fp64
 *
 * Query head h reads KV head h / G with G = Hq / Hkv (consecutive query
 * heads share one KV head).  A page id outside [0, P) reads as zeros.
 * A row with no admissible key (L_b - (k+1) + i < 0) outputs zeros.
 * scale <= 0 selects 1/sqrt(D).
 * ---------------------------------------------------------------------- */
int oracle_verify_attention(int32_t batch, int32_t n_q_heads, int32_t n_kv_heads,
                            int32_t head_dim, int32_t page_size,
                            int32_t max_pages_per_seq, int32_t num_pages,
                            double scale, const uint16_t* q,
                            const uint16_t* k_pages, const uint16_t* v_pages,
                            const int32_t* page_table, const int32_t* ctx_lens,
                            int32_t n_draft, double* out) {
    if (batch < 0 || n_q_heads <= 0 || n_kv_heads <= 0 || head_dim <= 0 ||
        page_size <= 0 || max_pages_per_seq <= 0 || num_pages < 0 || n_draft < 0)
        return ORC_BAD_ARG;
    if (n_q_heads % n_kv_heads != 0) return ORC_BAD_ARG;
    if (batch == 0) return ORC_OK;

    const int64_t n_rows = (int64_t)n_draft + 1;
    const int64_t group = n_q_heads / n_kv_heads;
    const int64_t D = head_dim;
    const int64_t ps = page_size;
    const int64_t l_cap = (int64_t)max_pages_per_seq * ps;
    if (scale <= 0.0) scale = 1.0 / sqrt((double)head_dim);

    int status = ORC_OK;
#pragma omp parallel for collapse(2) schedule(dynamic, 1)
    for (int64_t b = 0; b < batch; ++b) {
        for (int64_t h = 0; h < n_q_heads; ++h) {
            int64_t L = ctx_lens[b];
            if (L < 0) L = 0;
            if (L > l_cap) L = l_cap;
            const int64_t kvh = h / group;
            double* s = (double*)malloc((size_t)(L > 0 ? L : 1) * sizeof(double));
            double* o = (double*)malloc((size_t)D * sizeof(double));
            if (!s || !o) {
#pragma omp atomic write
                status = ORC_NO_MEM;
                free(s);
                free(o);
                continue;
            }
            for (int64_t i = 0; i < n_rows; ++i) {
                const uint16_t* qv = q + ((b * n_rows + i) * n_q_heads + h) * D;
                double* dst = out + ((b * n_rows + i) * n_q_heads + h) * D;
                const int64_t last = L - n_rows + i; /* highest admissible key */
                if (last < 0) {
                    for (int64_t d = 0; d < D; ++d) dst[d] = 0.0;
                    continue;
                }
                /* scores s_j = scale * q . K_j, j = 0..last */
                for (int64_t j = 0; j <= last; ++j) {
                    const int64_t page = page_table[b * max_pages_per_seq + j / ps];
                    double dot = 0.0;
                    if (page >= 0 && page < num_pages) {
                        const uint16_t* kr =
                            k_pages + ((page * n_kv_heads + kvh) * ps + j % ps) * D;
                        for (int64_t d = 0; d < D; ++d)
                            dot += bf16_bits_to_double(qv[d]) * bf16_bits_to_double(kr[d]);
                    }
                    s[j] = scale * dot;
                }
                /* stable softmax: max, then exp and sum */
                double m = s[0];
                for (int64_t j = 1; j <= last; ++j)
                    if (s[j] > m) m = s[j];
                double l = 0.0;
                for (int64_t j = 0; j <= last; ++j) {
                    s[j] = exp(s[j] - m);
                    l += s[j];
                }
                for (int64_t d = 0; d < D; ++d) o[d] = 0.0;
                for (int64_t j = 0; j <= last; ++j) {
                    const int64_t page = page_table[b * max_pages_per_seq + j / ps];
                    if (page < 0 || page >= num_pages) continue; /* zero row */
                    const uint16_t* vr =
                        v_pages + ((page * n_kv_heads + kvh) * ps + j % ps) * D;
                    for (int64_t d = 0; d < D; ++d) o[d] += s[j] * bf16_bits_to_double(vr[d]);
                }
                for (int64_t d = 0; d < D; ++d) dst[d] = o[d] / l;
            }
            free(s);
            free(o);
        }
    }
    return status;
}

/* ------------------------------------------------------------------------
 * 2. Speculative acceptance.
 * ---------------------------------------------------------------------- */

/* p = softmax(z / T) for one row, T > 0: max, then exp((z-m)/T), then sum,
 * then divide.  Returns the sum of exponentials (the normaliser). */
double oracle_row_probs(const void* row, int32_t dtype, int32_t vocab,
                        double temperature, double* p) {
    double m = logit_at(row, dtype, 0);
    for (int64_t v = 1; v < vocab; ++v) {
        const double z = logit_at(row, dtype, v);
        if (z > m) m = z;
    }
    double S = 0.0;
    for (int64_t v = 0; v < vocab; ++v) {
        p[v] = exp((logit_at(row, dtype, v) - m) / temperature);
        S += p[v];
    }
    for (int64_t v = 0; v < vocab; ++v) p[v] /= S;
    return S;
}

/* Residual distribution of a rejection: r(v) = max(0, p(v) - q(v)),
 * Z = sum_v r(v) in ascending v.  Returns Z. */
double oracle_residual(const double* p, const double* q, int32_t vocab, double* r) {
    double Z = 0.0;
    for (int64_t v = 0; v < vocab; ++v) {
        const double d = p[v] - q[v];
        r[v] = d > 0.0 ? d : 0.0;
        Z += r[v];
    }
    return Z;
}

/* Inverse-CDF draw over unnormalised weights r with total Z: the smallest v
 * whose running sum (ascending v) exceeds u*Z; if rounding leaves none, the
 * largest v with r(v) > 0.  *margin receives the distance of u from the two
 * CDF values that bracket the chosen cell, both divided by Z. */
int32_t oracle_inverse_cdf(const double* r, double Z, int32_t vocab, double u,
                           double* margin) {
    const double t = u * Z;
    double cum = 0.0, before = 0.0;
    int32_t pick = -1;
    for (int32_t v = 0; v < vocab; ++v) {
        before = cum;
        cum += r[v];
        if (cum > t) {
            pick = v;
            break;
        }
    }
    if (pick < 0) {
        for (int32_t v = vocab - 1; v >= 0; --v)
            if (r[v] > 0.0) {
                pick = v;
                break;
            }
        if (pick < 0) pick = 0; /* all-zero weights cannot arise from a softmax */
        before = cum;
    }
    if (margin) {
        const double m1 = fabs(u - cum / Z), m0 = fabs(u - before / Z);
        *margin = m1 < m0 ? m1 : m0;
    }
    return pick;
}

/* argmax with the lowest id on ties. */
int32_t oracle_row_argmax(const void* row, int32_t dtype, int32_t vocab) {
    int32_t best = 0;
    double bv = logit_at(row, dtype, 0);
    for (int32_t v = 1; v < vocab; ++v) {
        const double z = logit_at(row, dtype, v);
        if (z > bv) {
            bv = z;
            best = v;
        }
    }
    return best;
}

/*
 * target   [B, k+1, V]  fp32 (dtype 0) or bf16 bits (dtype 1)
 * draft    [B, k,   V]  same dtype; ignored (may be NULL) when T == 0
 * tokens   [B, k]       int32 draft tokens x_i
 * uniforms [B, k+1]     fp64 here (the fp32 entry below widens them);
 *                       u_0..u_{k-1} for the accept tests, u_k for the single
 *                       final draw (residual or bonus)
 * out_tokens [B, k+1]   x_0..x_{a-1}, then the drawn token, then -1
 * out_n_accepted [B]    a
 * out_margin [B]        (may be NULL) smallest |u_i - p_i(x_i)/q_i(x_i)| over
 *                       the accept tests that decided the output (positions
 *                       0..a); +inf when there is none (greedy, or a = 0
 *                       through an invalid token)
 * out_draw_margin [B]   (may be NULL) distance of u_k from the two CDF values
 *                       C(v-1)/Z and C(v)/Z that bracket the drawn token v;
 *                       +inf for greedy
 *
 * A draft token outside [0, V) counts as rejected (its ratio is 0).
 */
int oracle_spec_accept_f64u(int32_t batch, int32_t vocab, int32_t dtype,
                            const void* target, const void* draft,
                            const int32_t* tokens, const double* uniforms,
                            int32_t n_draft, double temperature, int32_t* out_tokens,
                            int32_t* out_n_accepted, double* out_margin,
                            double* out_draw_margin) {
    if (batch < 0 || vocab <= 0 || n_draft < 0 || (dtype != 0 && dtype != 1))
        return ORC_BAD_ARG;
    if (!(temperature >= 0.0)) return ORC_BAD_ARG;
    if (temperature > 0.0 && n_draft > 0 && !draft) return ORC_BAD_ARG;
    const int64_t k = n_draft;
    const int64_t V = vocab;
    const size_t esz = dtype == 0 ? 4 : 2;
    int status = ORC_OK;

#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t b = 0; b < batch; ++b) {
        const char* trow0 = (const char*)target + (size_t)(b * (k + 1) * V) * esz;
        const char* drow0 = draft ? (const char*)draft + (size_t)(b * k * V) * esz : NULL;
        const int32_t* x = tokens + b * k;
        const double* u = uniforms + b * (k + 1);
        int32_t* out = out_tokens + b * (k + 1);
        int64_t a = k;
        double margin = INFINITY, draw_margin = INFINITY;

        if (temperature == 0.0) {
            /* greedy: argmax agreement */
            int32_t g = 0;
            for (int64_t i = 0; i <= k; ++i) {
                g = oracle_row_argmax(trow0 + (size_t)(i * V) * esz, dtype, vocab);
                if (i == k || x[i] != g) {
                    a = i;
                    break;
                }
            }
            for (int64_t i = 0; i < a; ++i) out[i] = x[i];
            out[a] = g;
        } else {
            double* p = (double*)malloc((size_t)V * sizeof(double));
            double* q = (double*)malloc((size_t)V * sizeof(double));
            double* r = (double*)malloc((size_t)V * sizeof(double));
            if (!p || !q || !r) {
#pragma omp atomic write
                status = ORC_NO_MEM;
                free(p);
                free(q);
                free(r);
                continue;
            }
            /* accept tests, in order, until the first rejection */
            for (int64_t i = 0; i < k; ++i) {
                oracle_row_probs(trow0 + (size_t)(i * V) * esz, dtype, vocab, temperature, p);
                oracle_row_probs(drow0 + (size_t)(i * V) * esz, dtype, vocab, temperature, q);
                double ratio = 0.0;
                if (x[i] >= 0 && x[i] < vocab)
                    ratio = q[x[i]] > 0.0 ? p[x[i]] / q[x[i]] : INFINITY;
                const double gap = fabs(u[i] - ratio);
                if (gap < margin) margin = gap;
                if (!(u[i] < ratio)) {
                    a = i;
                    break;
                }
            }
            double Z;
            if (a < k) {
                /* p and q still hold row a */
                Z = oracle_residual(p, q, vocab, r);
                if (!(Z > 0.0)) { /* p == q up to rounding: fall back to p */
                    Z = 0.0;
                    for (int64_t v = 0; v < V; ++v) {
                        r[v] = p[v];
                        Z += r[v];
                    }
                }
            } else {
                oracle_row_probs(trow0 + (size_t)(k * V) * esz, dtype, vocab, temperature, p);
                Z = 0.0;
                for (int64_t v = 0; v < V; ++v) {
                    r[v] = p[v];
                    Z += r[v];
                }
            }
            const int32_t pick = oracle_inverse_cdf(r, Z, vocab, u[k], &draw_margin);
            for (int64_t i = 0; i < a; ++i) out[i] = x[i];
            out[a] = pick;
            free(p);
            free(q);
            free(r);
        }
        for (int64_t i = a + 1; i <= k; ++i) out[i] = -1;
        out_n_accepted[b] = (int32_t)a;
        if (out_margin) out_margin[b] = margin;
        if (out_draw_margin) out_draw_margin[b] = draw_margin;
    }
    return status;
}

/* The library's own uniform type is fp32; widen exactly and run the core. */
int oracle_spec_accept(int32_t batch, int32_t vocab, int32_t dtype,
                       const void* target, const void* draft,
                       const int32_t* tokens, const float* uniforms,
                       int32_t n_draft, double temperature, int32_t* out_tokens,
                       int32_t* out_n_accepted, double* out_margin,
                       double* out_draw_margin) {
    if (batch < 0 || n_draft < 0) return ORC_BAD_ARG;
    const size_t n = (size_t)batch * (size_t)(n_draft + 1);
    double* u = (double*)malloc((n ? n : 1) * sizeof(double));
    if (!u) return ORC_NO_MEM;
    for (size_t i = 0; i < n; ++i) u[i] = (double)uniforms[i];
    const int rc = oracle_spec_accept_f64u(batch, vocab, dtype, target, draft, tokens, u,
                                           n_draft, temperature, out_tokens,
                                           out_n_accepted, out_margin, out_draw_margin);
    free(u);
    return rc;
}

/* ------------------------------------------------------------------------
 * 4. Draft-side sampling.
 *
 * For each row b: T > 0 draws out[b] = inverse CDF of p = softmax(z_b / T)
 * at uniforms[b] (the total Z is the computed sum of p, as in the final draw
 * of the acceptance step); T == 0 takes the argmax (lowest id on ties).
 * out_margin[b] (may be NULL) is the distance of u from the two CDF values
 * bracketing the drawn cell (+inf for greedy).
 * ---------------------------------------------------------------------- */
int oracle_sample(int32_t batch, int32_t vocab, int32_t dtype, const void* logits,
                  const double* uniforms, double temperature, int32_t* out_tokens,
                  double* out_margin) {
    if (batch < 0 || vocab <= 0 || (dtype != 0 && dtype != 1)) return ORC_BAD_ARG;
    if (!(temperature >= 0.0)) return ORC_BAD_ARG;
    const size_t esz = dtype == 0 ? 4 : 2;
    int status = ORC_OK;
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t b = 0; b < batch; ++b) {
        const char* row = (const char*)logits + (size_t)b * (size_t)vocab * esz;
        double margin = INFINITY;
        if (temperature == 0.0) {
            out_tokens[b] = oracle_row_argmax(row, dtype, vocab);
        } else {
            double* p = (double*)malloc((size_t)vocab * sizeof(double));
            if (!p) {
#pragma omp atomic write
                status = ORC_NO_MEM;
                continue;
            }
            oracle_row_probs(row, dtype, vocab, temperature, p);
            double Z = 0.0;
            for (int64_t v = 0; v < vocab; ++v) Z += p[v];
            out_tokens[b] = oracle_inverse_cdf(p, Z, vocab, uniforms[b], &margin);
            free(p);
        }
        if (out_margin) out_margin[b] = margin;
    }
    return status;
}

/* ------------------------------------------------------------------------
 * 5. Paged KV cache.
 *
 * Append: rows are bf16 bit patterns.  For request b, new row i, KV head h:
 * pos = L_b - n_new + i with L_b clamped to [0, max_pages * ps]; when
 * pos >= 0 and the page id is in [0, num_pages), copy the D values into
 * pool[page][h][pos % ps].  Commit: L_b <- max(0, L_b - n_draft + a_b).
 * ---------------------------------------------------------------------- */
int oracle_kv_append(int32_t batch, int32_t n_kv_heads, int32_t head_dim, int32_t page_size,
                     int32_t max_pages, int32_t num_pages, const uint16_t* new_k,
                     const uint16_t* new_v, uint16_t* k_pages, uint16_t* v_pages,
                     const int32_t* page_table, const int32_t* ctx_lens, int32_t n_new) {
    if (batch < 0 || n_kv_heads <= 0 || head_dim <= 0 || page_size <= 0 || max_pages <= 0 ||
        num_pages <= 0 || n_new < 1)
        return ORC_BAD_ARG;
    const int64_t cap = (int64_t)max_pages * page_size;
    for (int64_t b = 0; b < batch; ++b) {
        int64_t L = ctx_lens[b];
        if (L < 0) L = 0;
        if (L > cap) L = cap;
        for (int64_t i = 0; i < n_new; ++i) {
            const int64_t pos = L - n_new + i;
            if (pos < 0) continue;
            const int64_t page = page_table[b * max_pages + pos / page_size];
            if (page < 0 || page >= num_pages) continue;
            for (int64_t h = 0; h < n_kv_heads; ++h) {
                const int64_t src = ((b * n_new + i) * n_kv_heads + h) * head_dim;
                const int64_t dst = ((page * n_kv_heads + h) * page_size + pos % page_size) * head_dim;
                for (int64_t e = 0; e < head_dim; ++e) {
                    k_pages[dst + e] = new_k[src + e];
                    v_pages[dst + e] = new_v[src + e];
                }
            }
        }
    }
    return ORC_OK;
}

int oracle_kv_commit(int32_t batch, int32_t* ctx_lens, const int32_t* n_accepted, int32_t n_draft) {
    if (batch < 0 || n_draft < 0) return ORC_BAD_ARG;
    for (int64_t b = 0; b < batch; ++b) {
        const int64_t L = (int64_t)ctx_lens[b] - n_draft + n_accepted[b];
        ctx_lens[b] = (int32_t)(L > 0 ? L : 0);
    }
    return ORC_OK;
}

/* ------------------------------------------------------------------------
 * 6. Semantic routing.
 *
 * emb [B, d] and centroids [N, d] are bf16 bit patterns, widened exactly.
 * S(b, i) = (e_b . c_i) / (|e_b| |c_i|), 0 when either norm is 0; every
 * product and sum in fp64, ascending index.  out_best[b] = argmax_i S (the
 * lowest i on ties; -1 when N == 0), out_score[b] = that S (-inf when
 * N == 0), out_group[b] = out_best[b] if out_score[b] >= tau else -1.
 * out_margin[b] (may be NULL) = best score minus the runner-up (+inf when
 * N < 2); out_tau_margin[b] (may be NULL) = |best score - tau|.
 * ---------------------------------------------------------------------- */
static double bf16_at(const uint16_t* p, int64_t i) { return bf16_bits_to_double(p[i]); }

int oracle_route(int32_t batch, int32_t n_groups, int32_t dim, const uint16_t* emb,
                 const uint16_t* centroids, double tau, int32_t* out_group, int32_t* out_best,
                 double* out_score, double* out_margin, double* out_tau_margin) {
    if (batch < 0 || n_groups < 0 || dim <= 0) return ORC_BAD_ARG;
    double* cn = (double*)malloc(((size_t)n_groups + 1) * sizeof(double));
    if (!cn) return ORC_NO_MEM;
    for (int64_t i = 0; i < n_groups; ++i) {
        double s = 0.0;
        for (int64_t k = 0; k < dim; ++k) {
            const double c = bf16_at(centroids, i * dim + k);
            s += c * c;
        }
        cn[i] = sqrt(s);
    }
#pragma omp parallel for schedule(dynamic, 16)
    for (int64_t b = 0; b < batch; ++b) {
        double en = 0.0;
        for (int64_t k = 0; k < dim; ++k) {
            const double e = bf16_at(emb, b * dim + k);
            en += e * e;
        }
        en = sqrt(en);
        double best = -INFINITY, second = -INFINITY;
        int32_t arg = -1;
        for (int64_t i = 0; i < n_groups; ++i) {
            double dot = 0.0;
            for (int64_t k = 0; k < dim; ++k) dot += bf16_at(emb, b * dim + k) * bf16_at(centroids, i * dim + k);
            const double s = (en > 0.0 && cn[i] > 0.0) ? dot / (en * cn[i]) : 0.0;
            if (s > best) {
                second = best;
                best = s;
                arg = (int32_t)i;
            } else if (s > second) {
                second = s;
            }
        }
        out_best[b] = arg;
        out_score[b] = best;
        out_group[b] = (arg >= 0 && best >= tau) ? arg : -1;
        if (out_margin) out_margin[b] = n_groups >= 2 ? best - second : INFINITY;
        if (out_tau_margin) out_tau_margin[b] = fabs(best - tau);
    }
    free(cn);
    return ORC_OK;
}

/* ------------------------------------------------------------------------
 * 7. Token-tree verification (the multi-candidate variant of the
 *    draft-and-verify step that the paper cites among the SpecDec variants
 *    in Sec. 2: a tree of drafted candidates verified in one target pass,
 *    then a walk that keeps one root-to-node path).
 *
 * A request's tree has n nodes in topological order.  Node 0 is the root,
 * the last committed token, which is not verified; node c >= 1 holds the
 * drafted token tokens[c] and its parent parents[c], which must lie in
 * [0, c) -- a node whose parent does not is detached: it is never reached
 * by the walk and its ancestry stops at itself.  anc(c) = {c} plus anc of
 * its parent.  The K/V rows of node m sit at key position L_b - n + m.
 *
 * Attention: node i of request b, query head h, sees every prefix key
 * j < L_b - n and the tree keys L_b - n + m for m in anc(i); the same
 * softmax(q.K*scale).V as section 1 over that key set, in ascending key
 * order.  Keys at negative positions (L_b < n) do not exist.  A node that
 * sees no key outputs zeros.
 *
 * Acceptance (T > 0): the walk starts at the root with the target
 * distribution p_u = softmax(z_t,u / T) of the current node u as its
 * running distribution r.  The children of u (the nodes whose parent is u,
 * ascending index) are tested in turn against the draft distribution
 * q_u = softmax(z_d,u / T) that drafted them: child c with token x is
 * accepted iff u_{c-1} < r(x) / q_u(x) (+inf when q_u(x) == 0, 0 when x is
 * not a token id).  A rejection replaces r by max(0, r - q_u) normalised and
 * the next sibling is tested against it; if that residual has no positive
 * mass (r == q_u up to rounding) the remaining siblings are skipped and r
 * falls back to p_u.  An accepted child is emitted and becomes u; when no
 * child is accepted (or u is a leaf) one token is drawn from r by the
 * inverse CDF of section 2 at u_{n-1}, and the step ends.  When every
 * node's children are independent draws from that node's q_u, the emitted
 * tokens follow the target's law exactly (each test is one speculative
 * sampling step whose fallback is again such a step).  A chain
 * (parents[c] = c - 1) is exactly the rule of section 2 with k = n - 1.
 * Greedy (T == 0): at node u, g = argmax z_t,u (lowest id on ties); the
 * first child whose token equals g is accepted, else g is emitted.
 *
 * target [B, n, V], draft [B, n, V] (row u = the distribution node u's
 * children were drafted from; rows of leaves are not read; draft may be
 * NULL when T == 0), parents / tokens [B, n] int32, uniforms [B, n] fp64
 * (u_{c-1} tests node c, u_{n-1} is the draw).  out_tokens [B, n]: the
 * accepted tokens, the emitted token, then -1; out_path [B, n]: the
 * accepted nodes in walk order, then -1; out_n [B]: accepted count.
 * out_margin / out_draw_margin as in section 2 (over the tests performed).
 * ---------------------------------------------------------------------- */
static int tree_parent(const int32_t* par, int64_t c) {
    if (c <= 0) return -1;
    const int32_t p = par[c];
    return (p >= 0 && p < c) ? p : -1;
}

int oracle_tree_attention(int32_t batch, int32_t n_q_heads, int32_t n_kv_heads,
                          int32_t head_dim, int32_t page_size, int32_t max_pages_per_seq,
                          int32_t num_pages, double scale, const uint16_t* q,
                          const uint16_t* k_pages, const uint16_t* v_pages,
                          const int32_t* page_table, const int32_t* ctx_lens,
                          const int32_t* parents, int32_t n_nodes, double* out) {
    if (batch < 0 || n_q_heads <= 0 || n_kv_heads <= 0 || head_dim <= 0 ||
        page_size <= 0 || max_pages_per_seq <= 0 || num_pages < 0 || n_nodes < 1)
        return ORC_BAD_ARG;
    if (n_q_heads % n_kv_heads != 0) return ORC_BAD_ARG;
    if (batch == 0) return ORC_OK;
    const int64_t n = n_nodes, group = n_q_heads / n_kv_heads, D = head_dim, ps = page_size;
    const int64_t l_cap = (int64_t)max_pages_per_seq * ps;
    if (scale <= 0.0) scale = 1.0 / sqrt((double)head_dim);

    int status = ORC_OK;
#pragma omp parallel for collapse(2) schedule(dynamic, 1)
    for (int64_t b = 0; b < batch; ++b) {
        for (int64_t h = 0; h < n_q_heads; ++h) {
            int64_t L = ctx_lens[b];
            if (L < 0) L = 0;
            if (L > l_cap) L = l_cap;
            const int64_t kvh = h / group;
            const int32_t* par = parents + b * n;
            int64_t* keys = (int64_t*)malloc((size_t)(L + 1) * sizeof(int64_t));
            double* s = (double*)malloc((size_t)(L + 1) * sizeof(double));
            char* in_anc = (char*)malloc((size_t)n);
            double* o = (double*)malloc((size_t)D * sizeof(double));
            if (!keys || !s || !in_anc || !o) {
#pragma omp atomic write
                status = ORC_NO_MEM;
                free(keys);
                free(s);
                free(in_anc);
                free(o);
                continue;
            }
            for (int64_t i = 0; i < n; ++i) {
                const uint16_t* qv = q + ((b * n + i) * n_q_heads + h) * D;
                double* dst = out + ((b * n + i) * n_q_heads + h) * D;
                /* the key set of node i, ascending */
                for (int64_t m = 0; m < n; ++m) in_anc[m] = 0;
                for (int64_t m = i; m >= 0; m = tree_parent(par, m)) in_anc[m] = 1;
                int64_t nk = 0;
                for (int64_t j = 0; j < L; ++j) {
                    const int64_t m = j - (L - n);
                    if (m < 0 || in_anc[m]) keys[nk++] = j;
                }
                if (nk == 0) {
                    for (int64_t d = 0; d < D; ++d) dst[d] = 0.0;
                    continue;
                }
                for (int64_t t = 0; t < nk; ++t) {
                    const int64_t j = keys[t];
                    const int64_t page = page_table[b * max_pages_per_seq + j / ps];
                    double dot = 0.0;
                    if (page >= 0 && page < num_pages) {
                        const uint16_t* kr = k_pages + ((page * n_kv_heads + kvh) * ps + j % ps) * D;
                        for (int64_t d = 0; d < D; ++d)
                            dot += bf16_bits_to_double(qv[d]) * bf16_bits_to_double(kr[d]);
                    }
                    s[t] = scale * dot;
                }
                double m = s[0];
                for (int64_t t = 1; t < nk; ++t)
                    if (s[t] > m) m = s[t];
                double l = 0.0;
                for (int64_t t = 0; t < nk; ++t) {
                    s[t] = exp(s[t] - m);
                    l += s[t];
                }
                for (int64_t d = 0; d < D; ++d) o[d] = 0.0;
                for (int64_t t = 0; t < nk; ++t) {
                    const int64_t j = keys[t];
                    const int64_t page = page_table[b * max_pages_per_seq + j / ps];
                    if (page < 0 || page >= num_pages) continue;
                    const uint16_t* vr = v_pages + ((page * n_kv_heads + kvh) * ps + j % ps) * D;
                    for (int64_t d = 0; d < D; ++d) o[d] += s[t] * bf16_bits_to_double(vr[d]);
                }
                for (int64_t d = 0; d < D; ++d) dst[d] = o[d] / l;
            }
            free(keys);
            free(s);
            free(in_anc);
            free(o);
        }
    }
    return status;
}

int oracle_tree_accept_f64u(int32_t batch, int32_t vocab, int32_t dtype, const void* target,
                            const void* draft, const int32_t* parents, const int32_t* tokens,
                            const double* uniforms, int32_t n_nodes, double temperature,
                            int32_t* out_tokens, int32_t* out_path, int32_t* out_n,
                            double* out_margin, double* out_draw_margin) {
    if (batch < 0 || vocab <= 0 || n_nodes < 1 || (dtype != 0 && dtype != 1)) return ORC_BAD_ARG;
    if (!(temperature >= 0.0)) return ORC_BAD_ARG;
    if (temperature > 0.0 && n_nodes > 1 && !draft) return ORC_BAD_ARG;
    const int64_t n = n_nodes, V = vocab;
    const size_t esz = dtype == 0 ? 4 : 2;
    int status = ORC_OK;

#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t b = 0; b < batch; ++b) {
        const char* trow0 = (const char*)target + (size_t)(b * n * V) * esz;
        const char* drow0 = draft ? (const char*)draft + (size_t)(b * n * V) * esz : NULL;
        const int32_t* par = parents + b * n;
        const int32_t* x = tokens + b * n;
        const double* u = uniforms + b * n;
        int32_t* out = out_tokens + b * n;
        int32_t* path = out_path + b * n;
        int64_t depth = 0, node = 0;
        double margin = INFINITY, draw_margin = INFINITY;
        int32_t emit = 0;

        if (temperature == 0.0) {
            for (;;) {
                const int32_t g = oracle_row_argmax(trow0 + (size_t)(node * V) * esz, dtype, vocab);
                int64_t next = -1;
                for (int64_t c = node + 1; c < n; ++c)
                    if (tree_parent(par, c) == node && x[c] == g) {
                        next = c;
                        break;
                    }
                if (next < 0) {
                    emit = g;
                    break;
                }
                out[depth] = x[next];
                path[depth] = (int32_t)next;
                ++depth;
                node = next;
            }
        } else {
            double* p = (double*)malloc((size_t)V * sizeof(double));
            double* qd = (double*)malloc((size_t)V * sizeof(double));
            double* r = (double*)malloc((size_t)V * sizeof(double));
            if (!p || !qd || !r) {
#pragma omp atomic write
                status = ORC_NO_MEM;
                free(p);
                free(qd);
                free(r);
                continue;
            }
            for (;;) {
                oracle_row_probs(trow0 + (size_t)(node * V) * esz, dtype, vocab, temperature, p);
                for (int64_t v = 0; v < V; ++v) r[v] = p[v];
                int have_q = 0;
                int64_t next = -1;
                for (int64_t c = node + 1; c < n; ++c) {
                    if (tree_parent(par, c) != node) continue;
                    if (!have_q) {
                        oracle_row_probs(drow0 + (size_t)(node * V) * esz, dtype, vocab, temperature, qd);
                        have_q = 1;
                    }
                    double ratio = 0.0;
                    if (x[c] >= 0 && x[c] < vocab)
                        ratio = qd[x[c]] > 0.0 ? r[x[c]] / qd[x[c]] : INFINITY;
                    const double gap = fabs(u[c - 1] - ratio);
                    if (gap < margin) margin = gap;
                    if (u[c - 1] < ratio) {
                        next = c;
                        break;
                    }
                    /* rejected: the next sibling is tested against the residual */
                    double Z = 0.0;
                    for (int64_t v = 0; v < V; ++v) {
                        const double d = r[v] - qd[v];
                        r[v] = d > 0.0 ? d : 0.0;
                        Z += r[v];
                    }
                    if (!(Z > 0.0)) {
                        for (int64_t v = 0; v < V; ++v) r[v] = p[v];
                        break;
                    }
                    for (int64_t v = 0; v < V; ++v) r[v] /= Z;
                }
                if (next < 0) {
                    double Z = 0.0;
                    for (int64_t v = 0; v < V; ++v) Z += r[v];
                    emit = oracle_inverse_cdf(r, Z, vocab, u[n - 1], &draw_margin);
                    break;
                }
                out[depth] = x[next];
                path[depth] = (int32_t)next;
                ++depth;
                node = next;
            }
            free(p);
            free(qd);
            free(r);
        }
        out[depth] = emit;
        for (int64_t i = depth + 1; i < n; ++i) out[i] = -1;
        for (int64_t i = depth; i < n; ++i) path[i] = -1;
        out_n[b] = (int32_t)depth;
        if (out_margin) out_margin[b] = margin;
        if (out_draw_margin) out_draw_margin[b] = draw_margin;
    }
    return status;
}

int oracle_tree_accept(int32_t batch, int32_t vocab, int32_t dtype, const void* target,
                       const void* draft, const int32_t* parents, const int32_t* tokens,
                       const float* uniforms, int32_t n_nodes, double temperature,
                       int32_t* out_tokens, int32_t* out_path, int32_t* out_n,
                       double* out_margin, double* out_draw_margin) {
    if (batch < 0 || n_nodes < 1) return ORC_BAD_ARG;
    const size_t cnt = (size_t)batch * (size_t)n_nodes;
    double* u = (double*)malloc((cnt ? cnt : 1) * sizeof(double));
    if (!u) return ORC_NO_MEM;
    for (size_t i = 0; i < cnt; ++i) u[i] = (double)uniforms[i];
    const int rc = oracle_tree_accept_f64u(batch, vocab, dtype, target, draft, parents, tokens, u,
                                           n_nodes, temperature, out_tokens, out_path, out_n,
                                           out_margin, out_draw_margin);
    free(u);
    return rc;
}

/* Commit of an accepted tree path: the K/V rows of the accepted nodes
 * path[0..a) move, in walk order, to the key positions right after the
 * root, L_b - n + 1 + i (node path[i] sat at L_b - n + path[i] >= that
 * position, so an ascending copy never overwrites a row it still needs),
 * and L_b becomes L_b - n + 1 + a.  Rows with a negative position or a
 * page id outside [0, num_pages) are skipped, as in the append. */
int oracle_kv_commit_tree(int32_t batch, int32_t n_kv_heads, int32_t head_dim, int32_t page_size,
                          int32_t max_pages, int32_t num_pages, uint16_t* k_pages,
                          uint16_t* v_pages, const int32_t* page_table, int32_t* ctx_lens,
                          const int32_t* path, const int32_t* n_accepted, int32_t n_nodes) {
    if (batch < 0 || n_kv_heads <= 0 || head_dim <= 0 || page_size <= 0 || max_pages <= 0 ||
        num_pages <= 0 || n_nodes < 1)
        return ORC_BAD_ARG;
    const int64_t cap = (int64_t)max_pages * page_size;
    for (int64_t b = 0; b < batch; ++b) {
        int64_t L = ctx_lens[b];
        if (L < 0) L = 0;
        if (L > cap) L = cap;
        int64_t a = n_accepted[b];
        if (a < 0) a = 0;
        if (a > n_nodes - 1) a = n_nodes - 1;
        const int64_t base = L - n_nodes;
        for (int64_t i = 0; i < a; ++i) {
            const int64_t node = path[b * n_nodes + i];
            if (node < 1 || node >= n_nodes) continue;
            const int64_t src = base + node, dst = base + 1 + i;
            if (src == dst || src < 0 || dst < 0) continue;
            const int64_t ps_ = page_size;
            const int64_t sp = page_table[b * max_pages + src / ps_];
            const int64_t dp = page_table[b * max_pages + dst / ps_];
            if (sp < 0 || sp >= num_pages || dp < 0 || dp >= num_pages) continue;
            for (int64_t h = 0; h < n_kv_heads; ++h) {
                const int64_t so = ((sp * n_kv_heads + h) * ps_ + src % ps_) * head_dim;
                const int64_t d0 = ((dp * n_kv_heads + h) * ps_ + dst % ps_) * head_dim;
                for (int64_t e = 0; e < head_dim; ++e) {
                    k_pages[d0 + e] = k_pages[so + e];
                    v_pages[d0 + e] = v_pages[so + e];
                }
            }
        }
        const int64_t nl = base + 1 + a;
        ctx_lens[b] = (int32_t)(nl > 0 ? nl : 0);
    }
    return ORC_OK;
}
