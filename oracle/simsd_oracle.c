/*
 * simsd_oracle.c -- plain fp64 CPU oracle for the SimSD verification step.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously-correct
 * statement of what the verification step computes.  Only the tests, the
 * smoke check and the CPU-baseline leg of the benchmark may load it; the
 * product path never calls it, and it shares no code, header or constant
 * with the CUDA library.
 *
 * Paper: "SimSD: Simple Speculative Decoding in Diffusion Language Models".
 *   - Sec. 3.1 "Input Layout Prepare": prompt, data section D (B reference
 *     tokens), mask section D~ (B prediction slots); D_k and D~_k are the
 *     same response position.
 *   - Sec. 3.1 "Temporal Attention Mask", Eq. (1): the four-case visibility
 *     rule over response positions; prompt visible to every response
 *     position; padding rows and columns zeroed.
 *   - Sec. 3.1 "Position Encoding Alignment": D~_k reuses the RoPE index of
 *     D_k; rotary position embedding as in Su et al. (RoFormer), in the
 *     rotate-half layout of the Qwen-family SDAR models.  Sec. 4 ablation
 *     (Table 4) "without aligned RoPE": mask slots take their physical
 *     positions after the data section instead.
 *   - Sec. 3.2 "Target Model Verification": slot with tau = r holds the r-th
 *     draft; acceptance along the draft order, longest prefix before the
 *     first rejection; Eq. (2) with one-hot distributions (temperature 0)
 *     reduces to "accept iff the target argmax equals the draft".
 *   - Sec. 3.3 "Adaptation under Blockwise Decoding and KV Cache": the
 *     prefix K/V is reused from the cache; only new positions are computed.
 *
 * Readings where the paper is silent (each one is listed in the design
 * notes): slot k in [0,gamma) is D_k and slot gamma+k is D~_k; step-map
 * value 0 marks a padding position; a step map that is not a partial
 * permutation of 1..gamma makes the whole sequence padding; argmax ties go
 * to the lowest index and NaN ranks above every number (first NaN wins);
 * the accepted count excludes the correction token; the committed K/V of
 * an accepted draft is its data-slot K/V, appended in tau order.
 *
 * Everything is computed in double precision, in the order the definitions
 * state, with no blocking or fusion.  OpenMP only distributes independent
 * output rows over threads; each row is computed by one thread in a fixed
 * order, so results do not depend on the thread count.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* error bits (the oracle's own copy of the documented meanings) */
#define OR_ERR_STEP_MAP 1
#define OR_ERR_PREFIX_LEN 2
#define OR_ERR_PAGE 4
#define OR_ERR_DRAFT 8
#define OR_ERR_ACCEPT_LEN 32

#define OR_SECT_D 0
#define OR_SECT_DT 1
#define OR_SECT_PAD 255

/* ---------------------------------------------------------------------- */
/* Sec. 3.1: step map -> per-slot temporal label, section and RoPE index.  */
/* ---------------------------------------------------------------------- */

/* Checks that step_map row b is a partial permutation of 1..gamma (0 marks
 * padding).  Returns 1 when valid. */
/* Step-map codes besides the drafted labels 1..gamma.  Sec. 3.2 verifies
 * only the gamma drafted positions of a block; with fewer drafts than
 * undecoded positions, and when the target completes the block itself
 * (R < gamma), the block also holds positions that stay [MASK] through the
 * step and positions decoded earlier in the block.
 *    0  padding: both slots of the position are padding (Eq. (1), zeroed
 *       rows and columns);
 *   -1  undrafted: the position stays a mask placeholder; its data slot is
 *       padding and its mask slot carries tau = gamma + 1, later than every
 *       drafted step;
 *   -2  decoded: the position already holds a clean token; its data slot
 *       carries tau = 0 (known before every step, like a prompt token) and
 *       its mask slot is padding. */
#define OR_STEP_UNDRAFTED (-1)
#define OR_STEP_DECODED (-2)

static int step_map_row_valid(const int32_t *mu, int gamma) {
    for (int k = 0; k < gamma; ++k) {
        if (mu[k] < OR_STEP_DECODED || mu[k] > gamma) return 0;
        if (mu[k] <= 0) continue;
        for (int k2 = 0; k2 < k; ++k2)
            if (mu[k2] == mu[k]) return 0;
    }
    return 1;
}

/* Per-slot labels for one sequence.  Slot k (k < gamma) is D_k, slot gamma+k
 * is D~_k; a drafted position gives both tau = mu_k (Sec. 3.1 "Temporal
 * Attention Mask"); the codes above set the other kinds.  An invalid map
 * marks every slot as padding.  The RoPE index of both D_k and D~_k is the
 * absolute position of D_k, i.e. n + k, where n is the cached prefix length
 * (Sec. 3.1 "Position Encoding Alignment"). */
static int labels_for_sequence(const int32_t *mu, int n, int gamma, int32_t *tau,
                               uint8_t *sect, int32_t *rope) {
    int ok = step_map_row_valid(mu, gamma);
    for (int k = 0; k < gamma; ++k) {
        int v = ok ? mu[k] : 0;
        int td = 0, tm = 0;
        uint8_t sd = OR_SECT_PAD, sm = OR_SECT_PAD;
        if (v > 0) {
            td = tm = v;
            sd = OR_SECT_D;
            sm = OR_SECT_DT;
        } else if (v == OR_STEP_UNDRAFTED) {
            tm = gamma + 1;
            sm = OR_SECT_DT;
        } else if (v == OR_STEP_DECODED) {
            td = 0;
            sd = OR_SECT_D;
        }
        tau[k] = td;
        tau[gamma + k] = tm;
        sect[k] = sd;
        sect[gamma + k] = sm;
        rope[k] = n + k;
        rope[gamma + k] = n + k;
    }
    return ok ? 0 : OR_ERR_STEP_MAP;
}

/* Eq. (1), written case by case.  i is the attending (row) slot, j the
 * attended (column) slot.  Padding rows and columns are zero (Sec. 3.1, the
 * sentence after Eq. (1)). */
static int eq1_visible(uint8_t si, int ti, uint8_t sj, int tj) {
    if (si == OR_SECT_PAD || sj == OR_SECT_PAD) return 0;
    if (si == OR_SECT_D && sj == OR_SECT_D && tj <= ti) return 1;   /* case 1 */
    if (si == OR_SECT_D && sj == OR_SECT_DT && tj > ti) return 1;   /* case 2 */
    if (si == OR_SECT_DT && sj == OR_SECT_D && tj < ti) return 1;   /* case 3 */
    if (si == OR_SECT_DT && sj == OR_SECT_DT && tj >= ti) return 1; /* case 4 */
    return 0;                                                       /* otherwise */
}

/* Builds tau/section/rope_pos and the response-block mask for every sequence.
 *   step_map  [Bt][gamma] int32, or NULL for the identity map mu = (1..gamma)
 *   prefix_len[Bt]
 *   tau, rope_pos [Bt][2gamma] int32; section [Bt][2gamma] uint8
 *   mask_bits [Bt][2gamma] uint64 (bit j of row i = A_ij), may be NULL
 *   dense     [Bt][2gamma][2gamma] uint8, may be NULL
 * Returns the OR of the error bits. */
int oracle_build_mask(const int32_t *step_map, const int32_t *prefix_len, int Bt, int gamma,
                      int32_t *tau, uint8_t *section, int32_t *rope_pos, uint64_t *mask_bits,
                      uint8_t *dense) {
    int S = 2 * gamma, err = 0;
    int32_t *ident = (int32_t *)malloc(sizeof(int32_t) * (size_t)(gamma > 0 ? gamma : 1));
    for (int k = 0; k < gamma; ++k) ident[k] = k + 1;
    for (int b = 0; b < Bt; ++b) {
        const int32_t *mu = step_map ? step_map + (size_t)b * gamma : ident;
        int32_t *t = tau + (size_t)b * S;
        uint8_t *s = section + (size_t)b * S;
        err |= labels_for_sequence(mu, prefix_len[b], gamma, t, s, rope_pos + (size_t)b * S);
        for (int i = 0; i < S; ++i) {
            uint64_t bits = 0;
            for (int j = 0; j < S; ++j) {
                int v = eq1_visible(s[i], t[i], s[j], t[j]);
                if (v) bits |= (uint64_t)1 << j;
                if (dense) dense[((size_t)b * S + i) * S + j] = (uint8_t)v;
            }
            if (mask_bits) mask_bits[(size_t)b * S + i] = bits;
        }
    }
    free(ident);
    return err;
}

/* ---------------------------------------------------------------------- */
/* Masked attention of the verification forward (Sec. 3.2, Sec. 3.3).     */
/* ---------------------------------------------------------------------- */

/* Widens one stored element to double.  dtype 0: IEEE binary32; dtype 1:
 * bfloat16 (the upper 16 bits of a binary32). */
static double load_elem(const void *base, size_t idx, int dtype) {
    if (dtype == 0) return (double)((const float *)base)[idx];
    uint32_t bits = (uint32_t)((const uint16_t *)base)[idx] << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

/* Rounds v to the stored type, nearest with ties to even, and stores it. */
static void store_elem(void *base, size_t idx, int dtype, double v) {
    if (dtype == 0) {
        ((float *)base)[idx] = (float)v;
        return;
    }
    double r = v;
    if (v != 0.0 && isfinite(v)) {
        int e;
        double m = frexp(v, &e);       /* v = m 2^e, 0.5 <= |m| < 1 */
        r = ldexp(nearbyint(ldexp(m, 8)), e - 8); /* 8 significant bits */
    }
    float f = (float)r;                /* exact: r has 8 significant bits */
    uint32_t bits;
    memcpy(&bits, &f, sizeof bits);
    ((uint16_t *)base)[idx] = (uint16_t)(bits >> 16);
}

/* Rotary position embedding (Su et al., RoFormer) in the rotate-half layout:
 * for i in [0, d/2) the pair (x_i, x_{i+d/2}) is rotated by the angle
 * pos * theta^(-2i/d), i.e. x_i + j x_{i+d/2} is multiplied by e^{j angle}. */
static void rope_rotate(double *x, int d, double pos, double theta) {
    int half = d / 2;
    for (int i = 0; i < half; ++i) {
        double ang = pos * pow(theta, -2.0 * i / d);
        double c = cos(ang), sn = sin(ang);
        double a = x[i], b = x[i + half];
        x[i] = a * c - b * sn;
        x[i + half] = b * c + a * sn;
    }
}

/* out[b][s][h][:] = sum_j softmax_j(scale * q.k_j) v_j over the keys the
 * row may see: every cached prefix row of sequence b (the prompt / earlier
 * blocks, visible to all response positions) read through the page table,
 * plus each new slot t with A_st = 1 under Eq. (1).  Query head h reads KV
 * head h / (Hq/Hkv).
 *
 * Layouts (row-major):
 *   q, out  [Bt][2gamma][Hq][d]
 *   k_new, v_new [Bt][2gamma][Hkv][d]
 *   k_cache, v_cache [num_pages][Hkv][page_size][d]
 *   block_table [Bt][max_pages]; prefix row p of sequence b lives in page
 *   block_table[b][p / page_size] at offset p % page_size.
 * A sequence whose prefix length is outside [0, max_pages*page_size], whose
 * needed pages are outside [0, num_pages), or whose step map is invalid gets
 * all-zero output rows and sets the matching error bit.  Padding rows are
 * zero.
 * rope_theta > 0: q and k_new hold values before the rotary embedding; each
 * q row and each k_new row of slot t is rotated at the position of slot t
 * first (the cached keys are stored rotated already).  rope_mode 1: the
 * aligned RoPE copy of Sec. 3.1 (D_k and D~_k both at n + k); rope_mode 2:
 * physical positions (slot t at n + t, the ablation of Table 4).
 * Returns the error bits. */
int oracle_verify_attention(int dtype, const void *q, const void *k_new, const void *v_new,
                            const void *k_cache, const void *v_cache, const int32_t *block_table,
                            int max_pages, int page_size, int num_pages, const int32_t *prefix_len,
                            const int32_t *step_map, int Bt, int gamma, int Hq, int Hkv, int d,
                            double scale, double rope_theta, int rope_mode, double *out, int nthreads) {
    const int S = 2 * gamma, g = Hq / Hkv;
    int err = 0;
    int32_t *tau = (int32_t *)malloc(sizeof(int32_t) * (size_t)Bt * S);
    uint8_t *sect = (uint8_t *)malloc((size_t)Bt * S);
    int32_t *rope = (int32_t *)malloc(sizeof(int32_t) * (size_t)Bt * S);
    int32_t *nvalid = (int32_t *)malloc(sizeof(int32_t) * (size_t)Bt);
    err |= oracle_build_mask(step_map, prefix_len, Bt, gamma, tau, sect, rope, NULL, NULL);

    for (int b = 0; b < Bt; ++b) {
        int n = prefix_len[b], ok = 1;
        if (n < 0 || (long long)n > (long long)max_pages * page_size) {
            err |= OR_ERR_PREFIX_LEN;
            ok = 0;
        } else {
            int npages = (n + page_size - 1) / page_size;
            for (int p = 0; p < npages; ++p) {
                int pg = block_table[(size_t)b * max_pages + p];
                if (pg < 0 || pg >= num_pages) {
                    err |= OR_ERR_PAGE;
                    ok = 0;
                }
            }
        }
        nvalid[b] = ok ? n : -1;
    }

    /* rotated copies of q and k_new when the inputs are not rotated yet */
    double *qr = NULL, *kr = NULL;
    if (rope_theta > 0.0) {
        qr = (double *)malloc(sizeof(double) * (size_t)Bt * S * Hq * d);
        kr = (double *)malloc(sizeof(double) * (size_t)Bt * S * Hkv * d);
        for (int b = 0; b < Bt; ++b) {
            for (int t = 0; t < S; ++t) {
                double pos = rope_mode == 2 ? (double)prefix_len[b] + t : (double)rope[(size_t)b * S + t];
                for (int h = 0; h < Hq; ++h) {
                    size_t o = (((size_t)b * S + t) * Hq + h) * d;
                    for (int c = 0; c < d; ++c) qr[o + c] = load_elem(q, o + c, dtype);
                    rope_rotate(qr + o, d, pos, rope_theta);
                }
                for (int h = 0; h < Hkv; ++h) {
                    size_t o = (((size_t)b * S + t) * Hkv + h) * d;
                    for (int c = 0; c < d; ++c) kr[o + c] = load_elem(k_new, o + c, dtype);
                    rope_rotate(kr + o, d, pos, rope_theta);
                }
            }
        }
    }

    long long rows = (long long)Bt * S * Hq;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#else
    (void)nthreads;
#endif
#pragma omp parallel for schedule(dynamic, 4)
    for (long long row = 0; row < rows; ++row) {
        int h = (int)(row % Hq);
        int s = (int)((row / Hq) % S);
        int b = (int)(row / ((long long)Hq * S));
        int kvh = h / g;
        double *o = out + (size_t)row * d;
        for (int c = 0; c < d; ++c) o[c] = 0.0;
        int n = nvalid[b];
        uint8_t si = sect[(size_t)b * S + s];
        if (n < 0 || si == OR_SECT_PAD) continue;

        /* gather the visible keys: (source array, element offset) pairs */
        int cap = n + S;
        size_t *koff = (size_t *)malloc(sizeof(size_t) * (size_t)cap);
        int *is_new = (int *)malloc(sizeof(int) * (size_t)cap);
        double *score = (double *)malloc(sizeof(double) * (size_t)cap);
        int cnt = 0;
        for (int p = 0; p < n; ++p) {
            int pg = block_table[(size_t)b * max_pages + p / page_size];
            koff[cnt] = (((size_t)pg * Hkv + kvh) * page_size + (size_t)(p % page_size)) * d;
            is_new[cnt] = 0;
            ++cnt;
        }
        int ti = tau[(size_t)b * S + s];
        for (int t = 0; t < S; ++t) {
            if (!eq1_visible(si, ti, sect[(size_t)b * S + t], tau[(size_t)b * S + t])) continue;
            koff[cnt] = (((size_t)b * S + t) * Hkv + kvh) * d;
            is_new[cnt] = 1;
            ++cnt;
        }
        size_t qoff = (size_t)row * d;
        /* pass 1: scaled dot products and their maximum */
        double m = -INFINITY;
        for (int j = 0; j < cnt; ++j) {
            const void *kb = is_new[j] ? k_new : k_cache;
            double acc = 0.0;
            for (int c = 0; c < d; ++c) {
                double qv = qr ? qr[qoff + c] : load_elem(q, qoff + c, dtype);
                double kv = (kr && is_new[j]) ? kr[koff[j] + c] : load_elem(kb, koff[j] + c, dtype);
                acc += qv * kv;
            }
            score[j] = acc * scale;
            if (score[j] > m) m = score[j];
        }
        /* pass 2: normalised weights times values */
        double z = 0.0;
        for (int j = 0; j < cnt; ++j) {
            score[j] = exp(score[j] - m);
            z += score[j];
        }
        for (int j = 0; j < cnt; ++j) {
            const void *vb = is_new[j] ? v_new : v_cache;
            double w = score[j] / z;
            for (int c = 0; c < d; ++c) o[c] += w * load_elem(vb, koff[j] + c, dtype);
        }
        free(koff);
        free(is_new);
        free(score);
    }
    free(tau);
    free(sect);
    free(rope);
    free(nvalid);
    free(qr);
    free(kr);
    return err;
}

/* ---------------------------------------------------------------------- */
/* Greedy acceptance (Sec. 3.2, Eq. (2) at temperature 0).                 */
/* ---------------------------------------------------------------------- */

/* logits [Bt][gamma+1][vocab] fp32, row r scores the draft with tau = r+1
 * (row gamma is only used when every draft is accepted).
 * draft  [Bt][gamma] int32 in tau order.
 * accepted_len[Bt] = number of leading drafts equal to the row argmax.
 * out_tokens[Bt][gamma+1] = accepted drafts, then the target's token at the
 * first rejected position (argmax of row a), then -1.
 * row_argmax[Bt][gamma+1] may be NULL.  Returns the error bits. */
int oracle_accept(const float *logits, const int32_t *draft, int Bt, int gamma, int vocab,
                  int32_t *accepted_len, int32_t *out_tokens, int32_t *row_argmax) {
    int err = 0;
    int32_t *am = (int32_t *)malloc(sizeof(int32_t) * (size_t)(gamma + 1));
    for (int b = 0; b < Bt; ++b) {
        for (int r = 0; r <= gamma; ++r) {
            const float *row = logits + ((size_t)b * (gamma + 1) + r) * vocab;
            int best = 0;
            double bv = (double)row[0];
            for (int v = 1; v < vocab; ++v) {
                double x = (double)row[v];
                if (isnan(bv)) break;             /* the first NaN is the maximum */
                if (isnan(x) || x > bv) {         /* strict '>': ties keep the lower index */
                    best = v;
                    bv = x;
                }
            }
            am[r] = best;
            if (row_argmax) row_argmax[(size_t)b * (gamma + 1) + r] = best;
        }
        int a = 0;
        while (a < gamma) {
            int dr = draft[(size_t)b * gamma + a];
            if (dr < 0 || dr >= vocab) {
                err |= OR_ERR_DRAFT;
                break;
            }
            if (dr != am[a]) break;
            ++a;
        }
        /* report every out-of-range draft, not only the first one reached */
        for (int r = a; r < gamma; ++r) {
            int dr = draft[(size_t)b * gamma + r];
            if (dr < 0 || dr >= vocab) err |= OR_ERR_DRAFT;
        }
        accepted_len[b] = a;
        int32_t *ot = out_tokens + (size_t)b * (gamma + 1);
        for (int r = 0; r <= gamma; ++r) ot[r] = -1;
        for (int r = 0; r < a; ++r) ot[r] = draft[(size_t)b * gamma + r];
        ot[a] = am[a];
    }
    free(am);
    return err;
}

/* ---------------------------------------------------------------------- */
/* Stochastic acceptance (Sec. 3.2, Eq. (2)).                              */
/* ---------------------------------------------------------------------- */

/* Softmax of logits/temperature over one row, in double. */
static void softmax_row(const float *x, int vocab, double inv_t, double *p) {
    double m = -INFINITY;
    for (int v = 0; v < vocab; ++v) {
        double z = (double)x[v] * inv_t;
        if (z > m) m = z;
    }
    double sum = 0.0;
    for (int v = 0; v < vocab; ++v) {
        p[v] = exp((double)x[v] * inv_t - m);
        sum += p[v];
    }
    for (int v = 0; v < vocab; ++v) p[v] /= sum;
}

/* Inverse-CDF draw from the unnormalised weights w[0..vocab): the smallest
 * v with w[0] + ... + w[v] > u * sum(w).  *margin = distance of u * sum(w)
 * to the nearest cumulative boundary, relative to sum(w). */
static int sample_index(const double *w, int vocab, double u, double *margin) {
    double total = 0.0;
    for (int v = 0; v < vocab; ++v) total += w[v];
    double t = u * total, c = 0.0;
    int pick = vocab - 1;
    double lo = 0.0, hi = total;
    for (int v = 0; v < vocab; ++v) {
        double c2 = c + w[v];
        if (c2 > t && w[v] > 0.0) {
            pick = v;
            lo = c;
            hi = c2;
            break;
        }
        c = c2;
    }
    if (margin) *margin = total > 0.0 ? fmin(t - lo, hi - t) / total : 0.0;
    return pick;
}

/* target_logits [Bt][gamma+1][vocab], draft_logits [Bt][gamma][vocab]
 * (float32); p = softmax(logits / temperature).  For r = 0..gamma-1 the
 * draft x_r (tau order) is accepted iff u_accept[b][r] < alpha_r =
 * min(1, p_theta^(r)(x_r) / p_phi^(r)(x_r)) (Eq. (2)), stopping at the first
 * rejection a.  The token at the first rejected position is drawn from the
 * residual max(0, p_theta^(a) - p_phi^(a)) renormalised (the
 * rejection-sampling correction that keeps the target distribution, Sec.
 * 3.2); when every draft is accepted it is drawn from p_theta^(gamma).  The
 * draw uses u_sample[b]: the smallest v whose cumulative weight exceeds
 * u_sample * total.  A draft id outside [0, vocab) sets OR_ERR_DRAFT and is
 * rejected (alpha 0).
 * Outputs: accepted_len[Bt], out_tokens[Bt][gamma+1] (accepted drafts, the
 * drawn token, then -1), alpha[Bt][gamma] (may be NULL; rows past the first
 * rejection are computed too), margin[Bt] (may be NULL: distance of the
 * draw's threshold to the nearest cumulative boundary, relative to the
 * total weight).  Returns the error bits. */
int oracle_accept_sampled(const float *target_logits, const float *draft_logits, const int32_t *draft,
                          const float *u_accept, const float *u_sample, double temperature, int Bt, int gamma,
                          int vocab, int32_t *accepted_len, int32_t *out_tokens, double *alpha, double *margin) {
    int err = 0;
    double inv_t = 1.0 / temperature;
    double *pt = (double *)malloc(sizeof(double) * (size_t)vocab);
    double *pd = (double *)malloc(sizeof(double) * (size_t)vocab);
    for (int b = 0; b < Bt; ++b) {
        int a = gamma;
        for (int r = 0; r < gamma; ++r) {
            int x = draft[(size_t)b * gamma + r];
            double al = 0.0;
            if (x < 0 || x >= vocab) {
                err |= OR_ERR_DRAFT;
            } else {
                softmax_row(target_logits + ((size_t)b * (gamma + 1) + r) * vocab, vocab, inv_t, pt);
                softmax_row(draft_logits + ((size_t)b * gamma + r) * vocab, vocab, inv_t, pd);
                al = pd[x] > 0.0 ? fmin(1.0, pt[x] / pd[x]) : 1.0;
            }
            if (alpha) alpha[(size_t)b * gamma + r] = al;
            if (a == gamma && !((double)u_accept[(size_t)b * gamma + r] < al)) a = r;
        }
        accepted_len[b] = a;
        int32_t *ot = out_tokens + (size_t)b * (gamma + 1);
        for (int r = 0; r <= gamma; ++r) ot[r] = r < a ? draft[(size_t)b * gamma + r] : -1;
        softmax_row(target_logits + ((size_t)b * (gamma + 1) + a) * vocab, vocab, inv_t, pt);
        if (a < gamma) {
            softmax_row(draft_logits + ((size_t)b * gamma + a) * vocab, vocab, inv_t, pd);
            double total = 0.0;
            for (int v = 0; v < vocab; ++v) {
                pd[v] = fmax(0.0, pt[v] - pd[v]);
                total += pd[v];
            }
            /* an empty residual (p_theta = p_phi) cannot reject; fall back to p_theta */
            ot[a] = sample_index(total > 0.0 ? pd : pt, vocab, (double)u_sample[b], margin ? margin + b : NULL);
        } else {
            ot[a] = sample_index(pt, vocab, (double)u_sample[b], margin ? margin + b : NULL);
        }
    }
    free(pt);
    free(pd);
    return err;
}

/* ---------------------------------------------------------------------- */
/* Commit of the accepted K/V to the paged cache (Sec. 3.2, Sec. 3.3).     */
/* ---------------------------------------------------------------------- */

/* For every layer l, sequence b, accepted draft r < a_b and KV head:
 * copy the data-slot row whose tau is r+1 into cache row n_b + r, then set
 * n_b += a_b.  Byte copies; elem_bytes is 2 or 4.
 *   k_new, v_new  [L][Bt][2gamma][Hkv][d]
 *   k_cache, v_cache [L][num_pages][Hkv][page_size][d]
 * A destination page outside the table or the pool sets OR_ERR_PAGE and that
 * row is skipped; a missing source slot sets OR_ERR_STEP_MAP and the row is
 * skipped; a negative prefix or an accepted length outside [0,gamma] leaves
 * the sequence untouched.
 * rope_theta > 0: k_new holds keys before the rotary embedding; the copied
 * key of data slot k is rotated at its position n_b + k (Sec. 3.1) and
 * rounded to the stored type, so that the cache holds rotated keys.
 * Returns the error bits. */
int oracle_kv_commit(int elem_bytes, const void *k_new, const void *v_new, int L,
                     const int32_t *step_map, const int32_t *accepted_len, void *k_cache,
                     void *v_cache, const int32_t *block_table, int max_pages, int page_size,
                     int num_pages, int32_t *prefix_len, int Bt, int gamma, int Hkv, int d,
                     double rope_theta) {
    const int S = 2 * gamma;
    int err = 0;
    size_t row_bytes = (size_t)d * elem_bytes;
    int dtype = elem_bytes == 4 ? 0 : 1;
    double *row = (double *)malloc(sizeof(double) * (size_t)(d > 0 ? d : 1));
    for (int b = 0; b < Bt; ++b) {
        int n = prefix_len[b], a = accepted_len[b];
        if (a < 0 || a > gamma) {
            err |= OR_ERR_ACCEPT_LEN;
            continue;
        }
        if (n < 0) {
            err |= OR_ERR_PREFIX_LEN;
            continue;
        }
        const int32_t *mu = step_map ? step_map + (size_t)b * gamma : NULL;
        int valid_map = mu ? step_map_row_valid(mu, gamma) : 1;
        for (int r = 0; r < a; ++r) {
            int src = -1;
            for (int k = 0; k < gamma; ++k) {
                int tk = mu ? mu[k] : k + 1;
                if (valid_map && tk == r + 1) src = k;
            }
            if (src < 0) {
                err |= OR_ERR_STEP_MAP;
                continue;
            }
            long long dst = (long long)n + r;
            long long pidx = dst / page_size;
            if (pidx >= max_pages) {
                err |= OR_ERR_PAGE;
                continue;
            }
            int pg = block_table[(size_t)b * max_pages + pidx];
            if (pg < 0 || pg >= num_pages) {
                err |= OR_ERR_PAGE;
                continue;
            }
            int off = (int)(dst % page_size);
            for (int l = 0; l < L; ++l) {
                for (int kvh = 0; kvh < Hkv; ++kvh) {
                    size_t s_el = ((((size_t)l * Bt + b) * S + src) * Hkv + kvh) * d;
                    size_t d_el = ((((size_t)l * num_pages + pg) * Hkv + kvh) * page_size + off) * d;
                    if (rope_theta > 0.0) {
                        for (int c = 0; c < d; ++c) row[c] = load_elem(k_new, s_el + c, dtype);
                        rope_rotate(row, d, (double)n + src, rope_theta);
                        for (int c = 0; c < d; ++c) store_elem(k_cache, d_el + c, dtype, row[c]);
                    } else {
                        memcpy((char *)k_cache + d_el * elem_bytes, (const char *)k_new + s_el * elem_bytes,
                               row_bytes);
                    }
                    memcpy((char *)v_cache + d_el * elem_bytes, (const char *)v_new + s_el * elem_bytes,
                           row_bytes);
                }
            }
        }
        prefix_len[b] = n + a;
    }
    free(row);
    return err;
}

/* Rotates rows of x [rows][d] in place at position pos (the oracle's RoPE,
 * exported for its pins). */
void oracle_rope_rotate(double *x, int rows, int d, double pos, double theta) {
    for (int r = 0; r < rows; ++r) rope_rotate(x + (size_t)r * d, d, pos, theta);
}

/* Number of OpenMP threads the oracle uses by default. */
int oracle_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
