/*
 * ELSAA reference oracle: plain, slow, CPU-only, fp64.
 *
 * TEST INFRASTRUCTURE ONLY. Only the tests, the smoke check and the
 * benchmark's CPU-baseline leg may load this library. The CUDA product path
 * never calls it and shares no code with it.
 *
 * One attention head at a time (Section 3: multi-head ELSAA applies the same
 * procedure independently per head). Every function follows the paper's
 * definitions step by step, in the paper's order and notation:
 *
 *   sort hash     Algorithm "sortLSH Sparse Exact Attention Branch", step Hash,
 *                 with the angular (sign of random projection) hash of
 *                 Section 3.2 / Appendix F and the Sort_LSH bits of Table 7.
 *   sort          same algorithm, step Sort (stable, non-decreasing keys).
 *   block attn    same algorithm, block loop and un-permute steps.
 *   RACE          Algorithm "RACE Low-Rank Attention Branch", every step.
 *   fusion        Eq. (5) multiplier and Eq. (6) gated fusion
 *                 (Algorithm 1, steps 6 and 8); the log-sum-exp form of the
 *                 multiplier from Algorithm "Causal ELSAA", step 6.
 *   dense         Eq. (1)-(2), exact softmax attention (for pins only).
 *
 * Readings taken where the paper is silent (each is also listed in the
 * design notes of the repository):
 *   - sort-hash bit p of a vector x is [<w_p, x> > 0], where the projection is
 *     evaluated as a sequential fp32 fused multiply-add chain over
 *     i = 0 .. d_h-1 starting from +0.0f. The CUDA path evaluates exactly the
 *     same chain, so both sides take the integer decision in the same
 *     precision. The fp64 projection sign is also computed and the number of
 *     disagreements is reported (expected to be ~0).
 *   - the code c = sum_p bit_p 2^p is ordered by its rank in the binary
 *     reflected Gray sequence ("sorted Hamming LSH", Section 3), so adjacent
 *     buckets in sort order differ in one hash bit (gray = 0: plain binary).
 *   - ties (equal keys) keep the lowest original index first (stable sort).
 *   - hypercube corner r has coordinate v_{r,b} = +1 if bit b of r is set,
 *     else -1.
 *   - the same epsilon floors O_sparse, O_lr and the multiplier; d_lr = Den
 *     without epsilon (Algorithm RACE, return step).
 *   - exp(z) is evaluated literally (Algorithm sortLSH, block step); only if
 *     a block's largest score leaves [-700, 700] is the identical shifted
 *     form exp(z - M) * exp(M) used, to stay inside the fp64 range.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ---------------------------------------------------------------- hashing */

/* Rank of code c in the binary reflected Gray sequence G(k) = k ^ (k >> 1):
 * the k with G(k) = c is the prefix XOR of c's bits from the top. */
static uint32_t gray_rank(uint32_t c) {
    uint32_t k = 0;
    while (c) {
        k ^= c;
        c >>= 1;
    }
    return k;
}

/* Sort hash of N vectors x[N][d_h] (fp32 values) with planes w[n_s][d_h].
 * key[i] = sort key of x_i. Returns the number of (vector, bit) pairs whose
 * fp64 projection sign differs from the fp32-chain sign. */
int64_t elsaa_oracle_sort_keys(const float *x, int N, int d_h, const float *w,
                               int n_s, int gray, uint16_t *key) {
    int64_t mismatches = 0;
    for (int i = 0; i < N; ++i) {
        const float *xi = x + (size_t)i * d_h;
        uint32_t c = 0;
        for (int p = 0; p < n_s; ++p) {
            const float *wp = w + (size_t)p * d_h;
            float acc = 0.0f;
            double acc64 = 0.0;
            for (int e = 0; e < d_h; ++e) {
                acc = fmaf(wp[e], xi[e], acc);
                acc64 += (double)wp[e] * (double)xi[e];
            }
            int bit = acc > 0.0f;
            int bit64 = acc64 > 0.0;
            if (bit != bit64) ++mismatches;
            c |= (uint32_t)bit << p;
        }
        key[i] = (uint16_t)(gray ? gray_rank(c) : c);
    }
    return mismatches;
}

/* ---------------------------------------------------------------- sorting */

/* Stable argsort of keys: perm[t] = original index of the t-th element in
 * non-decreasing key order, equal keys by increasing index. A plain
 * bottom-up merge sort that never lets a right-run element overtake an
 * equal left-run element, hence stable. */
void elsaa_oracle_stable_argsort(const uint16_t *key, int N, int32_t *perm) {
    for (int i = 0; i < N; ++i) perm[i] = i;
    int32_t *tmp = (int32_t *)malloc(sizeof(int32_t) * (size_t)(N > 0 ? N : 1));
    for (int width = 1; width < N; width *= 2) {
        for (int lo = 0; lo < N; lo += 2 * width) {
            int mid = lo + width < N ? lo + width : N;
            int hi = lo + 2 * width < N ? lo + 2 * width : N;
            int a = lo, b = mid, o = lo;
            while (a < mid && b < hi) {
                /* take from the left run unless the right key is strictly
                 * smaller: this keeps equal keys in their original order */
                if (key[perm[b]] < key[perm[a]]) tmp[o++] = perm[b++];
                else tmp[o++] = perm[a++];
            }
            while (a < mid) tmp[o++] = perm[a++];
            while (b < hi) tmp[o++] = perm[b++];
        }
        memcpy(perm, tmp, sizeof(int32_t) * (size_t)N);
    }
    free(tmp);
}

/* ---------------------------------------------------- sortLSH block branch */

/* Exact attention of one query against the b keys of its sorted key block.
 * q[d_h]; keys and values are the rows K[kidx[j]], V[kidx[j]], j < b.
 * Writes o[d_h] = diag(d + eps)^-1 sum_j exp(z_j) v_j, *d = sum_j exp(z_j),
 * *logd = log d. */
static void block_row(const double *q, const double *K, const double *V,
                      int d_h, const int32_t *kidx, int b, double scale,
                      double eps, double *o, double *d, double *logd) {
    double *z = (double *)malloc(sizeof(double) * (size_t)b);
    double zmax = -INFINITY;
    for (int j = 0; j < b; ++j) {
        const double *kj = K + (size_t)kidx[j] * d_h;
        double s = 0.0;
        for (int e = 0; e < d_h; ++e) s += q[e] * kj[e];
        z[j] = s * scale;
        if (z[j] > zmax) zmax = z[j];
    }
    int literal = zmax < 700.0 && zmax > -700.0;
    double shift = literal ? 0.0 : zmax;
    double den = 0.0;
    for (int e = 0; e < d_h; ++e) o[e] = 0.0;
    for (int j = 0; j < b; ++j) {
        double a = exp(z[j] - shift); /* A_t = exp(Z_t) */
        den += a;                     /* d_s = A_t 1 */
        const double *vj = V + (size_t)kidx[j] * d_h;
        for (int e = 0; e < d_h; ++e) o[e] += a * vj[e];
    }
    /* O_s = diag(d_s + eps)^-1 A_t V_s (shift-invariant form) */
    double floor_ = literal ? eps : eps * exp(-shift);
    for (int e = 0; e < d_h; ++e) o[e] /= (den + floor_);
    *logd = log(den) + shift;
    *d = literal ? den : exp(*logd);
    free(z);
}

/* Sorted key blocks that query block blk attends to: blk itself and nb
 * neighbouring sorted blocks on each side (Section 5's cost paragraph:
 * r neighbouring blocks give (2r + 1) s keys per query), clipped to the
 * T = N / b blocks that exist. The blocks are consecutive in perm_k, so the
 * keys are the sorted positions [lo b, (hi + 1) b). */
static void key_window(int blk, int nb, int T, int *lo, int *hi) {
    *lo = blk - nb > 0 ? blk - nb : 0;
    *hi = blk + nb < T - 1 ? blk + nb : T - 1;
}

/* Full sortLSH branch for one head, given the sorted orders perm_q, perm_k
 * (sorted position t -> original index). Query block t (positions
 * [t b, (t+1) b)) attends to key block t and its nb neighbours on each side.
 * Outputs are un-permuted: row perm_q[t] of O receives sorted row t.
 * N % b must be 0. */
void elsaa_oracle_sortlsh(const double *Q, const double *K, const double *V,
                          int N, int d_h, const int32_t *perm_q,
                          const int32_t *perm_k, int b, int nb, double scale,
                          double eps, double *O_sparse, double *d_sparse,
                          double *log_d_sparse) {
    for (int t = 0; t < N; ++t) {
        int lo, hi;
        key_window(t / b, nb, N / b, &lo, &hi);
        int i = perm_q[t];
        block_row(Q + (size_t)i * d_h, K, V, d_h, perm_k + (size_t)lo * b,
                  (hi - lo + 1) * b, scale, eps, O_sparse + (size_t)i * d_h,
                  d_sparse + i, log_d_sparse + i);
    }
}

/* Same branch for a subset of original query indices rows[0..n_rows). The
 * sorted position of each row is found through the inverse of perm_q. */
void elsaa_oracle_sortlsh_rows(const double *Q, const double *K,
                               const double *V, int N, int d_h,
                               const int32_t *perm_q, const int32_t *perm_k,
                               int b, int nb, double scale, double eps,
                               const int32_t *rows, int n_rows,
                               double *O_rows, double *d_rows,
                               double *logd_rows) {
    int32_t *pos = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    for (int t = 0; t < N; ++t) pos[perm_q[t]] = t;
    for (int k = 0; k < n_rows; ++k) {
        int i = rows[k];
        int lo, hi;
        key_window(pos[i] / b, nb, N / b, &lo, &hi);
        block_row(Q + (size_t)i * d_h, K, V, d_h, perm_k + (size_t)lo * b,
                  (hi - lo + 1) * b, scale, eps, O_rows + (size_t)k * d_h,
                  d_rows + k, logd_rows + k);
    }
    free(pos);
}

/* ------------------------------------------------------------ RACE branch */

/* Soft hash features of one vector x for table l:
 * [phi(x)]_r = exp(beta tanh(W x)^T v_r) / sum_r' exp(beta tanh(W x)^T v_r'),
 * r = 0 .. 2^gamma - 1, W = w_l[gamma][d_h]. The softmax is evaluated with its
 * largest logit subtracted (the same value, no overflow for large beta). */
static void race_phi(const double *x, int d_h, const double *w_l, int gamma,
                     double beta, double *phi) {
    double u[32];
    int R = 1 << gamma;
    for (int bb = 0; bb < gamma; ++bb) {
        double a = 0.0;
        for (int e = 0; e < d_h; ++e) a += w_l[(size_t)bb * d_h + e] * x[e];
        u[bb] = tanh(a);
    }
    double lmax = -INFINITY;
    for (int r = 0; r < R; ++r) {
        double l = 0.0;
        for (int bb = 0; bb < gamma; ++bb)
            l += u[bb] * (((r >> bb) & 1) ? 1.0 : -1.0);
        phi[r] = beta * l;
        if (phi[r] > lmax) lmax = phi[r];
    }
    double s = 0.0;
    for (int r = 0; r < R; ++r) {
        phi[r] = exp(phi[r] - lmax);
        s += phi[r];
    }
    for (int r = 0; r < R; ++r) phi[r] /= s;
}

/* Public feature map for tests: phi_out[L][R] of one vector. */
void elsaa_oracle_race_features(const double *x, int d_h, const double *w_race,
                                int L, int gamma, double beta,
                                double *phi_out) {
    int R = 1 << gamma;
    for (int l = 0; l < L; ++l)
        race_phi(x, d_h, w_race + (size_t)l * gamma * d_h, gamma, beta,
                 phi_out + (size_t)l * R);
}

/* Bucket summaries over all N keys: A[l][R] = Phi_K^T 1, B[l][R][d_h] =
 * Phi_K^T V, for every table l. */
void elsaa_oracle_race_summaries(const double *K, const double *V, int N,
                                 int d_h, const double *w_race, int L,
                                 int gamma, double beta, double *A,
                                 double *Bsum) {
    int R = 1 << gamma;
    double *phi = (double *)malloc(sizeof(double) * (size_t)R);
    memset(A, 0, sizeof(double) * (size_t)L * R);
    memset(Bsum, 0, sizeof(double) * (size_t)L * R * d_h);
    for (int l = 0; l < L; ++l) {
        const double *w_l = w_race + (size_t)l * gamma * d_h;
        for (int j = 0; j < N; ++j) {
            race_phi(K + (size_t)j * d_h, d_h, w_l, gamma, beta, phi);
            const double *vj = V + (size_t)j * d_h;
            for (int r = 0; r < R; ++r) {
                A[(size_t)l * R + r] += phi[r];
                double *brow = Bsum + ((size_t)l * R + r) * d_h;
                for (int e = 0; e < d_h; ++e) brow[e] += phi[r] * vj[e];
            }
        }
    }
    free(phi);
}

/* Query readout for rows[0..n_rows) (original indices) from summaries A, B:
 * Num = (1/L) sum_l Phi_Q^l B^l, Den = (1/L) sum_l Phi_Q^l A^l,
 * O_lr = diag(Den + eps)^-1 Num, d_lr = Den. */
void elsaa_oracle_race_readout_rows(const double *Q, int d_h,
                                    const double *w_race, int L, int gamma,
                                    double beta, double eps, const double *A,
                                    const double *Bsum, const int32_t *rows,
                                    int n_rows, double *O_rows,
                                    double *dlr_rows) {
    int R = 1 << gamma;
    double *phi = (double *)malloc(sizeof(double) * (size_t)R);
    double *num = (double *)malloc(sizeof(double) * (size_t)d_h);
    for (int k = 0; k < n_rows; ++k) {
        const double *qi = Q + (size_t)rows[k] * d_h;
        double den = 0.0;
        for (int e = 0; e < d_h; ++e) num[e] = 0.0;
        for (int l = 0; l < L; ++l) {
            race_phi(qi, d_h, w_race + (size_t)l * gamma * d_h, gamma, beta,
                     phi);
            for (int r = 0; r < R; ++r) {
                den += phi[r] * A[(size_t)l * R + r];
                const double *brow = Bsum + ((size_t)l * R + r) * d_h;
                for (int e = 0; e < d_h; ++e) num[e] += phi[r] * brow[e];
            }
        }
        den /= (double)L;
        for (int e = 0; e < d_h; ++e)
            O_rows[(size_t)k * d_h + e] = (num[e] / (double)L) / (den + eps);
        dlr_rows[k] = den;
    }
    free(num);
    free(phi);
}

/* ---------------------------------------------------------------- fusion */

/* Eq. (5): m = d_s / (d_s + lambda d_lr + eps); mode 1 (Sort_Lsh_RACE
 * ablation) sets m = 1. Eq. (6): O = g_s m O_s + g_lr O_lr.
 * Also returns the log-sum-exp form of m (Algorithm "Causal ELSAA" step 6)
 * in m_log for comparison. */
void elsaa_oracle_fuse_rows(int n_rows, int d_h, const double *O_s,
                            const double *d_s, const double *log_d_s,
                            const double *O_lr, const double *d_lr,
                            const double *lam, const double *g_s,
                            const double *g_lr, double eps, int mode,
                            double *O, double *m, double *m_log) {
    for (int k = 0; k < n_rows; ++k) {
        double mk = d_s[k] / (d_s[k] + lam[k] * d_lr[k] + eps);
        /* log D = logsumexp(log d_s, log lambda + log d_lr, log eps) */
        double a = log_d_s[k];
        double bterm = log(lam[k]) + log(d_lr[k]);
        double c = log(eps);
        double mx = a;
        if (bterm > mx) mx = bterm;
        if (c > mx) mx = c;
        double logD = mx + log(exp(a - mx) + exp(bterm - mx) + exp(c - mx));
        m_log[k] = exp(a - logD);
        if (mode == 1) mk = 1.0;
        m[k] = mk;
        for (int e = 0; e < d_h; ++e)
            O[(size_t)k * d_h + e] = g_s[k] * mk * O_s[(size_t)k * d_h + e] +
                                     g_lr[k] * O_lr[(size_t)k * d_h + e];
    }
}

/* ------------------------------------------------------- dense attention */

/* Eq. (1)-(2): d_i = sum_j exp(z_ij), o_i = sum_j exp(z_ij) v_j / d_i,
 * z = scale Q K^T, for rows[0..n_rows). Shifted by the row maximum. */
void elsaa_oracle_dense_rows(const double *Q, const double *K,
                             const double *V, int N, int d_h, double scale,
                             const int32_t *rows, int n_rows, double *O_rows,
                             double *logd_rows) {
    double *z = (double *)malloc(sizeof(double) * (size_t)N);
    for (int k = 0; k < n_rows; ++k) {
        const double *qi = Q + (size_t)rows[k] * d_h;
        double zmax = -INFINITY;
        for (int j = 0; j < N; ++j) {
            double s = 0.0;
            for (int e = 0; e < d_h; ++e) s += qi[e] * K[(size_t)j * d_h + e];
            z[j] = s * scale;
            if (z[j] > zmax) zmax = z[j];
        }
        double den = 0.0;
        double *o = O_rows + (size_t)k * d_h;
        for (int e = 0; e < d_h; ++e) o[e] = 0.0;
        for (int j = 0; j < N; ++j) {
            double a = exp(z[j] - zmax);
            den += a;
            for (int e = 0; e < d_h; ++e) o[e] += a * V[(size_t)j * d_h + e];
        }
        for (int e = 0; e < d_h; ++e) o[e] /= den;
        logd_rows[k] = log(den) + zmax;
    }
    free(z);
}

/* ------------------------------------------------------ top-k selector */
/*
 * An alternative selector for the sparse branch. Section 3 ("sorted Hamming
 * LSH") names learned top-k, sliding windows and global tokens as selectors
 * a future version could use in place of the sorted blocks; the paper
 * defines none of them. Reading taken here (each step also listed in the
 * design notes):
 *   1. after the hash and the stable sort of Algorithm sortLSH, block t of
 *      the sorted queries (positions [t b, (t+1) b)) and block u of the
 *      sorted keys are summarised by their sums qbar_t, kbar_u (fp32,
 *      sequential over increasing sorted position from +0.0f);
 *   2. block score s(t, u) = <qbar_t, kbar_u> (the canonical fp32 FMA chain
 *      of the sort hash); query block t takes its own key block t and the
 *      c - 1 other key blocks of largest score (equal scores: lower u);
 *   3. query i of block t scores every key j of those c blocks with
 *      <q_i, k_j> (the same chain, unscaled) and keeps the k of largest
 *      score (equal scores: lower original key index j);
 *   4. the sparse branch is the block step of Algorithm sortLSH over that
 *      set: d_s,i = sum_j exp(z_ij), O_s,i = sum_j exp(z_ij) V_j /
 *      (d_s,i + eps); RACE and the fusion are unchanged.
 * With c = 1 and k = b every query keeps its whole block: the sorted-block
 * branch. With c = N / b and k = N every query attends every key.
 */

/* The canonical fp32 chain sum_e a[e] b[e] over e = 0 .. d-1 (one rounding
 * per fused multiply-add, from +0.0f): the precision in which both this
 * oracle and the device take every selection decision. */
static float select_dot(const float *a, const float *b, int d) {
    float acc = 0.0f;
    for (int e = 0; e < d; ++e) acc = fmaf(a[e], b[e], acc);
    return acc;
}

/* Step 1: sums[t][e] = sum over sorted positions p = t b .. t b + b - 1 (in
 * that order) of x[perm[p]][e], fp32, for the N / b blocks. */
void elsaa_oracle_block_sums(const float *x, int N, int d_h,
                             const int32_t *perm, int b, float *sums) {
    int T = N / b;
    for (int t = 0; t < T; ++t)
        for (int e = 0; e < d_h; ++e) {
            float acc = 0.0f;
            for (int p = t * b; p < (t + 1) * b; ++p)
                acc = acc + x[(size_t)perm[p] * d_h + e];
            sums[(size_t)t * d_h + e] = acc;
        }
}

/* Step 2: cand[t][0] = t; cand[t][1 .. c) = the c - 1 blocks u != t of
 * largest s(t, u), in order of decreasing score (equal scores: lower u). */
void elsaa_oracle_topk_candidates(const float *qsum, const float *ksum,
                                  int T, int d_h, int c, int32_t *cand) {
    float *s = (float *)malloc(sizeof(float) * (size_t)T);
    char *taken = (char *)malloc((size_t)T);
    for (int t = 0; t < T; ++t) {
        for (int u = 0; u < T; ++u) {
            s[u] = select_dot(qsum + (size_t)t * d_h, ksum + (size_t)u * d_h,
                              d_h);
            taken[u] = 0;
        }
        cand[(size_t)t * c] = t;
        taken[t] = 1;
        for (int m = 1; m < c; ++m) {
            int best = -1;
            for (int u = 0; u < T; ++u)  /* strict >: lower u wins ties */
                if (!taken[u] && (best < 0 || s[u] > s[best])) best = u;
            cand[(size_t)t * c + m] = best;
            taken[best] = 1;
        }
    }
    free(taken);
    free(s);
}

/* Step 3 for the queries rows[0 .. n_rows) (original indices): query i at
 * sorted position p (block t = p / b) keeps the k candidate keys of largest
 * <q_i, k_j>, equal scores by lower j; sel[m][0 .. k) lists the keys of
 * rows[m] by increasing j. */
void elsaa_oracle_topk_select_rows(const float *q, const float *kx, int N,
                                   int d_h, const int32_t *perm_q,
                                   const int32_t *perm_k, int b,
                                   const int32_t *cand, int c, int k,
                                   const int32_t *rows, int n_rows,
                                   int32_t *sel) {
    int nc = c * b;
    int32_t *pos = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    int32_t *idx = (int32_t *)malloc(sizeof(int32_t) * (size_t)nc);
    float *sc = (float *)malloc(sizeof(float) * (size_t)nc);
    char *keep = (char *)malloc((size_t)nc);
    for (int p = 0; p < N; ++p) pos[perm_q[p]] = p;
    for (int r = 0; r < n_rows; ++r) {
        int i = rows[r], t = pos[i] / b;
        const float *qi = q + (size_t)i * d_h;
        for (int m = 0; m < c; ++m) {
            int u = cand[(size_t)t * c + m];
            for (int o = 0; o < b; ++o) {
                int j = perm_k[u * b + o];
                idx[m * b + o] = j;
                sc[m * b + o] = select_dot(qi, kx + (size_t)j * d_h, d_h);
            }
        }
        /* candidate a beats candidate x when its score is larger, or equal
         * with a lower key index: keep a when fewer than k candidates beat
         * it (the order is total: each key appears once) */
        for (int a = 0; a < nc; ++a) {
            int beaten = 0;
            for (int x = 0; x < nc; ++x)
                if (sc[x] > sc[a] || (sc[x] == sc[a] && idx[x] < idx[a]))
                    ++beaten;
            keep[a] = beaten < k;
        }
        /* the kept keys by increasing index */
        int32_t *out = sel + (size_t)r * k;
        int n = 0;
        for (int a = 0; a < nc; ++a)
            if (keep[a]) out[n++] = idx[a];
        for (int x = 1; x < n; ++x)  /* insertion sort */
            for (int y = x; y > 0 && out[y - 1] > out[y]; --y) {
                int32_t tmp = out[y];
                out[y] = out[y - 1];
                out[y - 1] = tmp;
            }
    }
    free(keep);
    free(sc);
    free(idx);
    free(pos);
}

/* Step 4 for rows[0 .. n_rows): the block step of Algorithm sortLSH over
 * each row's selected keys sel[m][0 .. k) (as step 3 lists them). */
void elsaa_oracle_sparse_sets_rows(const double *Q, const double *K,
                                   const double *V, int d_h,
                                   const int32_t *sel, int k, double scale,
                                   double eps, const int32_t *rows,
                                   int n_rows, double *O_rows,
                                   double *d_rows, double *logd_rows) {
    for (int m = 0; m < n_rows; ++m)
        block_row(Q + (size_t)rows[m] * d_h, K, V, d_h, sel + (size_t)m * k,
                  k, scale, eps, O_rows + (size_t)m * d_h, d_rows + m,
                  logd_rows + m);
}
