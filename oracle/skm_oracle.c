/*
 * skm_oracle.c -- plain, slow CPU oracle for the Lloyd k-means hot path of
 * "Stop Indexing at Full Precision: Revisiting Clustering for Vector
 * Embeddings" (arxiv 2608.14648).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * CPU-baseline leg of bench.py may load this library.  It shares no code,
 * header, table or constant with the CUDA library; it is compiled with
 * -O2 -ffp-contract=off and contains no blocking, fusion or reordering beyond
 * what each definition states.  Rows are spread over OpenMP threads; every
 * per-row computation is a plain sequential loop.
 *
 * Where the method has a plain definition (the nearest-centroid assignment of
 * Section 2.3 STEP 2, the mean of members of STEP 3, the SQ8 integer code-space
 * distance of Section 3.1) the oracle is that definition: fp64 or exact
 * integer arithmetic, ties to the lowest centroid index.  Where the method is
 * an encoding or an estimator (SQ8 codes, RabitQ 1-bit codes, the centroid SQ4
 * codes and Eq. final:rabitq), the oracle takes the paper's steps in order.
 * Where a float result decides an integer (a code, an argmin over estimated
 * distances), the oracle performs that float step in fp32 in the fixed
 * operation order the method is specified with, so that both sides take the
 * decision in the same precision.
 *
 * Parity status of each function is stated in its comment; the pins live in
 * tests/test_oracle_pins.py.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

int or_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void or_set_num_threads(int t) {
#ifdef _OPENMP
    if (t > 0) omp_set_num_threads(t);
#else
    (void)t;
#endif
}

static inline float bf16_bits_to_float(uint16_t b) {
    uint32_t u = ((uint32_t)b) << 16;
    float f;
    memcpy(&f, &u, 4);
    return f;
}

/* ------------------------------------------------------------------------ */
/* Section 2.3 STEP 2: nearest centroid under squared L2, plain definition.  */
/* ------------------------------------------------------------------------ */

/* dist(x, c) = sum_i (x_i - c_i)^2 in fp64; argmin over all k, ties to the
 * lowest index.  best/second receive the smallest and second-smallest fp64
 * distances (second is used only to report top-1/top-2 gaps, Fig. 3).
 * Pinned: brute force, scipy cdist, K=1, N=K identity, duplicates. */
void or_assign_f32(const float *X, int64_t n, int d, const float *C, int k,
                   int32_t *assign, double *best, double *second) {
#pragma omp parallel for schedule(dynamic, 64)
    for (int64_t p = 0; p < n; ++p) {
        const float *x = X + p * (int64_t)d;
        double b1 = INFINITY, b2 = INFINITY;
        int32_t a = -1;
        for (int j = 0; j < k; ++j) {
            const float *c = C + (int64_t)j * d;
            double s = 0.0;
            for (int i = 0; i < d; ++i) {
                double t = (double)x[i] - (double)c[i];
                s += t * t;
            }
            if (s < b1) {
                b2 = b1;
                b1 = s;
                a = j;
            } else if (s < b2) {
                b2 = s;
            }
        }
        assign[p] = a;
        if (best) best[p] = b1;
        if (second) second[p] = b2;
    }
}

/* Same definition for points stored as bfloat16 bit patterns (the projected
 * points of the PCA workload, stored in bf16; every bf16 value is exact in
 * fp32 and fp64). */
void or_assign_bf16(const uint16_t *Xb, int64_t n, int d, const float *C, int k,
                    int32_t *assign, double *best, double *second) {
#pragma omp parallel for schedule(dynamic, 64)
    for (int64_t p = 0; p < n; ++p) {
        const uint16_t *x = Xb + p * (int64_t)d;
        double b1 = INFINITY, b2 = INFINITY;
        int32_t a = -1;
        for (int j = 0; j < k; ++j) {
            const float *c = C + (int64_t)j * d;
            double s = 0.0;
            for (int i = 0; i < d; ++i) {
                double t = (double)bf16_bits_to_float(x[i]) - (double)c[i];
                s += t * t;
            }
            if (s < b1) {
                b2 = b1;
                b1 = s;
                a = j;
            } else if (s < b2) {
                b2 = s;
            }
        }
        assign[p] = a;
        if (best) best[p] = b1;
        if (second) second[p] = b2;
    }
}

/* ------------------------------------------------------------------------ */
/* Section 3.1 "SQ8 and SQ4": scalar quantization.                           */
/* The paper fits one global bias/scale; the workload here fits them per     */
/* dimension (b_i = min over points, s_i = (max - b_i) / 255).  A dimension  */
/* with max == min gets s_i = 1.                                             */
/* ------------------------------------------------------------------------ */

/* Section 3.1 "SQ8 and SQ4": B-bit codes have L = 2^B - 1 levels; per
 * dimension b = min x, s = (max x - b) / L (s = 1 when flat). */
void or_sq_fit(const float *X, int64_t n, int d, int levels, float *b, float *s) {
    for (int i = 0; i < d; ++i) {
        float lo = INFINITY, hi = -INFINITY;
        for (int64_t p = 0; p < n; ++p) {
            float v = X[p * (int64_t)d + i];
            if (v < lo) lo = v;
            if (v > hi) hi = v;
        }
        float sc = (hi - lo) / (float)levels;
        if (!(sc > 0.0f)) sc = 1.0f;
        b[i] = lo;
        s[i] = sc;
    }
}

void or_sq8_fit(const float *X, int64_t n, int d, float *b, float *s) {
    or_sq_fit(X, n, d, 255, b, s);
}

/* code = clip(round((x - b) / s), 0, 255), fp32 arithmetic, rounding half to
 * even.  Pinned: grid data reproduces codes; |decode - x| <= s/2. */
void or_sq_encode(const float *X, int64_t n, int d, int levels, const float *b, const float *s,
                  uint8_t *codes) {
    const float top = (float)levels;
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < n; ++p) {
        for (int i = 0; i < d; ++i) {
            float t = (X[p * (int64_t)d + i] - b[i]) / s[i];
            float q = rintf(t);
            if (!(q >= 0.0f)) q = 0.0f;
            if (q > top) q = top;
            codes[p * (int64_t)d + i] = (uint8_t)q;
        }
    }
}

void or_sq8_encode(const float *X, int64_t n, int d, const float *b, const float *s,
                   uint8_t *codes) {
    or_sq_encode(X, n, d, 255, b, s, codes);
}

/* Reconstruction x_i ~ code_i * s_i + b_i (fp32). */
void or_sq8_decode(const uint8_t *codes, int64_t n, int d, const float *b, const float *s,
                   float *Y) {
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < n; ++p)
        for (int i = 0; i < d; ++i)
            Y[p * (int64_t)d + i] = (float)codes[p * (int64_t)d + i] * s[i] + b[i];
}

/* Code-domain squared L2, exact in integers: sum_i (xbar_i - cbar_i)^2.
 * Pinned: exact int64 recomputation through numpy; brute force. */
void or_assign_sq8(const uint8_t *Xc, int64_t n, int d, const uint8_t *Cc, int k,
                   int32_t *assign, int64_t *best) {
#pragma omp parallel for schedule(dynamic, 64)
    for (int64_t p = 0; p < n; ++p) {
        const uint8_t *x = Xc + p * (int64_t)d;
        int64_t b1 = INT64_MAX;
        int32_t a = -1;
        for (int j = 0; j < k; ++j) {
            const uint8_t *c = Cc + (int64_t)j * d;
            int64_t s = 0;
            for (int i = 0; i < d; ++i) {
                int64_t t = (int64_t)x[i] - (int64_t)c[i];
                s += t * t;
            }
            if (s < b1) {
                b1 = s;
                a = j;
            }
        }
        assign[p] = a;
        if (best) best[p] = b1;
    }
}

/* STEP 3 in the quantized domain: per-dimension average of member codes,
 * rounded half to even in exact integer arithmetic.  Empty clusters keep
 * their codes.  Pinned: brute-force mean + rounding. */
void or_update_sq8(const uint8_t *Xc, int64_t n, int d, const int32_t *assign, int k,
                   uint8_t *C_inout, int64_t *counts) {
    int64_t *S = (int64_t *)calloc((size_t)k * d, sizeof(int64_t));
    for (int j = 0; j < k; ++j) counts[j] = 0;
    for (int64_t p = 0; p < n; ++p) {
        int32_t a = assign[p];
        counts[a] += 1;
        for (int i = 0; i < d; ++i) S[(int64_t)a * d + i] += Xc[p * (int64_t)d + i];
    }
    for (int j = 0; j < k; ++j) {
        int64_t m = counts[j];
        if (m == 0) continue;
        for (int i = 0; i < d; ++i) {
            int64_t t = S[(int64_t)j * d + i];
            int64_t q = t / m, r = t % m; /* t >= 0 */
            if (2 * r > m || (2 * r == m && (q & 1))) q += 1;
            C_inout[(int64_t)j * d + i] = (uint8_t)q;
        }
    }
    free(S);
}

/* ------------------------------------------------------------------------ */
/* STEP 3: centroid = mean of its members (fp64 sums, rounded to fp32).      */
/* Empty clusters keep their previous centroid.                              */
/* ------------------------------------------------------------------------ */

static void update_mean_common(const float *X, const uint16_t *Xb, int64_t n, int d,
                               const int32_t *assign, int k, float *C_inout,
                               int64_t *counts) {
    double *S = (double *)calloc((size_t)k * d, sizeof(double));
    for (int j = 0; j < k; ++j) counts[j] = 0;
    for (int64_t p = 0; p < n; ++p) {
        int32_t a = assign[p];
        counts[a] += 1;
        for (int i = 0; i < d; ++i) {
            double v = X ? (double)X[p * (int64_t)d + i]
                         : (double)bf16_bits_to_float(Xb[p * (int64_t)d + i]);
            S[(int64_t)a * d + i] += v;
        }
    }
    for (int j = 0; j < k; ++j) {
        if (counts[j] == 0) continue;
        for (int i = 0; i < d; ++i)
            C_inout[(int64_t)j * d + i] = (float)(S[(int64_t)j * d + i] / (double)counts[j]);
    }
    free(S);
}

void or_update_f32(const float *X, int64_t n, int d, const int32_t *assign, int k,
                   float *C_inout, int64_t *counts) {
    update_mean_common(X, NULL, n, d, assign, k, C_inout, counts);
}

void or_update_bf16(const uint16_t *Xb, int64_t n, int d, const int32_t *assign, int k,
                    float *C_inout, int64_t *counts) {
    update_mean_common(NULL, Xb, n, d, assign, k, C_inout, counts);
}

/* k-means objective (WCSS, Section 4): sum_n ||x_n - c_{a_n}||^2 in fp64. */
double or_objective_f32(const float *X, int64_t n, int d, const float *C,
                        const int32_t *assign) {
    double tot = 0.0;
#pragma omp parallel for reduction(+ : tot) schedule(static)
    for (int64_t p = 0; p < n; ++p) {
        const float *x = X + p * (int64_t)d;
        const float *c = C + (int64_t)assign[p] * d;
        double s = 0.0;
        for (int i = 0; i < d; ++i) {
            double t = (double)x[i] - (double)c[i];
            s += t * t;
        }
        tot += s;
    }
    return tot;
}

double or_objective_bf16(const uint16_t *Xb, int64_t n, int d, const float *C,
                         const int32_t *assign) {
    double tot = 0.0;
#pragma omp parallel for reduction(+ : tot) schedule(static)
    for (int64_t p = 0; p < n; ++p) {
        const uint16_t *x = Xb + p * (int64_t)d;
        const float *c = C + (int64_t)assign[p] * d;
        double s = 0.0;
        for (int i = 0; i < d; ++i) {
            double t = (double)bf16_bits_to_float(x[i]) - (double)c[i];
            s += t * t;
        }
        tot += s;
    }
    return tot;
}

/* ------------------------------------------------------------------------ */
/* Section 3.1 "RabitQ": 1-bit codes of the centred data points, SQ4 codes   */
/* of the centred centroids, Eq. l2_decomp / rabitq_l2 / final:rabitq.       */
/* ------------------------------------------------------------------------ */

/* Dataset mean m (fp64 sum, rounded to fp32). */
/* The dataset mean m of Section 3.1 "RabitQ" in exact fixed point (the      */
/* paper fixes no arithmetic for it): with 2^(E-1) <= max |x| < 2^E over all  */
/* coordinates (frexp) and L = ceil(log2 n), s = 61 - L - E (0 when every x   */
/* is 0); S_c = sum over the rows of rint(x_rc 2^s) as exact int64 (each      */
/* term below 2^(61-L) in magnitude); m_c = fl32(fl64(S_c) / (n 2^s)).  Row   */
/* shards summed at the same s give the same S_c.                            */
/* Parity: pinned against the fp64 mean (|m - mean| <= 2^-(s+1) + half an    */
/* fp32 ulp), exact means of grid data, and the shard sums.                  */
int or_mean_scale(float amax, int64_t n) {
    if (!(amax > 0.0f)) return 0;
    int E = 0;
    (void)frexpf(amax, &E); /* amax = f 2^E, f in [0.5, 1) */
    int L = 0;
    while (((int64_t)1 << L) < n) ++L;
    return 61 - L - E;
}

void or_column_sums_fixed(const float *X, int64_t n, int d, int s, int64_t *S) {
    for (int i = 0; i < d; ++i) {
        int64_t acc = 0;
        for (int64_t p = 0; p < n; ++p) acc += (int64_t)rint(ldexp((double)X[p * (int64_t)d + i], s));
        S[i] += acc;
    }
}

void or_mean_from_sums(const int64_t *S, int64_t n, int d, int s, float *m) {
    const double den = ldexp((double)n, s);
    for (int i = 0; i < d; ++i) m[i] = (float)((double)S[i] / den);
}

void or_rbq1_mean(const float *X, int64_t n, int d, float *m) {
    float amax = 0.0f;
    for (int64_t t = 0; t < n * (int64_t)d; ++t) amax = fmaxf(amax, fabsf(X[t]));
    const int s = or_mean_scale(amax, n);
    int64_t *S = (int64_t *)calloc((size_t)d, sizeof(int64_t));
    or_column_sums_fixed(X, n, d, s, S);
    or_mean_from_sums(S, n, d, s, m);
    free(S);
}

/* Per point: r = x - m (fp32); bit i = (r_i > 0), packed little-endian into
 * 32-bit words (bit j of word w is dimension 32w + j); nx2 = ||r||^2;
 * <xbar, x> = ||r||_1 / (sqrt(d) ||r||) so F = ||r|| / <xbar, x>
 * = sqrt(d) ||r||^2 / ||r||_1 (0 when r = 0); popx = number of set bits.
 * Pinned: exact reconstruction on sign-constant residuals, radius >= ||r||. */
void or_rbq1_encode(const float *X, int64_t n, int d, const float *m, uint32_t *codes,
                    float *nx2, float *F, int32_t *popx) {
    const int W = (d + 31) / 32;
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < n; ++p) {
        uint32_t *cw = codes + p * (int64_t)W;
        for (int w = 0; w < W; ++w) cw[w] = 0u;
        double s2 = 0.0, s1 = 0.0;
        int32_t pc = 0;
        for (int i = 0; i < d; ++i) {
            float r = X[p * (int64_t)d + i] - m[i];
            if (r > 0.0f) {
                cw[i / 32] |= (1u << (i % 32));
                pc += 1;
            }
            s2 += (double)r * (double)r;
            s1 += fabs((double)r);
        }
        nx2[p] = (float)s2;
        F[p] = (s1 > 0.0) ? (float)(sqrt((double)d) * s2 / s1) : 0.0f;
        popx[p] = pc;
    }
}

/* ||rho||^2 in fp64 in a fixed order: per 32-dimension block (zero-padded)
 * the squares are summed pairwise, v[l] += v[l + o] for o = 16, 8, 4, 2, 1,
 * and the block sums are added in increasing block order.  The paper fixes
 * no summation order; this one is the library's, so both sides agree bit for
 * bit.  Pinned against the sequential fp64 sum (relative 1e-14). */
static double sumsq_blocked(const float *r, int d) {
    double q2 = 0.0;
    for (int w = 0; w < (d + 31) / 32; ++w) {
        double v[32];
        for (int l = 0; l < 32; ++l) {
            int i = 32 * w + l;
            v[l] = (i < d) ? (double)r[i] * (double)r[i] : 0.0;
        }
        for (int o = 16; o >= 1; o >>= 1)
            for (int l = 0; l < o; ++l) v[l] = v[l] + v[l + o];
        q2 = q2 + v[0];
    }
    return q2;
}

double or_sumsq_blocked(const float *r, int d) { return sumsq_blocked(r, d); }

/* Centroid side, once per iteration: rho = c - m (fp32); per-centroid SQ4
 * with b = min rho, s = (max rho - b) / 15 (s = 1 when flat); ybar_i =
 * clip(round((rho_i - b) / s), 0, 15) with rounding half to even;
 * sumy = sum ybar; ny2 = ||rho||^2 (fp64, blocked order above, rounded to
 * fp32). */
void or_rbq1_centroid_sq4(const float *C, int k, int d, const float *m, uint8_t *ybar,
                          float *b, float *s, int32_t *sumy, float *ny2) {
    float *rho = (float *)malloc(sizeof(float) * (size_t)d);
    for (int j = 0; j < k; ++j) {
        const float *c = C + (int64_t)j * d;
        float lo = INFINITY, hi = -INFINITY;
        for (int i = 0; i < d; ++i) {
            float r = c[i] - m[i];
            rho[i] = r;
            if (r < lo) lo = r;
            if (r > hi) hi = r;
        }
        double q2 = sumsq_blocked(rho, d);
        float sc = (hi - lo) / 15.0f;
        if (!(sc > 0.0f)) sc = 1.0f;
        int32_t sy = 0;
        for (int i = 0; i < d; ++i) {
            float r = c[i] - m[i];
            float q = rintf((r - lo) / sc);
            if (!(q >= 0.0f)) q = 0.0f;
            if (q > 15.0f) q = 15.0f;
            ybar[(int64_t)j * d + i] = (uint8_t)q;
            sy += (int32_t)q;
        }
        b[j] = lo;
        s[j] = sc;
        sumy[j] = sy;
        ny2[j] = (float)q2;
    }
    free(rho);
}

/* Eq. final:rabitq into Eq. rabitq_l2, fp32, in this fixed order (the paper
 * fixes none; 1/sqrt(d) is folded into the centroid's SQ4 scale and bias):
 *   P   = sum_i xbar_i * ybar_i                      (exact integer)
 *   isd = 1/sqrt(d) rounded once to fp32
 *   sd  = s * isd,  bd = b * isd                     (per centroid)
 *   u   = fma(sd, 2P - sum ybar, bd * (2 popx - d))  (= <xbar, y_r - m> estimate)
 *   est = fma(-2 F, u, nx2 + ny2)                    (Eq. rabitq_l2)
 * argmin over est, ties to the lowest index. */
void or_rbq1_assign(const uint32_t *codes, const float *nx2, const float *F,
                    const int32_t *popx, int64_t n, int d, const uint8_t *ybar,
                    const float *b, const float *s, const int32_t *sumy,
                    const float *ny2, int k, int32_t *assign, float *est_best) {
    const int W = (d + 31) / 32;
    const float isd = (float)(1.0 / sqrt((double)d));
#pragma omp parallel for schedule(dynamic, 16)
    for (int64_t p = 0; p < n; ++p) {
        const uint32_t *cw = codes + p * (int64_t)W;
        const float pc = (float)(2 * popx[p] - d);
        const float f2 = -2.0f * F[p];
        float best = INFINITY;
        int32_t a = -1;
        for (int j = 0; j < k; ++j) {
            const uint8_t *y = ybar + (int64_t)j * d;
            int32_t P = 0;
            for (int i = 0; i < d; ++i)
                if ((cw[i / 32] >> (i % 32)) & 1u) P += y[i];
            const float sd = s[j] * isd;
            const float bd = b[j] * isd;
            const float u = fmaf(sd, (float)(2 * P - sumy[j]), bd * pc);
            const float est = fmaf(f2, u, nx2[p] + ny2[j]);
            if (est < best) {
                best = est;
                a = j;
            }
        }
        assign[p] = a;
        if (est_best) est_best[p] = best;
    }
}

/* Symmetric 1-bit variant (the centroid binarized like a point; XOR +
 * POPCOUNT).  Applying RabitQ's estimate <o, q> ~ <obar, q> / <obar, o> to
 * both unit vectors gives <x - m, y - m> ~ F_x F_y <obar_x, obar_y> with
 * obar = (2 bit - 1) / sqrt(d), i.e. F_x F_y (d - 2 h) / d for the Hamming
 * distance h = popc(xbar XOR ybar).  Centroid side, once per assignment:
 * rho = c - m (fp32), bits (rho_i > 0), ny2 = ||rho||^2 in the blocked fp64
 * order, l1 = ||rho||_1 in the same blocked order, and
 *   fy = fl32((ny2 / l1) / sqrt(d))   (fp64; fy = 0 when l1 = 0)  = F_y / d.
 * Estimate, fp32, in this order: u = fy * (float)(d - 2h) (exact integer),
 * est = fma(-2 F_x, u, nx2 + ny2); argmin, ties to the lowest index. */
static double sumabs_blocked(const float *r, int d) {
    double q = 0.0;
    for (int w = 0; w < (d + 31) / 32; ++w) {
        double v[32];
        for (int l = 0; l < 32; ++l) {
            int i = 32 * w + l;
            v[l] = (i < d) ? fabs((double)r[i]) : 0.0;
        }
        for (int o = 16; o >= 1; o >>= 1)
            for (int l = 0; l < o; ++l) v[l] = v[l] + v[l + o];
        q = q + v[0];
    }
    return q;
}

void or_rbq1_centroid_sym(const float *C, int k, int d, const float *m, uint32_t *ybits, float *fy,
                          float *ny2) {
    const int W = (d + 31) / 32;
    float *rho = (float *)malloc(sizeof(float) * (size_t)d);
    for (int j = 0; j < k; ++j) {
        uint32_t *yw = ybits + (int64_t)j * W;
        for (int w = 0; w < W; ++w) yw[w] = 0u;
        for (int i = 0; i < d; ++i) {
            rho[i] = C[(int64_t)j * d + i] - m[i];
            if (rho[i] > 0.0f) yw[i / 32] |= 1u << (i % 32);
        }
        const double q2 = sumsq_blocked(rho, d);
        const double l1 = sumabs_blocked(rho, d);
        ny2[j] = (float)q2;
        fy[j] = (l1 > 0.0) ? (float)((q2 / l1) / sqrt((double)d)) : 0.0f;
    }
    free(rho);
}

void or_rbq1_assign_sym(const uint32_t *codes, const float *nx2, const float *F, int64_t n, int d,
                        const uint32_t *ybits, const float *fy, const float *ny2, int k, int32_t *assign,
                        float *est_best) {
    const int W = (d + 31) / 32;
#pragma omp parallel for schedule(dynamic, 16)
    for (int64_t p = 0; p < n; ++p) {
        const uint32_t *cw = codes + p * (int64_t)W;
        const float f2 = -2.0f * F[p];
        float best = INFINITY;
        int32_t a = -1;
        for (int j = 0; j < k; ++j) {
            int h = 0; /* Hamming distance, bit by bit */
            for (int i = 0; i < d; ++i)
                h += (int)(((cw[i / 32] ^ ybits[(int64_t)j * W + i / 32]) >> (i % 32)) & 1u);
            const float u = fy[j] * (float)(d - 2 * h);
            const float est = fmaf(f2, u, nx2[p] + ny2[j]);
            if (est < best) {
                best = est;
                a = j;
            }
        }
        assign[p] = a;
        if (est_best) est_best[p] = best;
    }
}

/* Fixed-point exponent for the decode-average: e = 24 - ceil(log2 max F),
 * so F * 2^e <= 2^24 (the largest F keeps its 24-bit fp32 precision) and
 * sums over up to 2^24 members stay exact in int64; e = 0 when every F is 0. */
int or_rbq1_exponent(const float *F, int64_t n) {
    float mx = 0.0f;
    for (int64_t p = 0; p < n; ++p)
        if (F[p] > mx) mx = F[p];
    if (!(mx > 0.0f)) return 0;
    int ex;
    double fr = frexp((double)mx, &ex); /* mx = fr * 2^ex, fr in [0.5, 1) */
    int c = (fr == 0.5) ? ex - 1 : ex;  /* ceil(log2 mx) */
    return 24 - c;
}

/* Fused decode-average (Section 3.1 "RabitQ", last paragraph): the member
 * x_r is decoded as m_i + (1/sqrt(d)) F (2 xbar_i - 1) and the members are
 * averaged.  F enters as the integer Fq = round(F 2^e), so the sum over the
 * members is exact and independent of order:
 *   T_i = sum Fq xbar_i,  U = sum Fq,  sum F (2 xbar_i - 1) = (2 T_i - U) 2^-e
 *   c_i = m_i + (2 T_i - U) * f,  f = (2^-e / sqrt(d)) / count   (fp64, then fp32)
 * (one fp64 factor per cluster: 1/sqrt(d) rounded once, scaled by 2^-e exactly,
 * divided by the count; the paper fixes no evaluation order).
 * Empty clusters keep their centroid.  Pinned against the fp64 mean of
 * decoded vectors (relative 1e-9) and the exact-reconstruction case. */
void or_rbq1_update(const uint32_t *codes, const float *F, int64_t n, int d,
                    const float *m, int e, const int32_t *assign, int k, float *C_inout,
                    int64_t *counts) {
    const int W = (d + 31) / 32;
    const double isd = 1.0 / sqrt((double)d);
    int64_t *T = (int64_t *)calloc((size_t)k * d, sizeof(int64_t));
    int64_t *U = (int64_t *)calloc((size_t)k, sizeof(int64_t));
    for (int j = 0; j < k; ++j) counts[j] = 0;
    for (int64_t p = 0; p < n; ++p) {
        int32_t a = assign[p];
        int64_t fq = (int64_t)llrint(ldexp((double)F[p], e));
        counts[a] += 1;
        U[a] += fq;
        const uint32_t *cw = codes + p * (int64_t)W;
        for (int i = 0; i < d; ++i)
            if ((cw[i / 32] >> (i % 32)) & 1u) T[(int64_t)a * d + i] += fq;
    }
    for (int j = 0; j < k; ++j) {
        if (counts[j] == 0) continue;
        const double f = ldexp(isd, -e) / (double)counts[j];
        for (int i = 0; i < d; ++i) {
            const double v = (double)(2 * T[(int64_t)j * d + i] - U[j]);
            C_inout[(int64_t)j * d + i] = (float)((double)m[i] + v * f);
        }
    }
    free(T);
    free(U);
}

/* ------------------------------------------------------------------------ */
/* Section 3.1 "JLT / PCA" and the rotation of "SuperKMeans": projection     */
/* Y = (X - mu) P, fp64.                                                     */
/* ------------------------------------------------------------------------ */

void or_project(const float *X, int64_t n, int d, const float *mu, const float *P,
                int dout, double *Y) {
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < n; ++p) {
        const float *x = X + p * (int64_t)d;
        double *y = Y + p * (int64_t)dout;
        for (int j = 0; j < dout; ++j) y[j] = 0.0;
        for (int i = 0; i < d; ++i) {
            double xi = (double)x[i] - (mu ? (double)mu[i] : 0.0);
            for (int j = 0; j < dout; ++j) y[j] += xi * (double)P[(int64_t)i * dout + j];
        }
    }
}

/* Mean and population covariance (1/n) sum (x - mu)(x - mu)^T, fp64. */
void or_mean_cov(const float *X, int64_t n, int d, double *mu, double *cov) {
    for (int i = 0; i < d; ++i) {
        double s = 0.0;
        for (int64_t p = 0; p < n; ++p) s += (double)X[p * (int64_t)d + i];
        mu[i] = s / (double)n;
    }
#pragma omp parallel for schedule(dynamic, 4)
    for (int i = 0; i < d; ++i) {
        for (int j = 0; j <= i; ++j) {
            double s = 0.0;
            for (int64_t p = 0; p < n; ++p)
                s += ((double)X[p * (int64_t)d + i] - mu[i]) * ((double)X[p * (int64_t)d + j] - mu[j]);
            cov[(int64_t)i * d + j] = s / (double)n;
            cov[(int64_t)j * d + i] = s / (double)n;
        }
    }
}

/* Round fp64 values to bfloat16 (8 significant bits, half to even). */
void or_round_bf16(const double *y, int64_t n, uint16_t *out) {
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < n; ++p) {
        double v = y[p];
        float f;
        if (v == 0.0 || !isfinite(v)) {
            f = (float)v;
        } else {
            int ex;
            double fr = frexp(v, &ex); /* |fr| in [0.5, 1) */
            double q = rint(ldexp(fr, 8));
            f = (float)ldexp(q, ex - 8);
        }
        uint32_t u;
        memcpy(&u, &f, 4);
        out[p] = (uint16_t)(u >> 16);
    }
}

/* ------------------------------------------------------------------------ */
/* Section 2.3 STEP 3: empty clusters are handled by splitting large ones.   */
/* The paper only says that splitting large clusters helps; the library's   */
/* reading: clusters left empty by an update are visited in increasing      */
/* index order; each takes the current largest cluster L (most members,     */
/* ties to the lowest index; nothing is done once L has fewer than 2) and   */
/* the two become L's centroid moved symmetrically by a relative step       */
/* eps = 2^-10 with alternating signs per dimension:                         */
/*   new_j[i] = c_L[i] (1 + s_i eps),  new_L[i] = c_L[i] (1 - s_i eps),       */
/*   s_i = +1 for even i, -1 for odd i  (fp32 centroids, one rounding each); */
/* SQ8 code centroids move by one code step instead (clipped to [0, 255]).  */
/* L keeps ceil(n_L / 2) members and j receives floor(n_L / 2) for the       */
/* choice of later splits; the reported counts are not changed.             */
/* ------------------------------------------------------------------------ */
int or_split_empty_f32(float *C, const int64_t *counts, int k, int d) {
    int64_t *w = (int64_t *)malloc(sizeof(int64_t) * (size_t)k);
    int nsplit = 0;
    for (int j = 0; j < k; ++j) w[j] = counts[j];
    const float up = 1.0f + 0x1p-10f, dn = 1.0f - 0x1p-10f;
    for (int j = 0; j < k; ++j) {
        if (counts[j] != 0) continue;
        int L = 0;
        for (int t = 1; t < k; ++t)
            if (w[t] > w[L]) L = t;
        if (w[L] < 2) break;
        for (int i = 0; i < d; ++i) {
            const float c = C[(int64_t)L * d + i];
            const int even = (i % 2) == 0;
            C[(int64_t)j * d + i] = c * (even ? up : dn);
            C[(int64_t)L * d + i] = c * (even ? dn : up);
        }
        w[j] = w[L] / 2;
        w[L] = w[L] - w[j];
        nsplit += 1;
    }
    free(w);
    return nsplit;
}

int or_split_empty_sq8(uint8_t *C, const int64_t *counts, int k, int d) {
    int64_t *w = (int64_t *)malloc(sizeof(int64_t) * (size_t)k);
    int nsplit = 0;
    for (int j = 0; j < k; ++j) w[j] = counts[j];
    for (int j = 0; j < k; ++j) {
        if (counts[j] != 0) continue;
        int L = 0;
        for (int t = 1; t < k; ++t)
            if (w[t] > w[L]) L = t;
        if (w[L] < 2) break;
        for (int i = 0; i < d; ++i) {
            const int c = C[(int64_t)L * d + i];
            const int s = (i % 2) == 0 ? 1 : -1;
            int a = c + s, b = c - s;
            C[(int64_t)j * d + i] = (uint8_t)(a < 0 ? 0 : (a > 255 ? 255 : a));
            C[(int64_t)L * d + i] = (uint8_t)(b < 0 ? 0 : (b > 255 ? 255 : b));
        }
        w[j] = w[L] / 2;
        w[L] = w[L] - w[j];
        nsplit += 1;
    }
    free(w);
    return nsplit;
}

/* ------------------------------------------------------------------------ */
/* Randomized Hadamard rotation (a structured random orthogonal transform,   */
/* used in place of a dense random rotation before RabitQ / SuperKMeans,    */
/* Section 3.1): y = (1/sqrt(D)) H_D diag(sigma) [x - mean ; 0], with D the  */
/* smallest power of two >= d (the row is zero-padded), H_D the Sylvester    */
/* Hadamard matrix (H_1 = 1, H_2m = [[H_m, H_m], [H_m, -H_m]]) and sigma a   */
/* given +-1 vector.  fp64 in-place fast Walsh-Hadamard transform, then one */
/* rounding to fp32.                                                         */
/* ------------------------------------------------------------------------ */
void or_hadamard_rotate(const float *X, int64_t n, int d, const float *mean, const float *sigma,
                        int D, float *Y) {
    const double scale = 1.0 / sqrt((double)D);
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < n; ++p) {
        double *v = (double *)malloc(sizeof(double) * (size_t)D);
        for (int i = 0; i < D; ++i) {
            double x = 0.0;
            if (i < d) x = (double)X[p * (int64_t)d + i] - (mean ? (double)mean[i] : 0.0);
            v[i] = x * (double)sigma[i];
        }
        for (int h = 1; h < D; h <<= 1)
            for (int i = 0; i < D; i += 2 * h)
                for (int j = i; j < i + h; ++j) {
                    const double a = v[j], b = v[j + h];
                    v[j] = a + b;
                    v[j + h] = a - b;
                }
        for (int i = 0; i < D; ++i) Y[p * (int64_t)D + i] = (float)(v[i] * scale);
        free(v);
    }
}

/* Unprojection of projected centroids back to the original space (Section 4,
 * "Dimensionality Reduction and Vector Search", approach 2): x = y P^T + mu,
 * fp64, with P the d x dout projection matrix (row-major). */
void or_unproject(const float *Y, int64_t n, int dout, const float *P, const float *mu, int d, double *X) {
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < n; ++p) {
        const float *y = Y + p * (int64_t)dout;
        for (int i = 0; i < d; ++i) {
            double s = mu ? (double)mu[i] : 0.0;
            for (int j = 0; j < dout; ++j) s += (double)y[j] * (double)P[(int64_t)i * dout + j];
            X[p * (int64_t)d + i] = s;
        }
    }
}

/* ------------------------------------------------------------------------ */
/* Section 3.1 "LVQ4": locally-adaptive 4-bit codes with a per-vector bias   */
/* and scale, distances by Eq. final:lvq, fused decode-average update.       */
/* ------------------------------------------------------------------------ */

/* Per vector v (a point or, once per iteration, a centroid): b = min v_i,
 * s = (max v_i - b) / 15 in fp32 (s = 1 when the vector is flat, the same
 * reading as the flat SQ dimension), code_i = clip(round((v_i - b) / s), 0,
 * 15) in fp32, rounding half to even.  With S = sum code_i and
 * Q = sum code_i^2 (exact integers) the vector's constant terms of the
 * expanded distance are, in fp64 evaluated left to right and rounded once
 * to fp32,
 *   N = s*s*Q + 2*b*s*S + d*b*b     (the squared norm of the decoded vector)
 *   A = s*S + d*b                   (the sum of the decoded vector)
 *   G = s*S                         (s times the code sum)
 * fac[p] = (s, b, N, A); G is returned separately (it is the centroid-side
 * term s_y sum ybar).  Pinned: codes of data on the 15-step grid, the
 * reconstruction error bound s/2, flat vectors, N and A against the decoded
 * vector's fp64 norm and sum. */
void or_lvq4_encode(const float *V, int64_t n, int d, uint8_t *codes, float *fac, float *G) {
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < n; ++p) {
        const float *v = V + p * (int64_t)d;
        float lo = INFINITY, hi = -INFINITY;
        for (int i = 0; i < d; ++i) {
            if (v[i] < lo) lo = v[i];
            if (v[i] > hi) hi = v[i];
        }
        float s = (hi - lo) / 15.0f;
        if (!(s > 0.0f)) s = 1.0f;
        int64_t S = 0, Q = 0;
        for (int i = 0; i < d; ++i) {
            float q = rintf((v[i] - lo) / s);
            if (!(q >= 0.0f)) q = 0.0f;
            if (q > 15.0f) q = 15.0f;
            const int c = (int)q;
            codes[p * (int64_t)d + i] = (uint8_t)c;
            S += c;
            Q += (int64_t)c * c;
        }
        const double sd = (double)s, bd = (double)lo, dd = (double)d;
        const double N = sd * sd * (double)Q + 2.0 * bd * sd * (double)S + dd * bd * bd;
        const double A = sd * (double)S + dd * bd;
        fac[4 * p + 0] = s;
        fac[4 * p + 1] = lo;
        fac[4 * p + 2] = (float)N;
        fac[4 * p + 3] = (float)A;
        if (G) G[p] = (float)(sd * (double)S);
    }
}

/* Eq. final:lvq, fp32, in this fixed order (the paper fixes none):
 *   P   = sum_i xbar_i ybar_i                          (exact integer)
 *   key = fma(b_y, -2 A_x, N_y)
 *   key = fma(G_y, -2 b_x, key)                        G_y = s_y sum ybar
 *   key = fma(-2 s_x, s_y * P, key)                    (s_y * P one rounding)
 * The row's own N_x does not change which centroid is nearest: the argmin is
 * taken over key (ties to the lowest index) and the reported distance is
 * N_x + key of the winner (one fp32 addition).  xfac / yfac: (s, b, N, A)
 * per point / centroid, Gy per centroid. */
void or_lvq4_assign(const uint8_t *xc, const float *xfac, int64_t n, int d, const uint8_t *yc,
                    const float *yfac, const float *Gy, int k, int32_t *assign, float *dist) {
#pragma omp parallel for schedule(dynamic, 16)
    for (int64_t p = 0; p < n; ++p) {
        const uint8_t *x = xc + p * (int64_t)d;
        const float sx2 = -2.0f * xfac[4 * p + 0];
        const float bx2 = -2.0f * xfac[4 * p + 1];
        const float ax2 = -2.0f * xfac[4 * p + 3];
        float best = INFINITY;
        int32_t a = -1;
        for (int j = 0; j < k; ++j) {
            const uint8_t *y = yc + (int64_t)j * d;
            int64_t P = 0;
            for (int i = 0; i < d; ++i) P += (int64_t)x[i] * y[i];
            float key = fmaf(yfac[4 * j + 1], ax2, yfac[4 * j + 2]);
            key = fmaf(Gy[j], bx2, key);
            const float t = yfac[4 * j + 0] * (float)P;
            key = fmaf(sx2, t, key);
            if (key < best) {
                best = key;
                a = j;
            }
        }
        assign[p] = a;
        if (dist) dist[p] = xfac[4 * p + 2] + best;
    }
}

/* Fixed-point exponent of the decode-average: with M = max over points of
 * max(s, |b|), e = 31 - ceil(log2 M) (0 when M = 0), so that round(s 2^e) and
 * |round(b 2^e)| are at most 2^31. */
int or_lvq4_exponent(const float *fac, int64_t n) {
    float mx = 0.0f;
    for (int64_t p = 0; p < n; ++p) {
        const float s = fac[4 * p + 0], b = fabsf(fac[4 * p + 1]);
        if (s > mx) mx = s;
        if (b > mx) mx = b;
    }
    if (!(mx > 0.0f)) return 0;
    int ex;
    double fr = frexp((double)mx, &ex);
    int c = (fr == 0.5) ? ex - 1 : ex; /* ceil(log2 mx) */
    return 31 - c;
}

/* Fused decode-average (Section 3.1 "LVQ4", last paragraph): a member decodes
 * to s xbar_i + b and the members of a cluster are averaged.  s and b enter as
 * the integers Sq = round(s 2^e) and Bq = round(b 2^e), so the sums are exact
 * and independent of order:
 *   T_i = sum Sq xbar_i,  U = sum Bq
 *   c_i = (T_i + U) * f,  f = 2^-e / count    (int64 -> fp64, then fp32)
 * Empty clusters keep their centroid.  Pinned against the fp64 mean of the
 * decoded members (relative 1e-8) and exactly representable members. */
void or_lvq4_update(const uint8_t *xc, const float *xfac, int64_t n, int d, int e,
                    const int32_t *assign, int k, float *C_inout, int64_t *counts) {
    int64_t *T = (int64_t *)calloc((size_t)k * d, sizeof(int64_t));
    int64_t *U = (int64_t *)calloc((size_t)k, sizeof(int64_t));
    for (int j = 0; j < k; ++j) counts[j] = 0;
    for (int64_t p = 0; p < n; ++p) {
        const int32_t a = assign[p];
        const int64_t sq = (int64_t)llrint(ldexp((double)xfac[4 * p + 0], e));
        const int64_t bq = (int64_t)llrint(ldexp((double)xfac[4 * p + 1], e));
        counts[a] += 1;
        U[a] += bq;
        for (int i = 0; i < d; ++i) T[(int64_t)a * d + i] += sq * (int64_t)xc[p * (int64_t)d + i];
    }
    for (int j = 0; j < k; ++j) {
        if (counts[j] == 0) continue;
        const double f = ldexp(1.0, -e) / (double)counts[j];
        for (int i = 0; i < d; ++i) {
            const double v = (double)(T[(int64_t)j * d + i] + U[j]);
            C_inout[(int64_t)j * d + i] = (float)(v * f);
        }
    }
    free(T);
    free(U);
}

/* ------------------------------------------------------------------------ */
/* STEP 1 (Section 2.3): Forgy initialisation from a seed -- the first k     */
/* entries of a uniformly random permutation of 0..n-1.                      */
/*                                                                           */
/* Random bits: Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random  */
/* numbers: as easy as 1, 2, 3", SC'11): ten rounds on a 4 x 32-bit counter   */
/* under a 2 x 32-bit key; each round multiplies counter words 0 and 2 by     */
/* 0xD2511F53 and 0xCD9E8D57 (64-bit products split into high and low        */
/* halves) and forms (hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0); the key is     */
/* advanced by the Weyl constants (0x9E3779B9, 0xBB67AE85) between rounds.   */
/* Parity: pinned by the published known-answer vectors of Philox4x32-10.    */
/* ------------------------------------------------------------------------ */
void or_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2], uint32_t out[4]) {
    uint32_t c[4] = {ctr_in[0], ctr_in[1], ctr_in[2], ctr_in[3]};
    uint32_t k0 = key_in[0], k1 = key_in[1];
    for (int round = 0; round < 10; ++round) {
        if (round > 0) {
            k0 += 0x9E3779B9u;
            k1 += 0xBB67AE85u;
        }
        uint64_t p0 = (uint64_t)0xD2511F53u * (uint64_t)c[0];
        uint64_t p1 = (uint64_t)0xCD9E8D57u * (uint64_t)c[2];
        uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        uint32_t n0 = hi1 ^ c[1] ^ k0;
        uint32_t n2 = hi0 ^ c[3] ^ k1;
        c[0] = n0;
        c[1] = lo1;
        c[2] = n2;
        c[3] = lo0;
    }
    out[0] = c[0];
    out[1] = c[1];
    out[2] = c[2];
    out[3] = c[3];
}

/* Fisher-Yates on the identity sequence a = (0, 1, ..., n-1), positions      */
/* i = 0 .. k-1 only: draw i is Philox4x32-10 of counter (i mod 2^32,        */
/* i div 2^32, 0x466F7267, 0) under key (seed mod 2^32, seed div 2^32);      */
/* r = w0 2^32 + w1; j = i + floor(r (n - i) / 2^64); swap a[i] and a[j].     */
/* out[0..k) = a[0..k).  Parity: pinned by the permutation properties (every */
/* index once, k = n a full permutation, uniform first entry).               */
void or_forgy_indices(uint64_t seed, int64_t n, int k, int64_t *out) {
    int64_t *a = (int64_t *)malloc(sizeof(int64_t) * (size_t)n);
    for (int64_t i = 0; i < n; ++i) a[i] = i;
    const uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    for (int64_t i = 0; i < k; ++i) {
        const uint32_t ctr[4] = {(uint32_t)i, (uint32_t)((uint64_t)i >> 32), 0x466F7267u, 0u};
        uint32_t w[4];
        or_philox4x32_10(ctr, key, w);
        const uint64_t r = ((uint64_t)w[0] << 32) | (uint64_t)w[1];
        const uint64_t span = (uint64_t)(n - i);
        const uint64_t off = (uint64_t)(((unsigned __int128)r * span) >> 64);
        const int64_t j = i + (int64_t)off;
        const int64_t t = a[i];
        a[i] = a[j];
        a[j] = t;
        out[i] = a[i];
    }
    free(a);
}

/* ------------------------------------------------------------------------ */
/* SuperKMeans with RabitQ codes (Section 3.1 "SuperKMeans": for RabitQ the  */
/* L2 distance decomposes over dimension segments, ||x - y||^2 = sum over    */
/* segments of ||x_t - y_t||^2, each segment estimated with its own          */
/* factors; pruning checkpoints after 12.5% and 25% of d).                   */
/* Segments: [0, d1), [d1, d2), [d2, d) with d1 = 32 max(1, floor((d + 128)  */
/* / 256)) (d/8 rounded to whole 32-dimension words) and d2 = 2 d1.          */
/* Per point and segment t, with r = x - m (the global mean): nx2_t =        */
/* ||r_t||^2, F_t = sqrt(d_t) ||r_t||^2 / ||r_t||_1 (0 when r_t = 0), both   */
/* fp64 left to right rounded once; popx_t = set bits of the segment.        */
/* Parity: the segment factors against their definitions; with the whole of  */
/* d as one segment the estimate is the plain RabitQ one; on data lying on   */
/* both grids the segment estimates are the exact segment distances.         */
/* ------------------------------------------------------------------------ */
void or_rbq1_seg_bounds(int d, int *d1, int *d2) {
    int w = (d + 128) / 256;
    if (w < 1) w = 1;
    *d1 = 32 * w;
    *d2 = 2 * (*d1);
}

void or_rbq1_seg_encode(const float *X, int64_t n, int d, const float *m, int d1, int d2, float *nx2s,
                        float *Fs, int32_t *popxs) {
    const int lo[3] = {0, d1, d2}, hi[3] = {d1, d2, d};
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < n; ++p) {
        for (int t = 0; t < 3; ++t) {
            double s2 = 0.0, s1 = 0.0;
            int32_t pc = 0;
            for (int i = lo[t]; i < hi[t]; ++i) {
                float r = X[p * (int64_t)d + i] - m[i];
                if (r > 0.0f) pc += 1;
                s2 += (double)r * (double)r;
                s1 += fabs((double)r);
            }
            nx2s[p * 3 + t] = (float)s2;
            Fs[p * 3 + t] = (s1 > 0.0) ? (float)(sqrt((double)(hi[t] - lo[t])) * s2 / s1) : 0.0f;
            popxs[p * 3 + t] = pc;
        }
    }
}

/* Per centroid: the SQ4 codes of or_rbq1_centroid_sq4 (over all d), and per  */
/* segment the code sum and ||rho_t||^2 (the blocked fp64 order of           */
/* sumsq_blocked over the segment's words).                                   */
void or_rbq1_seg_centroid(const float *C, int k, int d, const float *m, int d1, int d2, uint8_t *ybar,
                          float *b, float *s, int32_t *sumy3, float *ny2s) {
    int32_t *sumy = (int32_t *)malloc(sizeof(int32_t) * (size_t)k);
    float *ny2 = (float *)malloc(sizeof(float) * (size_t)k);
    or_rbq1_centroid_sq4(C, k, d, m, ybar, b, s, sumy, ny2);
    float *rho = (float *)malloc(sizeof(float) * (size_t)d);
    const int lo[3] = {0, d1, d2}, hi[3] = {d1, d2, d};
    for (int j = 0; j < k; ++j) {
        for (int i = 0; i < d; ++i) rho[i] = C[(int64_t)j * d + i] - m[i];
        for (int t = 0; t < 3; ++t) {
            int32_t sy = 0;
            for (int i = lo[t]; i < hi[t]; ++i) sy += ybar[(int64_t)j * d + i];
            sumy3[(int64_t)j * 3 + t] = sy;
            ny2s[(int64_t)j * 3 + t] = (float)sumsq_blocked(rho + lo[t], hi[t] - lo[t]);
        }
    }
    free(rho);
    free(sumy);
    free(ny2);
}

/* Segment estimate of Eq. rabitq_l2 with Eq. final:rabitq on the segment, in  */
/* the library's fp32 order: isd_t = fl(1/sqrt(d_t)), sd = s isd_t, bd = b    */
/* isd_t, u = fma(sd, 2 P_t - sumy_t, bd (2 popx_t - d_t)), est = fma(-2 F_t,  */
/* u, nx2_t + ny2_t).  Partial estimates D1 = est_0, D2 = D1 + est_1,         */
/* D3 = D2 + est_2 (fp32).                                                    */
/* Pruning (an order-independent reading of the checkpoints): the bound is    */
/* beta = D3 of the row's seed centroid (its previous assignment, entries     */
/* outside [0, k) and prev = NULL meaning centroid 0); at checkpoint t (after */
/* e_t = d1, d2 dimensions) a centroid other than the seed is dropped when    */
/* D_t > fl32(beta g_t), g_t the checkpoint's factor: ADSampling's test       */
/* D_t d / e_t > beta (1 + eps0 / sqrt(e_t))^2 gives g_t = fl32((e_t / d)     */
/* (1 + eps0 / sqrt(e_t))^2) (or_rbq1_seg_factors, eps0 = 2.1), g_t = 1 the   */
/* exact test; the result is the candidate (seed included) with the smallest  */
/* D3, ties to the lowest index.  est_best receives that D3.                  */
void or_rbq1_seg_factors(int d, int d1, int d2, double eps0, float *g) {
    const int e[2] = {d1, d2};
    for (int t = 0; t < 2; ++t) {
        const double a = 1.0 + eps0 / sqrt((double)e[t]);
        g[t] = (float)(((double)e[t] / (double)d) * a * a);
    }
}

/* The partial estimates D1, D2, D3 of point p against centroid j. */
static void seg_partials(const uint32_t *cw, const float *nx2s, const float *Fs, const int32_t *popxs, int64_t p,
                         int d, const int lo[3], const int hi[3], const float isd[3], const uint8_t *y, float b,
                         float s, const int32_t *sumy3, const float *ny2s, float D[3]) {
    for (int t = 0; t < 3; ++t) {
        if (hi[t] == lo[t]) { /* an empty segment adds nothing */
            D[t] = (t == 0) ? 0.0f : D[t - 1];
            continue;
        }
        int32_t P = 0;
        for (int i = lo[t]; i < hi[t]; ++i)
            if ((cw[i / 32] >> (i % 32)) & 1u) P += y[i];
        const float sd = s * isd[t];
        const float bd = b * isd[t];
        const float pc = (float)(2 * popxs[p * 3 + t] - (hi[t] - lo[t]));
        const float u = fmaf(sd, (float)(2 * P - sumy3[t]), bd * pc);
        const float est = fmaf(-2.0f * Fs[p * 3 + t], u, nx2s[p * 3 + t] + ny2s[t]);
        D[t] = (t == 0) ? est : D[t - 1] + est;
    }
}

void or_rbq1_seg_assign(const uint32_t *codes, const float *nx2s, const float *Fs, const int32_t *popxs,
                        int64_t n, int d, int d1, int d2, const uint8_t *ybar, const float *b, const float *s,
                        const int32_t *sumy3, const float *ny2s, int k, const int32_t *prev, const float *g,
                        int32_t *assign, float *est_best) {
    const int W = (d + 31) / 32;
    const int lo[3] = {0, d1, d2}, hi[3] = {d1, d2, d};
    float isd[3];
    for (int t = 0; t < 3; ++t) isd[t] = hi[t] > lo[t] ? (float)(1.0 / sqrt((double)(hi[t] - lo[t]))) : 0.0f;
#pragma omp parallel for schedule(dynamic, 16)
    for (int64_t p = 0; p < n; ++p) {
        const uint32_t *cw = codes + p * (int64_t)W;
        int seed = prev ? prev[p] : 0;
        if (seed < 0 || seed >= k) seed = 0;
        float D[3];
        seg_partials(cw, nx2s, Fs, popxs, p, d, lo, hi, isd, ybar + (int64_t)seed * d, b[seed], s[seed],
                     sumy3 + (int64_t)seed * 3, ny2s + (int64_t)seed * 3, D);
        const float beta = D[2];
        float best = INFINITY;
        int32_t a = -1;
        for (int j = 0; j < k; ++j) {
            seg_partials(cw, nx2s, Fs, popxs, p, d, lo, hi, isd, ybar + (int64_t)j * d, b[j], s[j],
                         sumy3 + (int64_t)j * 3, ny2s + (int64_t)j * 3, D);
            if (j != seed && (D[0] > beta * g[0] || D[1] > beta * g[1])) continue;
            if (D[2] < best) {
                best = D[2];
                a = j;
            }
        }
        assign[p] = a;
        if (est_best) est_best[p] = best;
    }
}

/* Every pair's partial estimates D[p][j][0..2] (no pruning). */
void or_rbq1_seg_partials(const uint32_t *codes, const float *nx2s, const float *Fs, const int32_t *popxs,
                          int64_t n, int d, int d1, int d2, const uint8_t *ybar, const float *b, const float *s,
                          const int32_t *sumy3, const float *ny2s, int k, float *D) {
    const int W = (d + 31) / 32;
    const int lo[3] = {0, d1, d2}, hi[3] = {d1, d2, d};
    float isd[3];
    for (int t = 0; t < 3; ++t) isd[t] = hi[t] > lo[t] ? (float)(1.0 / sqrt((double)(hi[t] - lo[t]))) : 0.0f;
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < n; ++p)
        for (int j = 0; j < k; ++j)
            seg_partials(codes + p * (int64_t)W, nx2s, Fs, popxs, p, d, lo, hi, isd, ybar + (int64_t)j * d, b[j],
                         s[j], sumy3 + (int64_t)j * 3, ny2s + (int64_t)j * 3, D + (p * (int64_t)k + j) * 3);
}
