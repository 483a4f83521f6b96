// Host-side dense linear algebra for the projection step (Section 3.1:
// random orthogonal rotation for RabitQ/SuperKMeans; PCA):
//  - Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) + Box-Muller Gaussians
//  - explicit Q of a Householder QR (Golub & Van Loan, Sec. 5.2), signs fixed
//    so that R has a positive diagonal (a Haar-distributed rotation)
//  - symmetric eigen-decomposition: Householder reduction to tridiagonal
//    form, then implicit QL iterations with a Wilkinson-type shift
//    (Golub & Van Loan, Sec. 8.3; Bowdler-Martin-Reinsch-Wilkinson QL),
//    accumulating the orthogonal factors.  All fp64.
#include <math.h>
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <unordered_map>
#include <vector>

namespace skm {

// ------------------------------------------------------------- Philox4x32-10
static void philox4x32_10(uint32_t ctr[4], uint32_t key0, uint32_t key1) {
    for (int r = 0; r < 10; ++r) {
        const uint64_t p0 = (uint64_t)0xD2511F53u * ctr[0];
        const uint64_t p1 = (uint64_t)0xCD9E8D57u * ctr[2];
        const uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        const uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        const uint32_t n0 = hi1 ^ ctr[1] ^ key0;
        const uint32_t n2 = hi0 ^ ctr[3] ^ key1;
        ctr[0] = n0;
        ctr[1] = lo1;
        ctr[2] = n2;
        ctr[3] = lo0;
        key0 += 0x9E3779B9u;
        key1 += 0xBB67AE85u;
    }
}

// uniform in (0, 1]: 53 random bits
static inline double unit53(uint32_t hi, uint32_t lo) {
    const uint64_t a = (((uint64_t)hi << 32) | lo) >> 11;
    return ((double)a + 1.0) * (1.0 / 9007199254740992.0);
}

void philox_gaussians(uint64_t seed, int64_t count, double *out) {
    const uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
    const double two_pi = 6.283185307179586476925286766559;
    for (int64_t blk = 0; 2 * blk < count; ++blk) {
        uint32_t c[4] = {(uint32_t)blk, (uint32_t)((uint64_t)blk >> 32), 0u, 0u};
        philox4x32_10(c, k0, k1);
        const double u1 = unit53(c[0], c[1]), u2 = unit53(c[2], c[3]);
        const double rad = sqrt(-2.0 * log(u1));
        out[2 * blk] = rad * cos(two_pi * u2);
        if (2 * blk + 1 < count) out[2 * blk + 1] = rad * sin(two_pi * u2);
    }
}

// Forgy (Section 2.3 STEP 1) from a seed: positions 0..k-1 of a Fisher-Yates
// shuffle of (0, 1, ..., n-1); draw i = Philox4x32-10 of counter (i lo, i hi,
// 0x466F7267, 0) under key (seed lo, seed hi), r = w0 2^32 + w1, and position
// i swaps with i + floor(r (n - i) / 2^64).  Only the displaced positions are
// stored (a hash map), so the work and memory are O(k) whatever n is.
void forgy_indices(uint64_t seed, int64_t n, int k, int64_t *out) {
    const uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
    std::unordered_map<int64_t, int64_t> moved;
    moved.reserve((size_t)k * 2 + 16);
    auto at = [&](int64_t p) {
        auto it = moved.find(p);
        return it == moved.end() ? p : it->second;
    };
    for (int64_t i = 0; i < k; ++i) {
        uint32_t c[4] = {(uint32_t)i, (uint32_t)((uint64_t)i >> 32), 0x466F7267u, 0u};
        philox4x32_10(c, k0, k1);
        const uint64_t r = ((uint64_t)c[0] << 32) | c[1];
        const int64_t j = i + (int64_t)(((unsigned __int128)r * (uint64_t)(n - i)) >> 64);
        const int64_t vi = at(i), vj = at(j);
        moved[j] = vi;
        moved[i] = vj;
        out[i] = vj;
    }
}

// ------------------------------------------------ Householder QR, explicit Q
// A (d x d, row-major) is overwritten by Q with R's diagonal made positive.
void householder_qr_q(int d, double *A) {
    std::vector<double> V((size_t)d * d, 0.0);  // Householder vectors, column j in V[j*d..]
    std::vector<double> beta(d, 0.0), rdiag(d, 0.0);
    std::vector<double> col(d);
    for (int j = 0; j < d; ++j) {
        double nrm2 = 0.0;
        for (int i = j; i < d; ++i) nrm2 += A[(size_t)i * d + j] * A[(size_t)i * d + j];
        const double nrm = sqrt(nrm2);
        const double x0 = A[(size_t)j * d + j];
        double *v = &V[(size_t)j * d];
        if (nrm == 0.0) {
            beta[j] = 0.0;
            rdiag[j] = 0.0;
            continue;
        }
        const double alpha = (x0 >= 0.0) ? -nrm : nrm;  // R_jj = alpha
        v[j] = x0 - alpha;
        for (int i = j + 1; i < d; ++i) v[i] = A[(size_t)i * d + j];
        double vv = 0.0;
        for (int i = j; i < d; ++i) vv += v[i] * v[i];
        beta[j] = (vv > 0.0) ? 2.0 / vv : 0.0;
        rdiag[j] = alpha;
        // apply H_j = I - beta v v^T to A[j:, j:]
        for (int c = j; c < d; ++c) {
            double s = 0.0;
            for (int i = j; i < d; ++i) s += v[i] * A[(size_t)i * d + c];
            s *= beta[j];
            for (int i = j; i < d; ++i) A[(size_t)i * d + c] -= s * v[i];
        }
    }
    // Q = H_0 H_1 ... H_{d-1}: backward accumulation on the identity
    std::vector<double> Q((size_t)d * d, 0.0);
    for (int i = 0; i < d; ++i) Q[(size_t)i * d + i] = 1.0;
    for (int j = d - 1; j >= 0; --j) {
        if (beta[j] == 0.0) continue;
        const double *v = &V[(size_t)j * d];
        for (int c = j; c < d; ++c) {
            double s = 0.0;
            for (int i = j; i < d; ++i) s += v[i] * Q[(size_t)i * d + c];
            s *= beta[j];
            for (int i = j; i < d; ++i) Q[(size_t)i * d + c] -= s * v[i];
        }
    }
    // positive diagonal of R: flip column j of Q where R_jj < 0
    for (int j = 0; j < d; ++j)
        if (rdiag[j] < 0.0)
            for (int i = 0; i < d; ++i) Q[(size_t)i * d + j] = -Q[(size_t)i * d + j];
    memcpy(A, Q.data(), sizeof(double) * (size_t)d * d);
}

// ------------------------------------------------ symmetric eigen-decomposition
// In: A (n x n, row-major, symmetric).  Out: A's columns = eigenvectors,
// w = eigenvalues (unsorted).  Returns 0, or -1 if QL did not converge.
int symmetric_eigen(int n, double *A, double *w) {
    // Zt holds the accumulated orthogonal factor TRANSPOSED (row i = basis
    // vector i) so that every plane rotation touches two contiguous rows.
    std::vector<double> Zt((size_t)n * n, 0.0);
    std::vector<double> dg(n), e(n, 0.0);
    std::vector<double> a(A, A + (size_t)n * n);
    // Householder tridiagonalisation: for k, annihilate a[k+2:, k].
    std::vector<std::vector<double>> vs;
    std::vector<double> betas;
    std::vector<double> v(n), p(n), q(n);
    for (int k = 0; k + 2 < n; ++k) {
        double nrm2 = 0.0;
        for (int i = k + 1; i < n; ++i) nrm2 += a[(size_t)i * n + k] * a[(size_t)i * n + k];
        const double nrm = sqrt(nrm2);
        const double x0 = a[(size_t)(k + 1) * n + k];
        if (nrm == 0.0) {
            vs.emplace_back();
            betas.push_back(0.0);
            continue;
        }
        const double alpha = (x0 >= 0.0) ? -nrm : nrm;
        for (int i = 0; i < n; ++i) v[i] = 0.0;
        v[k + 1] = x0 - alpha;
        for (int i = k + 2; i < n; ++i) v[i] = a[(size_t)i * n + k];
        double vv = 0.0;
        for (int i = k + 1; i < n; ++i) vv += v[i] * v[i];
        const double beta = (vv > 0.0) ? 2.0 / vv : 0.0;
        // p = beta * A' v over the trailing block; q = p - (beta/2)(p.v) v;
        // A' <- A' - v q^T - q v^T
        for (int i = k + 1; i < n; ++i) {
            double s = 0.0;
            const double *row = &a[(size_t)i * n];
            for (int j = k + 1; j < n; ++j) s += row[j] * v[j];
            p[i] = beta * s;
        }
        double pv = 0.0;
        for (int i = k + 1; i < n; ++i) pv += p[i] * v[i];
        for (int i = k + 1; i < n; ++i) q[i] = p[i] - 0.5 * beta * pv * v[i];
        for (int i = k + 1; i < n; ++i) {
            double *row = &a[(size_t)i * n];
            for (int j = k + 1; j < n; ++j) row[j] -= v[i] * q[j] + q[i] * v[j];
        }
        a[(size_t)(k + 1) * n + k] = alpha;
        a[(size_t)k * n + k + 1] = alpha;
        for (int i = k + 2; i < n; ++i) {
            a[(size_t)i * n + k] = 0.0;
            a[(size_t)k * n + i] = 0.0;
        }
        vs.emplace_back(v.begin(), v.end());
        betas.push_back(beta);
    }
    for (int i = 0; i < n; ++i) dg[i] = a[(size_t)i * n + i];
    for (int i = 0; i + 1 < n; ++i) e[i] = a[(size_t)(i + 1) * n + i];
    e[n - 1] = 0.0;
    // Q = H_0 ... H_{n-3}; Zt = Q^T built by backward accumulation:
    // Q <- H_k Q for k descending, i.e. Zt <- Zt H_k.
    for (int i = 0; i < n; ++i) Zt[(size_t)i * n + i] = 1.0;
    for (int k = (int)betas.size() - 1; k >= 0; --k) {
        if (betas[k] == 0.0) continue;
        const std::vector<double> &vk = vs[k];
        for (int r = 0; r < n; ++r) {  // rows of Zt = columns of Q
            double *row = &Zt[(size_t)r * n];
            double s = 0.0;
            for (int i = k + 1; i < n; ++i) s += row[i] * vk[i];
            s *= betas[k];
            if (s != 0.0)
                for (int i = k + 1; i < n; ++i) row[i] -= s * vk[i];
        }
    }
    // Zt currently holds Q^T?  Zt started as I and was multiplied on the right
    // by H_{n-3} ... H_0 in that order, so Zt = H_{n-3} ... H_0 = Q^T.
    const double eps = 2.220446049250313e-16;
    for (int l = 0; l < n; ++l) {
        int iter = 0;
        for (;;) {
            int m = l;
            for (; m + 1 < n; ++m) {
                const double dd = fabs(dg[m]) + fabs(dg[m + 1]);
                if (fabs(e[m]) <= eps * dd) break;
            }
            if (m == l) break;
            if (++iter > 200) return -1;
            // shift: eigenvalue of the leading 2x2 block closer to dg[l]
            double g = (dg[l + 1] - dg[l]) / (2.0 * e[l]);
            double r = hypot(g, 1.0);
            g = dg[m] - dg[l] + e[l] / (g + (g >= 0.0 ? fabs(r) : -fabs(r)));
            double s = 1.0, c = 1.0, pp = 0.0;
            bool restarted = false;
            for (int i = m - 1; i >= l; --i) {
                const double f = s * e[i], b = c * e[i];
                r = hypot(f, g);
                e[i + 1] = r;
                if (r == 0.0) {
                    dg[i + 1] -= pp;
                    e[m] = 0.0;
                    restarted = true;
                    break;
                }
                s = f / r;
                c = g / r;
                g = dg[i + 1] - pp;
                r = (dg[i] - g) * s + 2.0 * c * b;
                pp = s * r;
                dg[i + 1] = g + pp;
                g = c * r - b;
                double *zi = &Zt[(size_t)i * n];
                double *zj = &Zt[(size_t)(i + 1) * n];
                for (int t = 0; t < n; ++t) {
                    const double ft = zj[t];
                    zj[t] = s * zi[t] + c * ft;
                    zi[t] = c * zi[t] - s * ft;
                }
            }
            if (restarted) continue;
            dg[l] -= pp;
            e[l] = g;
            e[m] = 0.0;
        }
    }
    for (int i = 0; i < n; ++i) {
        w[i] = dg[i];
        for (int t = 0; t < n; ++t) A[(size_t)t * n + i] = Zt[(size_t)i * n + t];
    }
    return 0;
}

}  // namespace skm
