// ace_offline.cpp — offline GSP / RCR tables (Algorithms 2 and 3), host CPU.
// Declared in ace_offline.h; no CUDA.
#include "ace_offline.h"

#include <stdint.h>
#include <string.h>

#include <atomic>
#include <cmath>
#include <thread>
#include <vector>

namespace {

double to_f64(const void* base, ace_dtype dt, size_t i) {
    if (dt == ACE_F32) return (double)static_cast<const float*>(base)[i];
    uint32_t u = (uint32_t)static_cast<const uint16_t*>(base)[i] << 16;
    float f;
    memcpy(&f, &u, 4);
    return (double)f;
}

// Row-major [rows, cols] block of the weight array starting at element `off`,
// as fp64, transposed to column-major ([cols][rows]) when `kmajor`.
void load_block(const void* base, ace_dtype dt, size_t off, int rows, int cols, bool kmajor, std::vector<double>& out) {
    out.resize((size_t)rows * cols);
    for (int r = 0; r < rows; ++r)
        for (int c = 0; c < cols; ++c) {
            const double v = to_f64(base, dt, off + (size_t)r * cols + c);
            out[kmajor ? (size_t)c * rows + r : (size_t)r * cols + c] = v;
        }
}

// C = A^T A for A stored k-major ([kdim][n], element (k, i) at a[k*n + i]),
// i.e. C[i][j] = sum_k a[k][i] a[k][j], both triangles filled. K is taken in
// chunks of 128 rows that stay in cache, 4 x 4 register tiles within a chunk;
// every entry is summed over k in increasing order (partial sums parked in C
// between chunks), so the result is that of one sequential sum.
void gram(const std::vector<double>& a, int kdim, int n, std::vector<double>& c) {
    constexpr int KC = 128;
    c.assign((size_t)n * n, 0.0);
    for (int k0 = 0; k0 < kdim; k0 += KC) {
        const int k1 = k0 + KC < kdim ? k0 + KC : kdim;
        for (int i0 = 0; i0 < n; i0 += 4) {
            for (int j0 = 0; j0 <= i0; j0 += 4) {
                const int ni = n - i0 < 4 ? n - i0 : 4, nj = n - j0 < 4 ? n - j0 : 4;
                double acc[4][4];
                for (int ii = 0; ii < 4; ++ii)
                    for (int jj = 0; jj < 4; ++jj)
                        acc[ii][jj] = (ii < ni && jj < nj) ? c[(size_t)(i0 + ii) * n + (j0 + jj)] : 0.0;
                if (ni == 4 && nj == 4) {
                    for (int k = k0; k < k1; ++k) {
                        const double* ak = &a[(size_t)k * n];
                        const double x0 = ak[i0], x1 = ak[i0 + 1], x2 = ak[i0 + 2], x3 = ak[i0 + 3];
                        const double y0 = ak[j0], y1 = ak[j0 + 1], y2 = ak[j0 + 2], y3 = ak[j0 + 3];
                        acc[0][0] += x0 * y0; acc[0][1] += x0 * y1; acc[0][2] += x0 * y2; acc[0][3] += x0 * y3;
                        acc[1][0] += x1 * y0; acc[1][1] += x1 * y1; acc[1][2] += x1 * y2; acc[1][3] += x1 * y3;
                        acc[2][0] += x2 * y0; acc[2][1] += x2 * y1; acc[2][2] += x2 * y2; acc[2][3] += x2 * y3;
                        acc[3][0] += x3 * y0; acc[3][1] += x3 * y1; acc[3][2] += x3 * y2; acc[3][3] += x3 * y3;
                    }
                } else {
                    for (int k = k0; k < k1; ++k) {
                        const double* ak = &a[(size_t)k * n];
                        for (int ii = 0; ii < ni; ++ii)
                            for (int jj = 0; jj < nj; ++jj) acc[ii][jj] += ak[i0 + ii] * ak[j0 + jj];
                    }
                }
                for (int ii = 0; ii < ni; ++ii)
                    for (int jj = 0; jj < nj; ++jj) c[(size_t)(i0 + ii) * n + (j0 + jj)] = acc[ii][jj];
            }
        }
    }
    for (int i = 0; i < n; ++i)                  // the upper triangle from the lower
        for (int j = i + 1; j < n; ++j) c[(size_t)i * n + j] = c[(size_t)j * n + i];
}

double frob_dot(const std::vector<double>& x, const std::vector<double>& y) {
    double s = 0.0;
    for (size_t i = 0; i < x.size(); ++i) s += x[i] * y[i];
    return s;
}

struct Job {
    int d, N, m;
    ace_dtype dt;
    const void *gamma, *wg, *wu, *wd;
    const std::vector<double>* protos;   // [N][d] RCR prototypes (after the optional gamma)
    const std::vector<double>* qnorm;    // [N] ||q_e||
    double eps;
    std::vector<double>* gsp_raw;
    std::vector<double>* rcr_raw;
};

// Raw GSP and RCR amplifications of expert e.
void expert(const Job& J, int e) {
    const int d = J.d, m = J.m;
    std::vector<double> gam(d);
    for (int i = 0; i < d; ++i) gam[i] = to_f64(J.gamma, J.dt, i);
    // G = Gamma W_gate^T as k-major [d][m]: element (k = input i, col j) = gamma_i w_gate[j][i]
    std::vector<double> a, gg, gu, gd;
    load_block(J.wg, J.dt, (size_t)e * m * d, m, d, true, a);          // [d][m]
    for (int k = 0; k < d; ++k)
        for (int j = 0; j < m; ++j) a[(size_t)k * m + j] *= gam[k];
    gram(a, d, m, gg);                                                   // G^T G   [m][m]
    load_block(J.wu, J.dt, (size_t)e * m * d, m, d, true, a);
    for (int k = 0; k < d; ++k)
        for (int j = 0; j < m; ++j) a[(size_t)k * m + j] *= gam[k];
    gram(a, d, m, gu);                                                   // U^T U
    // W_down (paper's m x d) = w_down[e]^T; W W^T = w_down[e]^T w_down[e]: rows of
    // w_down[e] ([d][m]) are already k-major for this Gram
    load_block(J.wd, J.dt, (size_t)e * d * m, d, m, false, a);          // [d][m]
    gram(a, d, m, gd);
    double fro_g2 = 0.0, fro_u2 = 0.0;
    for (int j = 0; j < m; ++j) {
        fro_g2 += gg[(size_t)j * m + j];
        fro_u2 += gu[(size_t)j * m + j];
    }
    const double fro_gd2 = std::fmax(frob_dot(gg, gd), 0.0);
    const double fro_ud2 = std::fmax(frob_dot(gu, gd), 0.0);
    const double a_up2 = fro_u2 * fro_gd2, a_gate2 = fro_g2 * fro_ud2;
    (*J.gsp_raw)[e] = std::pow(a_up2 * a_gate2, 0.25);                 // sqrt(a_up a_gate)

    // RCR: y = W_down (SiLU(W_gate q) * (W_up q))
    const double* q = &(*J.protos)[(size_t)e * d];
    std::vector<double> act(m);
    for (int j = 0; j < m; ++j) {
        double u = 0.0, v = 0.0;
        for (int i = 0; i < d; ++i) {
            u += to_f64(J.wg, J.dt, ((size_t)e * m + j) * d + i) * q[i];
            v += to_f64(J.wu, J.dt, ((size_t)e * m + j) * d + i) * q[i];
        }
        act[j] = u / (1.0 + std::exp(-u)) * v;
    }
    double yy = 0.0;
    for (int i = 0; i < d; ++i) {
        double y = 0.0;
        for (int j = 0; j < m; ++j) y += to_f64(J.wd, J.dt, ((size_t)e * d + i) * m + j) * act[j];
        yy += y * y;
    }
    (*J.rcr_raw)[e] = std::sqrt(yy) / ((*J.qnorm)[e] + J.eps);
}

}  // namespace

extern "C" ace_status ace_offline_tables(int d, int N, int m, ace_dtype dtype, const void* gamma, const void* router_w,
                                         const void* w_gate, const void* w_up, const void* w_down, double eps,
                                         int rcr_apply_gamma, int n_threads, float* gsp_out, float* rcr_out) {
    if (d <= 0 || N <= 0 || m <= 0) return ACE_ERR_INVALID_ARG;
    if (dtype != ACE_BF16 && dtype != ACE_F32) return ACE_ERR_INVALID_ARG;
    if (!gamma || !router_w || !w_gate || !w_up || !w_down || !gsp_out || !rcr_out) return ACE_ERR_INVALID_ARG;
    // RCR prototypes: centred router rows scaled to unit RMS (rho = 1)
    std::vector<double> mean(d, 0.0), protos((size_t)N * d), qnorm(N);
    for (int e = 0; e < N; ++e)
        for (int i = 0; i < d; ++i) mean[i] += to_f64(router_w, dtype, (size_t)e * d + i);
    for (int i = 0; i < d; ++i) mean[i] /= N;
    for (int e = 0; e < N; ++e) {
        double ss = 0.0;
        for (int i = 0; i < d; ++i) {
            const double w = to_f64(router_w, dtype, (size_t)e * d + i) - mean[i];
            protos[(size_t)e * d + i] = w;
            ss += w * w;
        }
        const double rms = std::sqrt(ss / d);
        double qq = 0.0;
        for (int i = 0; i < d; ++i) {
            double& q = protos[(size_t)e * d + i];
            q /= rms + eps;
            qq += q * q;
        }
        qnorm[e] = std::sqrt(qq);
        if (rcr_apply_gamma)
            for (int i = 0; i < d; ++i) protos[(size_t)e * d + i] *= to_f64(gamma, dtype, i);
    }
    std::vector<double> gsp_raw(N), rcr_raw(N);
    Job J{d, N, m, dtype, gamma, w_gate, w_up, w_down, &protos, &qnorm, eps, &gsp_raw, &rcr_raw};
    int nt = n_threads > 0 ? n_threads : (int)std::thread::hardware_concurrency();
    if (nt < 1) nt = 1;
    if (nt > N) nt = N;
    std::atomic<int> next(0);
    std::vector<std::thread> pool;
    for (int t = 0; t < nt; ++t)
        pool.emplace_back([&]() {
            for (int e = next++; e < N; e = next++) expert(J, e);
        });
    for (auto& th : pool) th.join();
    double sg = 0.0, sr = 0.0;
    for (int e = 0; e < N; ++e) {
        sg += gsp_raw[e];
        sr += rcr_raw[e];
    }
    const double mg = sg / N, mr = sr / N;
    for (int e = 0; e < N; ++e) {
        gsp_out[e] = (float)(gsp_raw[e] / (mg + eps));
        rcr_out[e] = (float)(rcr_raw[e] / (mr + eps));
    }
    return ACE_OK;
}
