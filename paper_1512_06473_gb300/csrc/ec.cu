// ec.cu -- error-corrected quantization of an FC layer (Sec. 3.3.1, Eq. 8-12).
//
// Minimises sum_n ||T_n - sum_m (D^(m) B^(m))^T S_n^(m)||^2 over calibration
// vectors (S_n, T_n) by block coordinate descent over the sub-spaces, in
// order.  The device keeps E = T - (current approximation), [N][Ct] in
// double.  For sub-space m, with A = S^(m) ([N][C'_s]) and the residual
// R = E + A old^T of Eq. 9 held fixed:
//   stats : G = A^T A and V = A^T E (partial sums over fixed row chunks,
//           added in chunk order);
//   u     : U[:, c_t] = V[:, c_t] + G D_old[k_old(c_t)]  (= A^T R), the
//           Cholesky factor of G (rank-deficient data sets a flag), and
//           copies of the old codewords and codes;
//   then `inner` times
//     order : outputs grouped by code (stable counting sort);
//     D     : Eq. 11, G D_k = mean_{c_t in L_k} U[:, c_t] (sum in c_t order),
//             solved with the Cholesky factor; an unused codeword keeps its
//             value; q_k = D_k^T G D_k;
//     B     : Eq. 12, k(c_t) = argmin_k q_k - 2 D_k^T U[:, c_t], ties to the
//             smallest k;
//   E     : E += A (D_old[k_old] - D_new[k_new])^T.
// Everything is double: this is the offline quantizer, run once per layer.
#include "qcnn_internal.cuh"

#include <algorithm>
#include <climits>

namespace qcnn {

constexpr int kEcChunk = 64;  // rows of S per partial sum

// E = T - sum_m S^(m) D[m][codes[m]]^T, one thread per (n, c_t).
__global__ void ec_init_kernel(const float *__restrict__ S, const float *__restrict__ T, int N,
                               int Cs, int Ct, int Csp, int K, const double *__restrict__ Dw,
                               const uint8_t *__restrict__ codes, double *__restrict__ E) {
    const int M = Cs / Csp;
    const long long total = (long long)N * Ct;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int ct = (int)(i % Ct);
        const long long n = i / Ct;
        double y = 0.0;
        for (int m = 0; m < M; ++m) {
            const double *d = Dw + ((size_t)m * K + codes[(size_t)m * Ct + ct]) * Csp;
            const float *s = S + n * Cs + (size_t)m * Csp;
            for (int j = 0; j < Csp; ++j) y = fma((double)s[j], d[j], y);
        }
        E[i] = (double)T[i] - y;
    }
}

// Vp[chunk][j][c_t] = sum_{n in chunk} A[n][j] E[n][c_t]; the blocks of the
// first output tile also write the chunk's part of G = A^T A,
// Gp[chunk][i][j].  grid (ceil(Ct / 256), ceil(N / kEcChunk)).
__global__ void __launch_bounds__(256) ec_stats_kernel(const float *__restrict__ S, int N, int Cs,
                                                       int Ct, int Csp, int m,
                                                       const double *__restrict__ E,
                                                       double *__restrict__ Vp,
                                                       double *__restrict__ Gp) {
    __shared__ double a[kEcChunk][kMaxCsp];
    const int n0 = blockIdx.y * kEcChunk, nn = min(kEcChunk, N - n0);
    for (int e = threadIdx.x; e < kEcChunk * kMaxCsp; e += blockDim.x) {
        const int r = e / kMaxCsp, j = e % kMaxCsp;
        a[r][j] = (r < nn && j < Csp) ? (double)S[(size_t)(n0 + r) * Cs + (size_t)m * Csp + j] : 0.0;
    }
    __syncthreads();
    const int ct = blockIdx.x * blockDim.x + threadIdx.x;
    if (ct < Ct) {
        double v[kMaxCsp];
#pragma unroll
        for (int j = 0; j < kMaxCsp; ++j) v[j] = 0.0;
#pragma unroll 8
        for (int r = 0; r < nn; ++r) {
            const double e = E[(size_t)(n0 + r) * Ct + ct];
#pragma unroll
            for (int j = 0; j < kMaxCsp; ++j) v[j] = fma(a[r][j], e, v[j]);
        }
        for (int j = 0; j < Csp; ++j) Vp[((size_t)blockIdx.y * Csp + j) * Ct + ct] = v[j];
    }
    if (blockIdx.x == 0 && threadIdx.x < Csp * Csp) {
        const int i = threadIdx.x / Csp, j = threadIdx.x % Csp;
        double g = 0.0;
        for (int r = 0; r < nn; ++r) g = fma(a[r][i], a[r][j], g);
        Gp[((size_t)blockIdx.y * Csp + i) * Csp + j] = g;
    }
}

// G = sum of the chunk parts, in chunk order (one thread per entry).
__global__ void ec_gram_kernel(int Csp, int nchunks, const double *__restrict__ Gp,
                               double *__restrict__ G) {
    const int e = threadIdx.x;
    if (e >= Csp * Csp) return;
    double g = 0.0;
    for (int c = 0; c < nchunks; ++c) g += Gp[(size_t)c * Csp * Csp + e];
    G[e] = g;
}

// In-place Cholesky of the Csp x Csp matrix in L (lower triangle used);
// false when it is not positive definite (relative pivot test).
__device__ bool cholesky(double *L, int n) {
    double scale = 0.0;
    for (int i = 0; i < n; ++i) scale = fmax(scale, L[i * n + i]);
    for (int j = 0; j < n; ++j) {
        double d = L[j * n + j];
        for (int k = 0; k < j; ++k) d -= L[j * n + k] * L[j * n + k];
        if (!(d > 1e-12 * scale)) return false;
        d = sqrt(d);
        L[j * n + j] = d;
        for (int i = j + 1; i < n; ++i) {
            double s = L[i * n + j];
            for (int k = 0; k < j; ++k) s -= L[i * n + k] * L[j * n + k];
            L[i * n + j] = s / d;
        }
    }
    return true;
}

// U = sum of the partials + G D_old[k_old(c_t)]; saves the old codes and
// codewords; block 0 factors G (flag on failure).
__global__ void __launch_bounds__(256) ec_u_kernel(int N, int Ct, int Csp, int K, int nchunks,
                                                   const double *__restrict__ Vp,
                                                   const double *__restrict__ G,
                                                   const double *__restrict__ Dm,
                                                   const uint8_t *__restrict__ codes_m,
                                                   double *__restrict__ U,
                                                   double *__restrict__ Dold,
                                                   uint8_t *__restrict__ kold,
                                                   double *__restrict__ Lf, int *__restrict__ flag) {
    const int ct = blockIdx.x * blockDim.x + threadIdx.x;
    if (blockIdx.x == 0) {
        for (int e = threadIdx.x; e < K * Csp; e += blockDim.x) Dold[e] = Dm[e];
        if (threadIdx.x == 0) {
            double L[kMaxCsp * kMaxCsp];
            for (int e = 0; e < Csp * Csp; ++e) L[e] = G[e];
            if (!cholesky(L, Csp)) *flag = 1;
            for (int e = 0; e < Csp * Csp; ++e) Lf[e] = L[e];
        }
    }
    if (ct >= Ct) return;
    const int k = min((int)codes_m[ct], K - 1);
    kold[ct] = (uint8_t)k;
    const double *d = Dm + (size_t)k * Csp;
    for (int j = 0; j < Csp; ++j) {
        double u = 0.0;
        for (int c = 0; c < nchunks; ++c) u += Vp[((size_t)c * Csp + j) * Ct + ct];
        for (int i = 0; i < Csp; ++i) u = fma(G[j * Csp + i], d[i], u);
        U[(size_t)j * Ct + ct] = u;
    }
}

// Eq. 11 for every k (one warp each: lanes take every 32nd member of L_k,
// then a fixed butterfly adds the lanes), then q_k = D_k^T G D_k.
__global__ void ec_codeword_kernel(int Ct, int Csp, int K, const double *__restrict__ U,
                                   const int *__restrict__ order, const int *__restrict__ starts,
                                   const double *__restrict__ G, const double *__restrict__ Lf,
                                   double *__restrict__ Dm, double *__restrict__ q) {
    const int k = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
    if (k >= K) return;
    const int s0 = starts[k], s1 = starts[k + 1];
    double part[kMaxCsp];
#pragma unroll
    for (int j = 0; j < kMaxCsp; ++j) part[j] = 0.0;
    for (int e = s0 + lane; e < s1; e += 32) {
        const int ct = order[e];
#pragma unroll
        for (int j = 0; j < kMaxCsp; ++j)
            if (j < Csp) part[j] += U[(size_t)j * Ct + ct];
    }
#pragma unroll
    for (int j = 0; j < kMaxCsp; ++j)
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) part[j] += __shfl_xor_sync(0xffffffffu, part[j], o);
    if (lane != 0) return;
    double *d = Dm + (size_t)k * Csp;
    if (s1 > s0) {
        double b[kMaxCsp];
        for (int j = 0; j < Csp; ++j) b[j] = part[j] / (double)(s1 - s0);
        // L y = b, L^T d = y
        for (int i = 0; i < Csp; ++i) {
            double s = b[i];
            for (int t = 0; t < i; ++t) s -= Lf[i * Csp + t] * b[t];
            b[i] = s / Lf[i * Csp + i];
        }
        for (int i = Csp - 1; i >= 0; --i) {
            double s = b[i];
            for (int t = i + 1; t < Csp; ++t) s -= Lf[t * Csp + i] * b[t];
            b[i] = s / Lf[i * Csp + i];
        }
        for (int j = 0; j < Csp; ++j) d[j] = b[j];
    }
    double qq = 0.0;
    for (int i = 0; i < Csp; ++i) {
        double gi = 0.0;
        for (int j = 0; j < Csp; ++j) gi = fma(G[i * Csp + j], d[j], gi);
        qq = fma(d[i], gi, qq);
    }
    q[k] = qq;
}

// Eq. 12 for every output.
__global__ void __launch_bounds__(256) ec_assign_kernel(int Ct, int Csp, int K,
                                                        const double *__restrict__ U,
                                                        const double *__restrict__ Dm,
                                                        const double *__restrict__ q,
                                                        uint8_t *__restrict__ codes_m) {
    __shared__ double dsh[kMaxK * kMaxCsp];
    __shared__ double qsh[kMaxK];
    for (int e = threadIdx.x; e < K * Csp; e += blockDim.x) dsh[e] = Dm[e];
    for (int e = threadIdx.x; e < K; e += blockDim.x) qsh[e] = q[e];
    __syncthreads();
    const int ct = blockIdx.x * blockDim.x + threadIdx.x;
    if (ct >= Ct) return;
    double u[kMaxCsp];
    for (int j = 0; j < Csp; ++j) u[j] = U[(size_t)j * Ct + ct];
    int best = 0;
    double best_c = 0.0;
    for (int k = 0; k < K; ++k) {
        double dot = 0.0;
        for (int j = 0; j < Csp; ++j) dot = fma(dsh[k * Csp + j], u[j], dot);
        const double c = qsh[k] - 2.0 * dot;
        if (k == 0 || c < best_c) {
            best = k;
            best_c = c;
        }
    }
    codes_m[ct] = (uint8_t)best;
}

// E += A (D_old[k_old] - D_new[k_new])^T, one thread per (n, c_t).
__global__ void ec_residual_kernel(const float *__restrict__ S, int N, int Cs, int Ct, int Csp,
                                   int m, const double *__restrict__ Dold,
                                   const uint8_t *__restrict__ kold,
                                   const double *__restrict__ Dm,
                                   const uint8_t *__restrict__ codes_m, double *__restrict__ E) {
    const long long total = (long long)N * Ct;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int ct = (int)(i % Ct);
        const long long n = i / Ct;
        const double *o = Dold + (size_t)kold[ct] * Csp, *w = Dm + (size_t)codes_m[ct] * Csp;
        const float *s = S + n * Cs + (size_t)m * Csp;
        double delta = 0.0;
        for (int j = 0; j < Csp; ++j) delta = fma((double)s[j], o[j] - w[j], delta);
        E[i] += delta;
    }
}

__global__ void ec_narrow_kernel(const double *__restrict__ in, float *__restrict__ out, int n) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
        out[i] = __double2float_rn(in[i]);
}

__global__ void ec_widen_kernel(const float *__restrict__ in, double *__restrict__ out, int n) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
        out[i] = (double)in[i];
}

struct EcWs {
    size_t E, Dw, Vp, Gp, U, G, Lf, Dold, kold, q, order, starts, flag, total;
};

EcWs ec_ws_layout(int N, int Cs, int Ct, int Csp, int K) {
    const int M = Cs / Csp, nch = cdiv(N, kEcChunk);
    EcWs w;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t o = off;
        off += align_up(bytes, kWsAlign);
        return o;
    };
    w.E = take((size_t)N * Ct * sizeof(double));
    w.Dw = take((size_t)M * K * Csp * sizeof(double));
    w.Vp = take((size_t)nch * Csp * Ct * sizeof(double));
    w.Gp = take((size_t)nch * Csp * Csp * sizeof(double));
    w.U = take((size_t)Csp * Ct * sizeof(double));
    w.G = take((size_t)Csp * Csp * sizeof(double));
    w.Lf = take((size_t)Csp * Csp * sizeof(double));
    w.Dold = take((size_t)K * Csp * sizeof(double));
    w.kold = take((size_t)Ct);
    w.q = take((size_t)K * sizeof(double));
    w.order = take((size_t)Ct * sizeof(int));
    w.starts = take((size_t)(K + 1) * sizeof(int));
    w.flag = take(sizeof(int));
    w.total = off;
    return w;
}

}  // namespace qcnn

using namespace qcnn;

namespace {

bool ec_args_ok(int N, int Cs, int Ct, int Csp, int K) {
    if (N <= 0 || Ct <= 0 || Cs <= 0 || Csp < 1 || Csp > kMaxCsp || K < 1 || K > kMaxK ||
        Cs % Csp != 0)
        return false;
    return (long long)N * Ct < INT_MAX && (long long)N * Cs < INT_MAX &&
           (long long)Cs / Csp * K * Csp < INT_MAX;
}

}  // namespace

extern "C" {

qcnn_status qcnn_ec_quantize_fc_workspace_size(int N, int Cs, int Ct, int Csp, int K,
                                               size_t *bytes) {
    if (!bytes || !ec_args_ok(N, Cs, Ct, Csp, K)) return QCNN_ERR_INVALID_ARG;
    *bytes = ec_ws_layout(N, Cs, Ct, Csp, K).total;
    return QCNN_OK;
}

qcnn_status qcnn_ec_quantize_fc(const float *S, const float *T, int N, int Cs, int Ct, int Csp,
                                int K, float *D, uint8_t *codes, int outer, int inner,
                                void *workspace, size_t workspace_bytes, void *stream) {
    if (!S || !T || !D || !codes || outer < 0 || inner < 0 || !ec_args_ok(N, Cs, Ct, Csp, K))
        return QCNN_ERR_INVALID_ARG;
    const EcWs L = ec_ws_layout(N, Cs, Ct, Csp, K);
    if (!workspace || workspace_bytes < L.total ||
        reinterpret_cast<uintptr_t>(workspace) % kWsAlign != 0)
        return QCNN_ERR_WORKSPACE;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    uint8_t *b = static_cast<uint8_t *>(workspace);
    double *E = reinterpret_cast<double *>(b + L.E);
    double *Dw = reinterpret_cast<double *>(b + L.Dw);
    double *Vp = reinterpret_cast<double *>(b + L.Vp);
    double *Gp = reinterpret_cast<double *>(b + L.Gp);
    double *U = reinterpret_cast<double *>(b + L.U);
    double *G = reinterpret_cast<double *>(b + L.G);
    double *Lf = reinterpret_cast<double *>(b + L.Lf);
    double *Dold = reinterpret_cast<double *>(b + L.Dold);
    uint8_t *kold = b + L.kold;
    double *q = reinterpret_cast<double *>(b + L.q);
    int *order = reinterpret_cast<int *>(b + L.order);
    int *starts = reinterpret_cast<int *>(b + L.starts);
    int *flag = reinterpret_cast<int *>(b + L.flag);
    const int M = Cs / Csp, nch = cdiv(N, kEcChunk), sms = num_sms();
    qcnn_status rc;
    if ((rc = cuda_status(cudaMemsetAsync(flag, 0, sizeof(int), st))) != QCNN_OK) return rc;
    const int nD = M * K * Csp;
    ec_widen_kernel<<<std::min(cdiv(nD, 256), sms * 8), 256, 0, st>>>(D, Dw, nD);
    if ((rc = after_launch()) != QCNN_OK) return rc;
    const long long NC = (long long)N * Ct;
    const int eblocks = (int)std::min<long long>((NC + 255) / 256, (long long)sms * 16);
    ec_init_kernel<<<eblocks, 256, 0, st>>>(S, T, N, Cs, Ct, Csp, K, Dw, codes, E);
    if ((rc = after_launch()) != QCNN_OK) return rc;
    const dim3 sgrid(cdiv(Ct, 256), nch);
    for (int t = 0; t < outer; ++t) {
        for (int m = 0; m < M; ++m) {
            double *Dm = Dw + (size_t)m * K * Csp;
            uint8_t *cm = codes + (size_t)m * Ct;
            ec_stats_kernel<<<sgrid, 256, 0, st>>>(S, N, Cs, Ct, Csp, m, E, Vp, Gp);
            if ((rc = after_launch()) != QCNN_OK) return rc;
            ec_gram_kernel<<<1, 64, 0, st>>>(Csp, nch, Gp, G);
            if ((rc = after_launch()) != QCNN_OK) return rc;
            ec_u_kernel<<<cdiv(Ct, 256), 256, 0, st>>>(N, Ct, Csp, K, nch, Vp, G, Dm, cm, U, Dold,
                                                       kold, Lf, flag);
            if ((rc = after_launch()) != QCNN_OK) return rc;
            for (int i = 0; i < inner; ++i) {
                kmeans_order_kernel<<<1, 1024, 0, st>>>(i == 0 ? kold : cm, Ct, K, order, starts);
                if ((rc = after_launch()) != QCNN_OK) return rc;
                ec_codeword_kernel<<<cdiv(K * 32, 256), 256, 0, st>>>(Ct, Csp, K, U, order,
                                                                      starts, G, Lf, Dm, q);
                if ((rc = after_launch()) != QCNN_OK) return rc;
                ec_assign_kernel<<<cdiv(Ct, 256), 256, 0, st>>>(Ct, Csp, K, U, Dm, q, cm);
                if ((rc = after_launch()) != QCNN_OK) return rc;
            }
            ec_residual_kernel<<<eblocks, 256, 0, st>>>(S, N, Cs, Ct, Csp, m, Dold, kold, Dm, cm, E);
            if ((rc = after_launch()) != QCNN_OK) return rc;
        }
    }
    ec_narrow_kernel<<<std::min(cdiv(nD, 256), sms * 8), 256, 0, st>>>(Dw, D, nD);
    if ((rc = after_launch()) != QCNN_OK) return rc;
    int h_flag = 0;
    if ((rc = cuda_status(cudaMemcpyAsync(&h_flag, flag, sizeof(int), cudaMemcpyDeviceToHost,
                                          st))) != QCNN_OK)
        return rc;
    if ((rc = sync_and_check(st)) != QCNN_OK) return rc;
    return h_flag ? QCNN_ERR_DATA : QCNN_OK;
}

}  // extern "C"
