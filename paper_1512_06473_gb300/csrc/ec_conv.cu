// ec_conv.cu -- error-corrected quantization of a conv layer (Sec. 3.3.2,
// Appendix B).
//
// Minimises sum_{n,p_t} ||sum_{(p_k,p_s)} sum_m (D^(m) B_pk^(m))^T S_{n,p_s}^(m)
// - T_{n,p_t}||^2 by block coordinate descent over the sub-spaces m, in order.
// The device keeps the residual E = T - (current approximation),
// [N][Ct][Ho*Wo] in double; every step below changes one term of the
// approximation and updates E in place, so E is always the residual the
// next step needs (Eq. B.2, B.5, B.7 are E plus the term being replaced).
// For sub-space m, `inner` times:
//   group : the (c_t, p_k) pairs of the sub-space by codeword (stable
//           counting sort), cut into per-channel segments;
//   D pass: for k = 0 .. K-1 in order (Eq. B.4 - B.6): with
//           z = sum_{p_k : k(c_t,p_k) = k} x(n, p_s(p_t, p_k)) over each
//           segment, G_k = sum z z^T and V = sum z E; the least-squares
//           solution is D_k + G_k^-1 V (normal equations of Eq. B.6 with
//           Q_k = E + D_k^T z); then E -= (D_k,new - D_k)^T z.  A codeword
//           without pairs keeps its value;
//   B pass: for p_k = 0 .. kh*kw-1 in order (Eq. B.7 - B.8): G = sum x x^T
//           and U[:, c_t] = sum x E + G D_k(c_t,p_k) over (n, p_t); each
//           channel takes argmin_k D_k^T G D_k - 2 D_k^T U[:, c_t] (ties to
//           the smallest k); then E -= (D_new - D_old)^T x.
// All partial sums are taken over a fixed partition and added in a fixed
// order.  Everything is double: the offline quantizer, run once per layer.
#include "qcnn_internal.cuh"

#include <algorithm>
#include <climits>

namespace qcnn {

struct EcConvGeo {
    int N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K, M, Ho, Wo, P, kk;
};

// x_j(n, p_s(p_t, p_k)) of sub-space m (zero outside the map).
__device__ __forceinline__ double ecx(const float *__restrict__ S, const EcConvGeo &g, int n, int m,
                                      int j, int pt, int pk) {
    const int oy = pt / g.Wo, ox = pt - oy * g.Wo;
    const int ky = pk / g.kw, kx = pk - ky * g.kw;
    const int iy = oy * g.stride - g.pad + ky, ix = ox * g.stride - g.pad + kx;
    if (iy < 0 || iy >= g.H || ix < 0 || ix >= g.W) return 0.0;
    return (double)S[(((size_t)n * g.Cs + (size_t)m * g.Csp + j) * g.H + iy) * g.W + ix];
}

// E = T - sum_m sum_pk D[m][k(c_t,p_k,m)]^T x, one thread per (n, c_t, p_t).
__global__ void ecc_init_kernel(const float *__restrict__ S, const float *__restrict__ T,
                                EcConvGeo g, const double *__restrict__ Dw,
                                const uint8_t *__restrict__ codes, double *__restrict__ E) {
    const long long total = (long long)g.N * g.Ct * g.P;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int pt = (int)(i % g.P);
        const long long r = i / g.P;
        const int ct = (int)(r % g.Ct), n = (int)(r / g.Ct);
        double y = 0.0;
        for (int m = 0; m < g.M; ++m)
            for (int pk = 0; pk < g.kk; ++pk) {
                const double *d = Dw + ((size_t)m * g.K + codes[((size_t)ct * g.kk + pk) * g.M + m]) * g.Csp;
                for (int j = 0; j < g.Csp; ++j) y = fma(ecx(S, g, n, m, j, pt, pk), d[j], y);
            }
        E[i] = (double)T[i] - y;
    }
}

// lin[c_t * kk + p_k] = codes[c_t][p_k][m]
__global__ void ecc_codes_of_kernel(const uint8_t *__restrict__ codes, EcConvGeo g, int m,
                                    uint8_t *__restrict__ lin) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < g.Ct * g.kk; i += gridDim.x * blockDim.x)
        lin[i] = codes[(size_t)i * g.M + m];
}

// For codeword k (one thread each): its pairs (sorted by c_t * kk + p_k) cut
// into segments of one channel: seg_ct / seg_start / seg_len [K][Ct], nseg[K].
__global__ void ecc_segments_kernel(const int *__restrict__ order, const int *__restrict__ starts,
                                    EcConvGeo g, int *__restrict__ seg_ct,
                                    int *__restrict__ seg_start, int *__restrict__ seg_len,
                                    int *__restrict__ nseg) {
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= g.K) return;
    int ns = 0;
    const int e0 = starts[k], e1 = starts[k + 1];
    for (int e = e0; e < e1;) {
        const int ct = order[e] / g.kk;
        int f = e + 1;
        while (f < e1 && order[f] / g.kk == ct) ++f;
        seg_ct[(size_t)k * g.Ct + ns] = ct;
        seg_start[(size_t)k * g.Ct + ns] = e;
        seg_len[(size_t)k * g.Ct + ns] = f - e;
        ++ns;
        e = f;
    }
    nseg[k] = ns;
}

constexpr int kEccBlocks = 128;   // fixed partition of the D-pass sums
constexpr int kEccThreads = 256;
constexpr int kEccStat = kMaxCsp * kMaxCsp + kMaxCsp;  // G (Csp x Csp) + V (Csp)

// Block reduction of `cnt` doubles per thread into vals[0..cnt) of thread 0,
// in a fixed order: a shuffle tree inside each warp, then the warps' sums in
// warp order.  sh holds kEccStat doubles per warp.
__device__ void ecc_block_reduce(double *vals, int cnt, double *sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    for (int c = 0; c < cnt; ++c) {
        double v = vals[c];
        for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
        if (lane == 0) sh[warp * kEccStat + c] = v;
    }
    __syncthreads();
    if (threadIdx.x == 0)
        for (int c = 0; c < cnt; ++c) {
            double t = sh[c];
            for (int w = 1; w < nw; ++w) t += sh[w * kEccStat + c];
            vals[c] = t;
        }
}

// D pass, codeword k: per block, G_k and V over the segments b, b + B, ...
__global__ void __launch_bounds__(kEccThreads) ecc_dstats_kernel(
    const float *__restrict__ S, EcConvGeo g, int m, int k, const double *__restrict__ E,
    const int *__restrict__ order, const int *__restrict__ seg_ct,
    const int *__restrict__ seg_start, const int *__restrict__ seg_len,
    const int *__restrict__ nseg, double *__restrict__ part) {
    __shared__ double sh[(kEccThreads / 32) * kEccStat];
    double acc[kEccStat];
    for (int c = 0; c < kEccStat; ++c) acc[c] = 0.0;
    const int ns = nseg[k];
    if ((int)blockIdx.x >= ns) return;  // no segment for this block: its part is not read
    const int items = g.N * g.P;
    for (int sgi = blockIdx.x; sgi < ns; sgi += gridDim.x) {
        const int ct = seg_ct[(size_t)k * g.Ct + sgi];
        const int s0 = seg_start[(size_t)k * g.Ct + sgi], len = seg_len[(size_t)k * g.Ct + sgi];
        for (int it = threadIdx.x; it < items; it += blockDim.x) {
            const int n = it / g.P, pt = it - n * g.P;
            double z[kMaxCsp];
            for (int j = 0; j < g.Csp; ++j) z[j] = 0.0;
            for (int q = 0; q < len; ++q) {
                const int pk = order[s0 + q] - ct * g.kk;
                for (int j = 0; j < g.Csp; ++j) z[j] += ecx(S, g, n, m, j, pt, pk);
            }
            const double e = E[((size_t)n * g.Ct + ct) * g.P + pt];
            for (int i = 0; i < g.Csp; ++i) {
                for (int j = 0; j < g.Csp; ++j) acc[i * g.Csp + j] = fma(z[i], z[j], acc[i * g.Csp + j]);
                acc[g.Csp * g.Csp + i] = fma(z[i], e, acc[g.Csp * g.Csp + i]);
            }
        }
    }
    const int cnt = g.Csp * g.Csp + g.Csp;
    ecc_block_reduce(acc, cnt, sh);
    if (threadIdx.x == 0)
        for (int c = 0; c < cnt; ++c) part[(size_t)blockIdx.x * kEccStat + c] = acc[c];
}

// In-place Cholesky (lower triangle); false if not positive definite.
__device__ bool ecc_cholesky(double *L, int n) {
    double scale = 0.0;
    for (int i = 0; i < n; ++i) scale = fmax(scale, L[i * n + i]);
    for (int j = 0; j < n; ++j) {
        double d = L[j * n + j];
        for (int t = 0; t < j; ++t) d -= L[j * n + t] * L[j * n + t];
        if (!(d > 1e-12 * scale)) return false;
        d = sqrt(d);
        L[j * n + j] = d;
        for (int i = j + 1; i < n; ++i) {
            double s = L[i * n + j];
            for (int t = 0; t < j; ++t) s -= L[i * n + t] * L[j * n + t];
            L[i * n + j] = s / d;
        }
    }
    return true;
}

// D pass, codeword k: add the parts of the blocks that had segments, in
// block order (one thread per statistic), solve, update D_k;
// delta = D_k,new - D_k,old (zero when k has no pairs).  Launch with at least
// kEccStat threads.
__global__ void ecc_dsolve_kernel(EcConvGeo g, int m, int k, int nblocks,
                                  const double *__restrict__ part, const int *__restrict__ nseg,
                                  double *__restrict__ Dw, double *__restrict__ delta,
                                  int *__restrict__ flag) {
    __shared__ double tot[kEccStat];
    const int C = g.Csp, cnt = C * C + C;
    const int nb = min(nblocks, nseg[k]);
    for (int c = threadIdx.x; c < cnt; c += blockDim.x) {
        double t = 0.0;
        for (int blk = 0; blk < nb; ++blk) t += part[(size_t)blk * kEccStat + c];
        tot[c] = t;
    }
    __syncthreads();
    if (threadIdx.x != 0) return;
    double *d = Dw + ((size_t)m * g.K + k) * C;
    if (nseg[k] == 0) {
        for (int j = 0; j < C; ++j) delta[j] = 0.0;
        return;
    }
    double L[kMaxCsp * kMaxCsp], b[kMaxCsp];
    for (int c = 0; c < C * C; ++c) L[c] = tot[c];
    for (int j = 0; j < C; ++j) b[j] = tot[C * C + j];
    if (!ecc_cholesky(L, C)) {
        *flag = 1;
        for (int j = 0; j < C; ++j) delta[j] = 0.0;
        return;
    }
    for (int i = 0; i < C; ++i) {  // L y = V, L^T s = y: the correction G_k^-1 V
        double s = b[i];
        for (int t = 0; t < i; ++t) s -= L[i * C + t] * b[t];
        b[i] = s / L[i * C + i];
    }
    for (int i = C - 1; i >= 0; --i) {
        double s = b[i];
        for (int t = i + 1; t < C; ++t) s -= L[t * C + i] * b[t];
        b[i] = s / L[i * C + i];
    }
    for (int j = 0; j < C; ++j) {
        delta[j] = b[j];
        d[j] += b[j];
    }
}

// D pass, codeword k: E -= delta^T z over its segments (same partition).
__global__ void __launch_bounds__(kEccThreads) ecc_dupdate_kernel(
    const float *__restrict__ S, EcConvGeo g, int m, int k, double *__restrict__ E,
    const int *__restrict__ order, const int *__restrict__ seg_ct,
    const int *__restrict__ seg_start, const int *__restrict__ seg_len,
    const int *__restrict__ nseg, const double *__restrict__ delta) {
    const int ns = nseg[k];
    const int items = g.N * g.P;
    double dl[kMaxCsp];
    for (int j = 0; j < g.Csp; ++j) dl[j] = delta[j];
    for (int sgi = blockIdx.x; sgi < ns; sgi += gridDim.x) {
        const int ct = seg_ct[(size_t)k * g.Ct + sgi];
        const int s0 = seg_start[(size_t)k * g.Ct + sgi], len = seg_len[(size_t)k * g.Ct + sgi];
        for (int it = threadIdx.x; it < items; it += blockDim.x) {
            const int n = it / g.P, pt = it - n * g.P;
            double v = 0.0;
            for (int q = 0; q < len; ++q) {
                const int pk = order[s0 + q] - ct * g.kk;
                for (int j = 0; j < g.Csp; ++j) v = fma(ecx(S, g, n, m, j, pt, pk), dl[j], v);
            }
            E[((size_t)n * g.Ct + ct) * g.P + pt] -= v;
        }
    }
}

constexpr int kEccChunk = 64;  // (n, p_t) items per partial sum of the B pass

// B pass, offset pk: Vp[chunk][j][c_t] = sum_{items in chunk} x_j E[n][c_t][p_t]
// and Gp[chunk] = sum x x^T.  grid (ceil(Ct / 256), ceil(N*P / kEccChunk)).
__global__ void __launch_bounds__(256) ecc_bstats_kernel(const float *__restrict__ S, EcConvGeo g,
                                                         int m, int pk,
                                                         const double *__restrict__ E,
                                                         double *__restrict__ Vp,
                                                         double *__restrict__ Gp) {
    __shared__ double xs[kEccChunk][kMaxCsp];
    const int i0 = blockIdx.y * kEccChunk, items = g.N * g.P, ni = min(kEccChunk, items - i0);
    for (int e = threadIdx.x; e < kEccChunk * kMaxCsp; e += blockDim.x) {
        const int r = e / kMaxCsp, j = e % kMaxCsp;
        double v = 0.0;
        if (r < ni && j < g.Csp) {
            const int it = i0 + r, n = it / g.P, pt = it - n * g.P;
            v = ecx(S, g, n, m, j, pt, pk);
        }
        xs[r][j] = v;
    }
    __syncthreads();
    const int ct = blockIdx.x * blockDim.x + threadIdx.x;
    if (ct < g.Ct) {
        double v[kMaxCsp];
        for (int j = 0; j < kMaxCsp; ++j) v[j] = 0.0;
        for (int r = 0; r < ni; ++r) {
            const int it = i0 + r, n = it / g.P, pt = it - n * g.P;
            const double e = E[((size_t)n * g.Ct + ct) * g.P + pt];
            for (int j = 0; j < kMaxCsp; ++j) v[j] = fma(xs[r][j], e, v[j]);
        }
        for (int j = 0; j < g.Csp; ++j) Vp[((size_t)blockIdx.y * g.Csp + j) * g.Ct + ct] = v[j];
    }
    if (blockIdx.x == 0 && threadIdx.x < g.Csp * g.Csp) {
        const int i = threadIdx.x / g.Csp, j = threadIdx.x % g.Csp;
        double s = 0.0;
        for (int r = 0; r < ni; ++r) s = fma(xs[r][i], xs[r][j], s);
        Gp[((size_t)blockIdx.y * g.Csp + i) * g.Csp + j] = s;
    }
}

// B pass, offset pk: G (chunk order), its Cholesky check, q_k = D_k^T G D_k
// (block 0); U[:, c_t] = sum of the chunk parts + G D_k(c_t,pk) and the old
// codes (all blocks).
__global__ void __launch_bounds__(256) ecc_bu_kernel(EcConvGeo g, int m, int pk, int nch,
                                                     const double *__restrict__ Vp,
                                                     const double *__restrict__ Gp,
                                                     const double *__restrict__ Dw,
                                                     const uint8_t *__restrict__ codes,
                                                     double *__restrict__ U, double *__restrict__ q,
                                                     uint8_t *__restrict__ kold,
                                                     int *__restrict__ flag) {
    __shared__ double G[kMaxCsp * kMaxCsp];
    const int C = g.Csp;
    for (int e = threadIdx.x; e < C * C; e += blockDim.x) {
        double s = 0.0;
        for (int c = 0; c < nch; ++c) s += Gp[(size_t)c * C * C + e];
        G[e] = s;
    }
    __syncthreads();
    const double *Dm = Dw + (size_t)m * g.K * C;
    if (blockIdx.x == 0) {
        if (threadIdx.x == 0) {
            double L[kMaxCsp * kMaxCsp];
            for (int e = 0; e < C * C; ++e) L[e] = G[e];
            if (!ecc_cholesky(L, C)) *flag = 1;
        }
        for (int k = threadIdx.x; k < g.K; k += blockDim.x) {
            const double *d = Dm + (size_t)k * C;
            double qq = 0.0;
            for (int i = 0; i < C; ++i) {
                double gi = 0.0;
                for (int j = 0; j < C; ++j) gi = fma(G[i * C + j], d[j], gi);
                qq = fma(d[i], gi, qq);
            }
            q[k] = qq;
        }
    }
    const int ct = blockIdx.x * blockDim.x + threadIdx.x;
    if (ct >= g.Ct) return;
    const int k = codes[((size_t)ct * g.kk + pk) * g.M + m];
    kold[ct] = (uint8_t)k;
    const double *d = Dm + (size_t)k * C;
    for (int j = 0; j < C; ++j) {
        double u = 0.0;
        for (int c = 0; c < nch; ++c) u += Vp[((size_t)c * C + j) * g.Ct + ct];
        for (int i = 0; i < C; ++i) u = fma(G[j * C + i], d[i], u);
        U[(size_t)j * g.Ct + ct] = u;
    }
}

// B pass, offset pk: k(c_t, pk) = argmin_k q_k - 2 D_k^T U[:, c_t].
__global__ void __launch_bounds__(256) ecc_bassign_kernel(EcConvGeo g, int m, int pk,
                                                          const double *__restrict__ U,
                                                          const double *__restrict__ Dw,
                                                          const double *__restrict__ q,
                                                          uint8_t *__restrict__ codes) {
    __shared__ double dsh[kMaxK * kMaxCsp];
    __shared__ double qsh[kMaxK];
    const int C = g.Csp;
    for (int e = threadIdx.x; e < g.K * C; e += blockDim.x) dsh[e] = Dw[(size_t)m * g.K * C + e];
    for (int e = threadIdx.x; e < g.K; e += blockDim.x) qsh[e] = q[e];
    __syncthreads();
    const int ct = blockIdx.x * blockDim.x + threadIdx.x;
    if (ct >= g.Ct) return;
    double u[kMaxCsp];
    for (int j = 0; j < C; ++j) u[j] = U[(size_t)j * g.Ct + ct];
    int best = 0;
    double best_c = 0.0;
    for (int k = 0; k < g.K; ++k) {
        double dot = 0.0;
        for (int j = 0; j < C; ++j) dot = fma(dsh[k * C + j], u[j], dot);
        const double c = qsh[k] - 2.0 * dot;
        if (k == 0 || c < best_c) {
            best = k;
            best_c = c;
        }
    }
    codes[((size_t)ct * g.kk + pk) * g.M + m] = (uint8_t)best;
}

// B pass, offset pk: E -= (D_new - D_old)^T x, one thread per (n, c_t, p_t).
__global__ void ecc_bupdate_kernel(const float *__restrict__ S, EcConvGeo g, int m, int pk,
                                   const double *__restrict__ Dw, const uint8_t *__restrict__ kold,
                                   const uint8_t *__restrict__ codes, double *__restrict__ E) {
    const long long total = (long long)g.N * g.Ct * g.P;
    const double *Dm = Dw + (size_t)m * g.K * g.Csp;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int pt = (int)(i % g.P);
        const long long r = i / g.P;
        const int ct = (int)(r % g.Ct), n = (int)(r / g.Ct);
        const int ko = kold[ct], kn = codes[((size_t)ct * g.kk + pk) * g.M + m];
        if (ko == kn) continue;
        double v = 0.0;
        for (int j = 0; j < g.Csp; ++j)
            v = fma(ecx(S, g, n, m, j, pt, pk), Dm[(size_t)ko * g.Csp + j] - Dm[(size_t)kn * g.Csp + j], v);
        E[i] += v;
    }
}

// codes >= K are clamped to K - 1 (the codes array is in/out)
__global__ void ecc_clamp_kernel(uint8_t *__restrict__ codes, long long n, int K) {
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x)
        if (codes[i] >= K) {
            QCNN_CHECK(false, QCNN_CHECK_CODE);
            codes[i] = (uint8_t)(K - 1);
        }
}

__global__ void ecc_cast_kernel(const double *__restrict__ in, float *__restrict__ out,
                                const float *__restrict__ fin, double *__restrict__ dout, int n) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        if (in) out[i] = __double2float_rn(in[i]);
        else dout[i] = (double)fin[i];
    }
}

struct EccWs {
    size_t E, Dw, lin, order, starts, seg_ct, seg_start, seg_len, nseg, part, delta, Vp, Gp, U, q,
        kold, flag, total;
};

EccWs ecc_ws_layout(const EcConvGeo &g) {
    EccWs w;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t o = off;
        off += align_up(bytes, kWsAlign);
        return o;
    };
    const int nch = cdiv(g.N * g.P, kEccChunk);
    w.E = take((size_t)g.N * g.Ct * g.P * sizeof(double));
    w.Dw = take((size_t)g.M * g.K * g.Csp * sizeof(double));
    w.lin = take((size_t)g.Ct * g.kk);
    w.order = take((size_t)g.Ct * g.kk * sizeof(int));
    w.starts = take((size_t)(g.K + 1) * sizeof(int));
    w.seg_ct = take((size_t)g.K * g.Ct * sizeof(int));
    w.seg_start = take((size_t)g.K * g.Ct * sizeof(int));
    w.seg_len = take((size_t)g.K * g.Ct * sizeof(int));
    w.nseg = take((size_t)g.K * sizeof(int));
    w.part = take((size_t)kEccBlocks * kEccStat * sizeof(double));
    w.delta = take(kMaxCsp * sizeof(double));
    w.Vp = take((size_t)nch * g.Csp * g.Ct * sizeof(double));
    w.Gp = take((size_t)nch * g.Csp * g.Csp * sizeof(double));
    w.U = take((size_t)g.Csp * g.Ct * sizeof(double));
    w.q = take((size_t)g.K * sizeof(double));
    w.kold = take((size_t)g.Ct);
    w.flag = take(sizeof(int));
    w.total = off;
    return w;
}

}  // namespace qcnn

using namespace qcnn;

namespace {

bool ecc_geo(int N, int Cs, int H, int W, int Ct, int kh, int kw, int stride, int pad, int Csp,
             int K, EcConvGeo *g) {
    if (N <= 0 || Cs <= 0 || H <= 0 || W <= 0 || Ct <= 0 || kh <= 0 || kw <= 0 || stride <= 0 ||
        pad < 0 || Csp < 1 || Csp > kMaxCsp || K < 1 || K > kMaxK || Cs % Csp != 0)
        return false;
    if (H + 2 * pad < kh || W + 2 * pad < kw) return false;
    const int Ho = (H + 2 * pad - kh) / stride + 1, Wo = (W + 2 * pad - kw) / stride + 1;
    if (Ho <= 0 || Wo <= 0) return false;
    if ((long long)N * Ct * Ho * Wo >= INT_MAX || (long long)N * Cs * H * W >= INT_MAX ||
        (long long)Ct * kh * kw >= INT_MAX / 8 || (long long)N * Ho * Wo >= INT_MAX)
        return false;
    *g = EcConvGeo{N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K, Cs / Csp, Ho, Wo, Ho * Wo, kh * kw};
    return true;
}

}  // namespace

extern "C" {

qcnn_status qcnn_ec_quantize_conv_workspace_size(int N, int Cs, int H, int W, int Ct, int kh,
                                                 int kw, int stride, int pad, int Csp, int K,
                                                 size_t *bytes) {
    EcConvGeo g;
    if (!bytes || !ecc_geo(N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K, &g))
        return QCNN_ERR_INVALID_ARG;
    *bytes = ecc_ws_layout(g).total;
    return QCNN_OK;
}

qcnn_status qcnn_ec_quantize_conv(const float *S, const float *T, int N, int Cs, int H, int W,
                                  int Ct, int kh, int kw, int stride, int pad, int Csp, int K,
                                  float *D, uint8_t *codes, int outer, int inner, void *workspace,
                                  size_t workspace_bytes, void *stream) {
    EcConvGeo g;
    if (!S || !T || !D || !codes || outer < 0 || inner < 0 ||
        !ecc_geo(N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K, &g))
        return QCNN_ERR_INVALID_ARG;
    const EccWs L = ecc_ws_layout(g);
    if (!workspace || workspace_bytes < L.total ||
        reinterpret_cast<uintptr_t>(workspace) % kWsAlign != 0)
        return QCNN_ERR_WORKSPACE;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    uint8_t *b = static_cast<uint8_t *>(workspace);
    double *E = reinterpret_cast<double *>(b + L.E);
    double *Dw = reinterpret_cast<double *>(b + L.Dw);
    uint8_t *lin = b + L.lin;
    int *order = reinterpret_cast<int *>(b + L.order);
    int *starts = reinterpret_cast<int *>(b + L.starts);
    int *seg_ct = reinterpret_cast<int *>(b + L.seg_ct);
    int *seg_start = reinterpret_cast<int *>(b + L.seg_start);
    int *seg_len = reinterpret_cast<int *>(b + L.seg_len);
    int *nseg = reinterpret_cast<int *>(b + L.nseg);
    double *part = reinterpret_cast<double *>(b + L.part);
    double *delta = reinterpret_cast<double *>(b + L.delta);
    double *Vp = reinterpret_cast<double *>(b + L.Vp);
    double *Gp = reinterpret_cast<double *>(b + L.Gp);
    double *U = reinterpret_cast<double *>(b + L.U);
    double *q = reinterpret_cast<double *>(b + L.q);
    uint8_t *kold = b + L.kold;
    int *flag = reinterpret_cast<int *>(b + L.flag);
    const int sms = num_sms();
    const int nD = g.M * g.K * g.Csp;
    const long long NCP = (long long)g.N * g.Ct * g.P;
    const int eblocks = (int)std::min<long long>((NCP + 255) / 256, (long long)sms * 16);
    const int nch = cdiv(g.N * g.P, kEccChunk);
    qcnn_status rc;
    auto chk = [&]() { return after_launch(); };
    if ((rc = cuda_status(cudaMemsetAsync(flag, 0, sizeof(int), st))) != QCNN_OK) return rc;
    const long long ncodes = (long long)g.Ct * g.kk * g.M;
    ecc_clamp_kernel<<<(int)std::min<long long>((ncodes + 255) / 256, (long long)sms * 8), 256, 0,
                       st>>>(codes, ncodes, g.K);
    if ((rc = chk()) != QCNN_OK) return rc;
    ecc_cast_kernel<<<std::min(cdiv(nD, 256), sms * 8), 256, 0, st>>>(nullptr, nullptr, D, Dw, nD);
    if ((rc = chk()) != QCNN_OK) return rc;
    ecc_init_kernel<<<eblocks, 256, 0, st>>>(S, T, g, Dw, codes, E);
    if ((rc = chk()) != QCNN_OK) return rc;
    for (int t = 0; t < outer; ++t) {
        for (int m = 0; m < g.M; ++m) {
            for (int i = 0; i < inner; ++i) {
                // D pass (Eq. B.4 - B.6): codewords in order
                ecc_codes_of_kernel<<<std::max(1, std::min(cdiv(g.Ct * g.kk, 256), sms * 4)), 256, 0,
                                      st>>>(codes, g, m, lin);
                if ((rc = chk()) != QCNN_OK) return rc;
                kmeans_order_kernel<<<1, 1024, 0, st>>>(lin, g.Ct * g.kk, g.K, order, starts);
                if ((rc = chk()) != QCNN_OK) return rc;
                ecc_segments_kernel<<<cdiv(g.K, 128), 128, 0, st>>>(order, starts, g, seg_ct,
                                                                     seg_start, seg_len, nseg);
                if ((rc = chk()) != QCNN_OK) return rc;
                for (int k = 0; k < g.K; ++k) {
                    ecc_dstats_kernel<<<kEccBlocks, kEccThreads, 0, st>>>(
                        S, g, m, k, E, order, seg_ct, seg_start, seg_len, nseg, part);
                    if ((rc = chk()) != QCNN_OK) return rc;
                    ecc_dsolve_kernel<<<1, 96, 0, st>>>(g, m, k, kEccBlocks, part, nseg, Dw, delta,
                                                        flag);
                    if ((rc = chk()) != QCNN_OK) return rc;
                    ecc_dupdate_kernel<<<kEccBlocks, kEccThreads, 0, st>>>(
                        S, g, m, k, E, order, seg_ct, seg_start, seg_len, nseg, delta);
                    if ((rc = chk()) != QCNN_OK) return rc;
                }
                // B pass (Eq. B.7 - B.8): kernel offsets in order
                for (int pk = 0; pk < g.kk; ++pk) {
                    ecc_bstats_kernel<<<dim3(cdiv(g.Ct, 256), nch), 256, 0, st>>>(S, g, m, pk, E, Vp,
                                                                                Gp);
                    if ((rc = chk()) != QCNN_OK) return rc;
                    ecc_bu_kernel<<<cdiv(g.Ct, 256), 256, 0, st>>>(g, m, pk, nch, Vp, Gp, Dw, codes,
                                                                   U, q, kold, flag);
                    if ((rc = chk()) != QCNN_OK) return rc;
                    ecc_bassign_kernel<<<cdiv(g.Ct, 256), 256, 0, st>>>(g, m, pk, U, Dw, q, codes);
                    if ((rc = chk()) != QCNN_OK) return rc;
                    ecc_bupdate_kernel<<<eblocks, 256, 0, st>>>(S, g, m, pk, Dw, kold, codes, E);
                    if ((rc = chk()) != QCNN_OK) return rc;
                }
            }
        }
    }
    ecc_cast_kernel<<<std::min(cdiv(nD, 256), sms * 8), 256, 0, st>>>(Dw, D, nullptr, nullptr, nD);
    if ((rc = chk()) != QCNN_OK) return rc;
    int h_flag = 0;
    if ((rc = cuda_status(cudaMemcpyAsync(&h_flag, flag, sizeof(int), cudaMemcpyDeviceToHost, st))) !=
        QCNN_OK)
        return rc;
    if ((rc = sync_and_check(st)) != QCNN_OK) return rc;
    return h_flag ? QCNN_ERR_DATA : QCNN_OK;
}

}  // extern "C"
