// quantize.cu -- learning the PQ parameters: k-means in every sub-space
// (Sec. 3.1, Eq. 4 for FC weights; Sec. 3.2, Eq. 6 for conv kernels).
//
// For sub-space m the points are the m-th sub-vectors of all weight vectors
// (FC: one per c_t; conv: one per (c_t, p_k), index p = c_t * kh*kw + p_k).
// All M sub-spaces run at once.  One Lloyd round is three launches:
//   1. assign: every point to its nearest centroid.  Squared distances are
//      evaluated term by term in binary32 (subtract, square, add, each
//      rounded, no fused multiply-add), ties to the smallest index -- the
//      integer decision is taken in one stated precision, so it can be
//      checked bit for bit.
//   2. order: a stable counting sort of each sub-space's points by cluster
//      (warp match + per-warp counts, the same ranking as the chunked conv
//      prep), giving each cluster's points in index order.
//   3. update: one thread per (m, k, j) sums its cluster's coordinates in
//      double in index order, divides by the count and rounds to binary32;
//      a cluster without points keeps its centroid.  The fixed order makes
//      the centroids reproducible bit for bit.
// After `iters` rounds a last assignment writes the codes in the layer's
// layout.  Points are padded to CSP4 = 4 or 8 coordinates with zeros, which
// adds exact zeros to the distances.
#include "qcnn_internal.cuh"

#include <algorithm>
#include <climits>

namespace qcnn {

constexpr int kSortThreads = 1024;

// points[m][p][0..CSP4) from W viewed as [Ct][Cs][kk] (kk = 1 for FC).
__global__ void pq_points_kernel(const float *__restrict__ W, int Ct, int Cs, int kk, int Csp,
                                 int csp4, int M, float *__restrict__ pts) {
    const long long P = (long long)Ct * kk;
    const long long total = (long long)M * P * csp4;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int j = (int)(i % csp4);
        const long long r = i / csp4;
        const long long p = r % P;
        const int m = (int)(r / P);
        const long long ct = p / kk, pk = p % kk;
        pts[i] = j < Csp ? W[(ct * Cs + (long long)m * Csp + j) * kk + pk] : 0.f;
    }
}

// cen[m][k][0..CSP4) from a dense [M][K][Csp] array (zero padding), or back.
__global__ void pad_centroids_kernel(const float *__restrict__ in, int M, int K, int Csp,
                                     int csp4, float *__restrict__ out, int to_padded) {
    const int total = M * K * csp4;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
        const int j = i % csp4, mk = i / csp4;
        if (to_padded)
            out[i] = j < Csp ? in[mk * Csp + j] : 0.f;
        else if (j < Csp)
            out[mk * Csp + j] = in[i];
    }
}

// Nearest centroid of every point of sub-space blockIdx.y.  assign[m][p];
// codes (if given) at codes[m * code_sm + p * code_sp].
template <int CSP4>
__global__ void __launch_bounds__(256) kmeans_assign_kernel(const float *__restrict__ pts, int P,
                                                            int K, const float *__restrict__ cen,
                                                            uint8_t *__restrict__ assign,
                                                            uint8_t *__restrict__ codes,
                                                            long long code_sm, long long code_sp) {
    __shared__ __align__(16) float cs[kMaxK * CSP4];
    const int m = blockIdx.y;
    for (int e = threadIdx.x; e < K * CSP4; e += blockDim.x)
        cs[e] = cen[(size_t)m * K * CSP4 + e];
    __syncthreads();
    const int p = blockIdx.x * blockDim.x + threadIdx.x;
    if (p >= P) return;
    float x[CSP4];
    const float4 *xp = reinterpret_cast<const float4 *>(pts + ((size_t)m * P + p) * CSP4);
#pragma unroll
    for (int q = 0; q < CSP4 / 4; ++q) {
        const float4 v = xp[q];
        x[4 * q] = v.x;
        x[4 * q + 1] = v.y;
        x[4 * q + 2] = v.z;
        x[4 * q + 3] = v.w;
    }
    int best = 0;
    float best_d = 0.f;
    for (int k = 0; k < K; ++k) {
        const float *c = cs + k * CSP4;
        float d = 0.f;
#pragma unroll
        for (int j = 0; j < CSP4; ++j) {
            const float diff = __fsub_rn(x[j], c[j]);
            d = __fadd_rn(d, __fmul_rn(diff, diff));
        }
        if (k == 0 || d < best_d) {
            best = k;
            best_d = d;
        }
    }
    assign[(size_t)m * P + p] = (uint8_t)best;
    if (codes) codes[(size_t)m * code_sm + (size_t)p * code_sp] = (uint8_t)best;
}

// One CTA per sub-space: order[m][*] = the sub-space's point indices grouped
// by cluster, index order inside a cluster; starts[m][k] = first slot of
// cluster k (starts[m][K] = P).
__global__ void __launch_bounds__(kSortThreads) kmeans_order_kernel(
    const uint8_t *__restrict__ assign, int P, int K, int *__restrict__ order,
    int *__restrict__ starts) {
    constexpr int NW = kSortThreads / 32;
    __shared__ int wcount[NW][kMaxK];  // per-warp counts of one round, then offsets
    __shared__ int base[kMaxK + 1];    // running start of each cluster
    const int m = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const uint8_t *a = assign + (size_t)m * P;
    // cluster sizes -> exclusive starts
    for (int k = tid; k <= K; k += kSortThreads) base[k] = 0;
    __syncthreads();
    for (int p = tid; p < P; p += kSortThreads) atomicAdd(&base[a[p] + 1], 1);
    __syncthreads();
    if (tid == 0)
        for (int k = 1; k <= K; ++k) base[k] += base[k - 1];
    __syncthreads();
    for (int k = tid; k <= K; k += kSortThreads) starts[(size_t)m * (K + 1) + k] = base[k];
    // stable scatter, kSortThreads points per round
    for (int p0 = 0; p0 < P; p0 += kSortThreads) {
        for (int e = tid; e < NW * K; e += kSortThreads) wcount[e / K][e % K] = 0;
        __syncthreads();
        const int p = p0 + tid;
        const int k = p < P ? a[p] : -1;
        const unsigned same = __match_any_sync(0xffffffffu, k);
        const int rank = __popc(same & ((1u << lane) - 1u));
        if (k >= 0 && rank == 0) wcount[warp][k] = __popc(same);
        __syncthreads();
        for (int c = tid; c < K; c += kSortThreads) {  // offsets over the warps, in order
            int run = base[c];
            for (int w = 0; w < NW; ++w) {
                const int v = wcount[w][c];
                wcount[w][c] = run;
                run += v;
            }
            base[c] = run;
        }
        __syncthreads();
        if (k >= 0) order[(size_t)m * P + wcount[warp][k] + rank] = p;
        __syncthreads();
    }
}

// One thread per (m, k, j): the mean of cluster k's coordinate j, summed in
// double in point-index order; unchanged when the cluster is empty.
__global__ void kmeans_update_kernel(const float *__restrict__ pts, int M, int P, int K,
                                     int Csp, int csp4, const int *__restrict__ order,
                                     const int *__restrict__ starts, float *__restrict__ cen) {
    const int total = M * K * Csp;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
        const int j = i % Csp, mk = i / Csp;
        const int k = mk % K, m = mk / K;
        const int s0 = starts[(size_t)m * (K + 1) + k], s1 = starts[(size_t)m * (K + 1) + k + 1];
        if (s1 == s0) continue;
        const int *ord = order + (size_t)m * P;
        const float *pm = pts + (size_t)m * P * csp4 + j;
        double s = 0.0;
        for (int e = s0; e < s1; ++e) s += (double)__ldg(pm + (size_t)__ldg(ord + e) * csp4);
        cen[(size_t)mk * csp4 + j] = __double2float_rn(s / (double)(s1 - s0));
    }
}

// ------------------------------------------------------------------ host --
struct KmeansWs {
    size_t pts, cen, assign, order, starts, total;
};

KmeansWs kmeans_ws_layout(int M, long long P, int Csp, int K, bool with_points) {
    const int csp4 = Csp <= 4 ? 4 : 8;
    KmeansWs w;
    size_t off = 0;
    w.pts = off;
    if (with_points) off += align_up((size_t)M * P * csp4 * sizeof(float), kWsAlign);
    w.cen = off;
    off += align_up((size_t)M * K * csp4 * sizeof(float), kWsAlign);
    w.assign = off;
    off += align_up((size_t)M * P, kWsAlign);
    w.order = off;
    off += align_up((size_t)M * P * sizeof(int), kWsAlign);
    w.starts = off;
    off += align_up((size_t)M * (K + 1) * sizeof(int), kWsAlign);
    w.total = off;
    return w;
}

qcnn_status run_kmeans(const float *pts, int M, int P, int Csp, int K, const float *init,
                       int iters, float *D, uint8_t *codes, long long code_sm,
                       long long code_sp, void *ws, const KmeansWs &L, cudaStream_t st) {
    const int csp4 = Csp <= 4 ? 4 : 8;
    uint8_t *base = static_cast<uint8_t *>(ws);
    float *cen = reinterpret_cast<float *>(base + L.cen);
    uint8_t *assign = base + L.assign;
    int *order = reinterpret_cast<int *>(base + L.order);
    int *starts = reinterpret_cast<int *>(base + L.starts);
    const int sms = num_sms();
    const int cen_blocks = std::max(1, std::min(cdiv(M * K * csp4, 256), sms * 8));
    pad_centroids_kernel<<<cen_blocks, 256, 0, st>>>(init, M, K, Csp, csp4, cen, 1);
    qcnn_status rc = after_launch();
    if (rc != QCNN_OK) return rc;
    const dim3 agrid(cdiv(P, 256), M);
    const int ublocks = std::max(1, std::min(cdiv(M * K * Csp, 256), sms * 16));
    for (int it = 0; it <= iters; ++it) {
        const bool last = it == iters;
        if (csp4 == 4)
            kmeans_assign_kernel<4><<<agrid, 256, 0, st>>>(pts, P, K, cen, assign,
                                                           last ? codes : nullptr, code_sm,
                                                           code_sp);
        else
            kmeans_assign_kernel<8><<<agrid, 256, 0, st>>>(pts, P, K, cen, assign,
                                                           last ? codes : nullptr, code_sm,
                                                           code_sp);
        if ((rc = after_launch()) != QCNN_OK) return rc;
        if (last) break;
        kmeans_order_kernel<<<M, kSortThreads, 0, st>>>(assign, P, K, order, starts);
        if ((rc = after_launch()) != QCNN_OK) return rc;
        kmeans_update_kernel<<<ublocks, 256, 0, st>>>(pts, M, P, K, Csp, csp4, order, starts,
                                                      cen);
        if ((rc = after_launch()) != QCNN_OK) return rc;
    }
    pad_centroids_kernel<<<cen_blocks, 256, 0, st>>>(cen, M, K, Csp, csp4, D, 0);
    return after_launch();
}

}  // namespace qcnn

using namespace qcnn;

namespace {

bool kmeans_args_ok(int M, long long P, int Csp, int K, int iters) {
    return M > 0 && P > 0 && Csp >= 1 && Csp <= kMaxCsp && K >= 1 && K <= kMaxK &&
           iters >= 0 && (long long)M * P * 8 < (long long)INT_MAX &&
           (long long)M * K * 8 < (long long)INT_MAX;
}

}  // namespace

extern "C" {

qcnn_status qcnn_kmeans_workspace_size(int M, int P, int Csp, int K, size_t *bytes) {
    if (!bytes || !kmeans_args_ok(M, P, Csp, K, 0)) return QCNN_ERR_INVALID_ARG;
    *bytes = kmeans_ws_layout(M, P, Csp, K, true).total;
    return QCNN_OK;
}

qcnn_status qcnn_kmeans(const float *points, int M, int P, int Csp, int K, const float *init,
                        int iters, float *D, uint8_t *assign, void *workspace,
                        size_t workspace_bytes, void *stream) {
    if (!points || !init || !D || !assign || !kmeans_args_ok(M, P, Csp, K, iters))
        return QCNN_ERR_INVALID_ARG;
    const KmeansWs L = kmeans_ws_layout(M, P, Csp, K, true);
    if (!workspace || workspace_bytes < L.total ||
        reinterpret_cast<uintptr_t>(workspace) % kWsAlign != 0)
        return QCNN_ERR_WORKSPACE;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const int csp4 = Csp <= 4 ? 4 : 8;
    float *pts = reinterpret_cast<float *>(static_cast<uint8_t *>(workspace) + L.pts);
    // points [M][P][Csp] -> zero-padded [M][P][csp4] (same pass as for centroids)
    const long long total = (long long)M * P * csp4;
    const int blocks = (int)std::min<long long>((total + 255) / 256, (long long)num_sms() * 16);
    pad_centroids_kernel<<<blocks, 256, 0, st>>>(points, M, P, Csp, csp4, pts, 1);
    qcnn_status rc = after_launch();
    if (rc != QCNN_OK) return rc;
    return run_kmeans(pts, M, P, Csp, K, init, iters, D, assign, P, 1, workspace, L, st);
}

qcnn_status qcnn_pq_quantize_workspace_size(int kind, int Ct, int Cs, int kh, int kw, int Csp,
                                            int K, size_t *bytes) {
    if (!bytes || Ct <= 0 || Cs <= 0 || Csp < 1 || Cs % Csp != 0) return QCNN_ERR_INVALID_ARG;
    if (kind == QCNN_LAYER_FC) kh = kw = 1;
    else if (kind != QCNN_LAYER_CONV || kh <= 0 || kw <= 0) return QCNN_ERR_INVALID_ARG;
    const long long P = (long long)Ct * kh * kw;
    if (P >= INT_MAX || !kmeans_args_ok(Cs / Csp, P, Csp, K, 0)) return QCNN_ERR_INVALID_ARG;
    *bytes = kmeans_ws_layout(Cs / Csp, P, Csp, K, true).total;
    return QCNN_OK;
}

qcnn_status qcnn_pq_quantize(int kind, const float *W, int Ct, int Cs, int kh, int kw, int Csp,
                             int K, const float *init, int iters, float *D, uint8_t *codes,
                             void *workspace, size_t workspace_bytes, void *stream) {
    size_t need = 0;
    qcnn_status rc = qcnn_pq_quantize_workspace_size(kind, Ct, Cs, kh, kw, Csp, K, &need);
    if (rc != QCNN_OK) return rc;
    if (!W || !init || !D || !codes || iters < 0) return QCNN_ERR_INVALID_ARG;
    if (!workspace || workspace_bytes < need ||
        reinterpret_cast<uintptr_t>(workspace) % kWsAlign != 0)
        return QCNN_ERR_WORKSPACE;
    if (kind == QCNN_LAYER_FC) kh = kw = 1;
    const int M = Cs / Csp, kk = kh * kw, csp4 = Csp <= 4 ? 4 : 8;
    const int P = Ct * kk;
    const KmeansWs L = kmeans_ws_layout(M, P, Csp, K, true);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    float *pts = reinterpret_cast<float *>(static_cast<uint8_t *>(workspace) + L.pts);
    const long long total = (long long)M * P * csp4;
    const int blocks = (int)std::min<long long>((total + 255) / 256, (long long)num_sms() * 16);
    pq_points_kernel<<<blocks, 256, 0, st>>>(W, Ct, Cs, kk, Csp, csp4, M, pts);
    rc = after_launch();
    if (rc != QCNN_OK) return rc;
    // codes: FC [M][Ct] (m stride P, p stride 1); conv [Ct][kk][M] (m stride 1, p stride M)
    const long long sm = kind == QCNN_LAYER_FC ? P : 1, sp = kind == QCNN_LAYER_FC ? 1 : M;
    return run_kmeans(pts, M, P, Csp, K, init, iters, D, codes, sm, sp, workspace, L, st);
}

}  // extern "C"
