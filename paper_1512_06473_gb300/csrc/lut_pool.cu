// lut_pool.cu -- the stand-alone look-up-table build (Sec. 3.1 / 3.2: the
// tables of inner products pre-computed for every input vector) and the
// max-pool used between the layers of the whole-network stack.
#include "qcnn_internal.cuh"

#include <cuda_bf16.h>

#include <algorithm>

namespace qcnn {

// lut[n][m][p][k] = sum_j x[n][m*Csp + j][p] * D[m][k][j].
// A CTA owns 32 consecutive (m, p) units of one image; its 32*K outputs are
// one contiguous, coalesced stretch of `lut`.  The kernel is bound by the
// table writes (K/Csp entries written per float read).  T = float, or
// __nv_bfloat16 for entries rounded to bfloat16 (nearest, ties to even).
constexpr int kLutUnits = 32;

template <typename T>
__global__ void __launch_bounds__(256) lut_build_kernel(const float *__restrict__ x, int Cs,
                                                        int P, const float *__restrict__ D,
                                                        int Csp, int K, int M,
                                                        T *__restrict__ lut) {
    __shared__ float xs[kLutUnits][kMaxCsp];
    grid_dep_sync();
    const int n = blockIdx.y;
    const long long units = (long long)M * P;
    const long long u0 = (long long)blockIdx.x * kLutUnits;
    for (int e = threadIdx.x; e < kLutUnits * kMaxCsp; e += blockDim.x) {
        const int ul = e / kMaxCsp, j = e % kMaxCsp;
        const long long u = u0 + ul;
        float v = 0.f;
        if (u < units && j < Csp) {
            const int m = (int)(u / P), p = (int)(u % P);
            v = x[((size_t)n * Cs + (size_t)m * Csp + j) * P + p];
        }
        xs[ul][j] = v;
    }
    __syncthreads();
    const int nu = (int)std::min<long long>(kLutUnits, units - u0);
    T *out = lut + ((size_t)n * units + u0) * K;
    for (int e = threadIdx.x; e < nu * K; e += blockDim.x) {
        const int ul = e / K, k = e % K;
        const int m = (int)((u0 + ul) / P);
        const float *dk = D + ((size_t)m * K + k) * Csp;
        float v = 0.f;
        for (int j = 0; j < Csp; ++j) v = fmaf(xs[ul][j], __ldg(dk + j), v);
        if constexpr (sizeof(T) == 2) out[e] = __float2bfloat16_rn(v);
        else out[e] = v;
    }
}

qcnn_status launch_lut_build(const float *x, int N, int Cs, int P, const float *D, int Csp,
                             int K, void *lut, int bf16, cudaStream_t st) {
    const int M = Cs / Csp;
    const long long units = (long long)M * P;
    dim3 grid((unsigned)((units + kLutUnits - 1) / kLutUnits), N);
    if (bf16)
        return launch_pdl(lut_build_kernel<__nv_bfloat16>, grid, dim3(256), 0, st, x, Cs, P, D,
                          Csp, K, M, static_cast<__nv_bfloat16 *>(lut));
    return launch_pdl(lut_build_kernel<float>, grid, dim3(256), 0, st, x, Cs, P, D, Csp, K, M,
                      static_cast<float *>(lut));
}

// k x k max-pool, stride s, no padding: one thread per output element.
// One thread per output, 32-bit index arithmetic (every element count is
// below 2^31); neighbouring windows share their overlap through L1.  x is
// usually the output of the kernel just before, so it is read with plain
// (coherent) loads.
__global__ void maxpool_kernel(const float *x, int total, int H, int W, int k, int s, int Ho,
                               int Wo, float *__restrict__ y) {
    grid_dep_sync();
    const int HoWo = Ho * Wo;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
        const int nc = i / HoWo, o = i - nc * HoWo;
        const int oy = o / Wo, ox = o - oy * Wo;
        const float *p = x + (size_t)nc * H * W + oy * s * W + ox * s;
        float v = p[0];
        for (int dy = 0; dy < k; ++dy)
            for (int dx = 0; dx < k; ++dx) v = fmaxf(v, p[dy * W + dx]);
        y[i] = v;
    }
}

qcnn_status launch_maxpool(const float *x, int N, int C, int H, int W, int k, int s, float *y,
                           cudaStream_t st) {
    const int Ho = (H - k) / s + 1, Wo = (W - k) / s + 1;
    const int total = N * C * Ho * Wo;
    const int blocks = std::max(1, std::min((total + 255) / 256, num_sms() * 8));
    return launch_pdl(maxpool_kernel, dim3(blocks), dim3(256), 0, st, x, total, H, W, k, s, Ho, Wo,
                      y);
}

// The same max-pool of a conv layer's output that is still in its split
// partial sums [groups][N][C][H][W] (Eq. 7 summed over sub-space ranges): one
// CTA per (n, c) plane first forms each element once -- the groups added in
// order from zero, then the bias, then ReLU, the arithmetic of
// conv_split_reduce_kernel, so the result is bit-identical to reducing and
// pooling in two launches -- into shared memory, where the windows read it.
__global__ void maxpool_partial_kernel(const float *part, int groups, size_t total, int C, int H,
                                       int W, int k, int s, int Ho, int Wo,
                                       const float *__restrict__ bias, int relu,
                                       float *__restrict__ y) {
    extern __shared__ float plane[];
    grid_dep_sync();
    const int HW = H * W;
    const size_t nc = blockIdx.x;
    const float *p = part + nc * HW;
    for (int e = threadIdx.x; e < HW; e += blockDim.x) {
        float v = 0.f;
#pragma unroll 16
        for (int g = 0; g < groups; ++g) v += p[(size_t)g * total + e];
        if (bias) v += bias[nc % C];
        if (relu) v = fmaxf(v, 0.f);
        plane[e] = v;
    }
    __syncthreads();
    for (int o = threadIdx.x; o < Ho * Wo; o += blockDim.x) {
        const int oy = o / Wo, ox = o - oy * Wo;
        const float *q = plane + oy * s * W + ox * s;
        float v = q[0];
        for (int dy = 0; dy < k; ++dy)
            for (int dx = 0; dx < k; ++dx) v = fmaxf(v, q[dy * W + dx]);
        y[nc * Ho * Wo + o] = v;
    }
}

qcnn_status launch_maxpool_partial(const PartialInput &in, int N, int C, int H, int W, int k,
                                   int s, float *y, cudaStream_t st) {
    if ((size_t)H * W > kPoolPlaneMax || in.groups < 1) return QCNN_ERR_UNSUPPORTED;
    const int Ho = (H - k) / s + 1, Wo = (W - k) / s + 1;
    const size_t total = (size_t)N * C * H * W;
    return launch_pdl(maxpool_partial_kernel, dim3((unsigned)(N * C)), dim3(256),
                      (size_t)H * W * sizeof(float), st, in.part, in.groups, total, C, H, W, k, s,
                      Ho, Wo, in.bias, in.relu, y);
}

}  // namespace qcnn
