// measure.cu -- the shared-memory load throughput of the current GPU, the
// denominator of the look-up stage's roofline (every look-up of Eq. 5 / 7
// is a shared-memory load in the fused kernels).
//
// One CTA per SM streams conflict-free loads from a 192 KB shared array
// (lanes of a warp on consecutive 4- or 16-byte words, so every warp
// instruction moves 128 or 512 bytes = 1 or 4 wavefronts of 128 B) for a
// fixed number of rounds; each CTA times itself with clock64() between two
// barriers.  The rate is wavefronts per SM per cycle of the slowest CTA:
// independent of the SM clock, so a GPU at any clock gives the same number.
#include "qcnn_internal.cuh"

namespace qcnn {
namespace {

constexpr int kProbeWarps = 16;
constexpr int kProbeWords = 48 * 1024;  // 192 KB of fp32 words
constexpr int kProbeRounds = 4096;
constexpr int kMaxProbeSms = 1024;

// Cycles of every CTA, and a sink that keeps the loads from being removed.
// Host code reads them with cudaMemcpyFromSymbol after the launch.
__device__ long long g_probe_cycles[kMaxProbeSms];
__device__ float g_probe_sink[kMaxProbeSms];

template <int VEC>
__global__ void __launch_bounds__(kProbeWarps * 32, 1) smem_load_probe_kernel(float sentinel) {
    extern __shared__ __align__(16) float s[];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int e = tid; e < kProbeWords; e += kProbeWarps * 32) s[e] = (float)(e & 255);
    __syncthreads();
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    const long long t0 = clock64();
    for (int r = 0; r < kProbeRounds; ++r) {
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            // row (warp + 8 i + r) mod 256 of 32 * VEC words: in bounds, and
            // 16-byte aligned for VEC == 4
            const int row = (warp + 8 * i + r) & 255;
            const int idx = (row * 32 + lane) * VEC;
            if constexpr (VEC == 1) {
                acc[i] += s[idx];
            } else {
                const float4 v = *reinterpret_cast<const float4 *>(s + idx);
                acc[i] += (v.x + v.y) + (v.z + v.w);
            }
        }
    }
    __syncthreads();
    const long long t1 = clock64();
    float t = 0.f;
    for (int i = 0; i < 8; ++i) t += acc[i];
    if (t == sentinel) g_probe_sink[blockIdx.x] = t;
    if (tid == 0) g_probe_cycles[blockIdx.x] = t1 - t0;
}

}  // namespace
}  // namespace qcnn

using namespace qcnn;

extern "C" qcnn_status qcnn_smem_load_rate(int vec_bytes, double *wavefronts_per_sm_clk,
                                           void *stream) {
    if (!wavefronts_per_sm_clk || (vec_bytes != 4 && vec_bytes != 16)) return QCNN_ERR_INVALID_ARG;
    *wavefronts_per_sm_clk = 0.0;
    const int sms = num_sms();
    if (sms < 1 || sms > kMaxProbeSms) return QCNN_ERR_UNSUPPORTED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    void (*k)(float) = vec_bytes == 16 ? smem_load_probe_kernel<4> : smem_load_probe_kernel<1>;
    const size_t smem = (size_t)kProbeWords * sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_status(e);
    for (int pass = 0; pass < 2; ++pass) {  // the first pass warms up
        k<<<sms, kProbeWarps * 32, smem, st>>>(-1.0f);
        const qcnn_status rc = after_launch();
        if (rc != QCNN_OK) return rc;
    }
    qcnn_status rc = cuda_status(cudaStreamSynchronize(st));
    if (rc != QCNN_OK) return rc;
    long long cyc[kMaxProbeSms];
    rc = cuda_status(cudaMemcpyFromSymbol(cyc, g_probe_cycles, sizeof(long long) * sms));
    if (rc != QCNN_OK) return rc;
    long long worst = 0;
    for (int i = 0; i < sms; ++i) worst = cyc[i] > worst ? cyc[i] : worst;
    if (worst <= 0) return QCNN_ERR_CUDA;
    const double wavefronts =
        (double)kProbeWarps * kProbeRounds * 8 * (vec_bytes == 16 ? 4 : 1);
    *wavefronts_per_sm_clk = wavefronts / (double)worst;
    return QCNN_OK;
}
