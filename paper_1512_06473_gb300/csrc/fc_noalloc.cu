// fc_noalloc.cu -- qcnn_fc_forward_noalloc: the FC layer response of
// qcnn_fc_forward for callers that cannot give the library any device
// memory.  Such callers exist: a plugin invoked inside another runtime's
// execution step, where that runtime owns all device memory and forbids new
// allocations, or a thin foreign-function caller with no device allocator
// of its own.  qcnn_fc_forward needs a workspace for the partial sums of a
// split sub-space range; here that scratch is a fixed array compiled into
// the library instead.
//
// The array lives in device memory of every GPU that loads the library,
// for as long as the process runs.  All calls share it and it keeps the
// last call's contents; every element a call reads back is written earlier
// in the same call, so nothing has to be cleared between calls.  Calls that
// overlap on the GPU (other streams, other host threads) race on it.
#include "qcnn_internal.cuh"

#include <mutex>

namespace {

constexpr size_t kScratchBytes = QCNN_FC_NOALLOC_SCRATCH_BYTES;
static_assert(kScratchBytes % 256 == 0, "scratch size must keep 256-byte alignment");

// Split partial sums [splits][N][Ct] of the FC kernel.  In host code this
// name is only a stand-in for the device symbol: its device address comes
// from cudaGetSymbolAddress below.
static __device__ __align__(256) float g_fc_scratch[kScratchBytes / sizeof(float)];

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
void *g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device; looked up once
// per device (the first call on each device does it).
qcnn_status scratch_address(void **out) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return qcnn::cuda_status(e);
    if (dev < 0 || dev >= kMaxDevices) return QCNN_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!g_scratch_addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_fc_scratch);
        if (e != cudaSuccess || !p) return qcnn::cuda_status(e != cudaSuccess ? e : cudaErrorInvalidSymbol);
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return QCNN_OK;
}

}  // namespace

extern "C" qcnn_status qcnn_fc_forward_noalloc(const float *x, int N, int Cs, int Ct,
                                               const float *D, int Csp, int K,
                                               const uint8_t *codes, const float *bias,
                                               float *y, int relu, void *stream) {
    size_t need = 0;
    qcnn_status rc = qcnn_fc_workspace_size(N, Cs, Ct, Csp, K, QCNN_LUT_FP32, &need);
    if (rc != QCNN_OK) return rc;
    if (!x || !D || !codes || !y) return QCNN_ERR_INVALID_ARG;
    if (need > kScratchBytes) return QCNN_ERR_WORKSPACE;  // larger than the fixed scratch
    void *scratch = nullptr;
    if (need > 0) {
        rc = scratch_address(&scratch);
        if (rc != QCNN_OK) return rc;
    }
    return qcnn_fc_forward(x, N, Cs, Ct, D, Csp, K, codes, bias, y, relu, QCNN_LUT_FP32, scratch,
                           need, stream);
}
