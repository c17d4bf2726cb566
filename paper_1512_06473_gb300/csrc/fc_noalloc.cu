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

// The plan is qcnn_fc_forward's, except that split counts whose partial sums
// would not fit the fixed scratch are not used (one split needs none).
extern "C" qcnn_status qcnn_fc_forward_noalloc(const float *x, int N, int Cs, int Ct,
                                               const float *D, int Csp, int K,
                                               const uint8_t *codes, const float *bias,
                                               float *y, int relu, void *stream) {
    return qcnn::fc_forward_limited(x, N, Cs, Ct, D, Csp, K, codes, bias, y, relu, kScratchBytes,
                                    scratch_address, reinterpret_cast<cudaStream_t>(stream));
}
