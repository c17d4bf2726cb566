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

#include <cuda.h>

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
struct ScratchAddr {
    void *addr = nullptr;
    unsigned long long ctx_id = 0;  // context the address belongs to
};
ScratchAddr g_scratch[kMaxDevices];

// Unique id of the calling thread's current CUDA context (cuCtxGetId), or 0
// when there is none or it cannot be had.  The driver functions are reached
// through the runtime's entry-point query, so the library needs no link to
// the driver library.  A device's primary context that is destroyed
// (cudaDeviceReset) and created again gets a new id, and with it the module
// holding the scratch array is loaded again at another address.
unsigned long long current_context_id() {
    using GetCurrent = CUresult (*)(CUcontext *);
    using GetId = CUresult (*)(CUcontext, unsigned long long *);
    static GetCurrent get_current = nullptr;
    static GetId get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<GetCurrent>(f);
        f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<GetId>(f);
        cudaGetLastError();
    });
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx ||
        get_id(ctx, &id) != CUDA_SUCCESS)
        return 0;
    return id;
}

// Device address of the scratch array in the current context.  It is
// looked up (cudaGetSymbolAddress) on the first call on each device and
// again whenever that device's context has changed since (or its id is
// unavailable); otherwise the cached address is used.
qcnn_status scratch_address(void **out) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return qcnn::cuda_status(e);
    if (dev < 0 || dev >= kMaxDevices) return QCNN_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_mutex);
    ScratchAddr &c = g_scratch[dev];
    const unsigned long long id = current_context_id();
    if (!c.addr || id == 0 || id != c.ctx_id) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_fc_scratch);
        if (e != cudaSuccess || !p) return qcnn::cuda_status(e != cudaSuccess ? e : cudaErrorInvalidSymbol);
        c.addr = p;
        c.ctx_id = current_context_id();  // the lookup may have created the context
    }
    *out = c.addr;
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
