// qcnn_internal.cuh -- declarations shared by the translation units of
// libqcnn (never installed; the public interface is include/qcnn.h).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "qcnn.h"  // include/ is on the include path of the build

namespace qcnn {

constexpr int kMaxCsp = 8;        // largest sub-space dimension C'_s served
constexpr int kMaxK = 256;        // codes are uint8
constexpr size_t kWsAlign = 256;  // alignment of every workspace carve-out

inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }
__host__ __device__ inline int cdiv(int a, int b) { return (a + b - 1) / b; }

// Number of SMs of the current device (cached per device).
int num_sms();

// Device-check record of debug builds (QCNN_DEBUG_CHECKS): every translation
// unit keeps its kernels' flags (QCNN_CHECK_* bits of include/qcnn.h) in a
// device word of its own and registers a host function that reads and clears
// it; collect_device_checks() ORs all of them into *flags.  Release builds
// register nothing and collect nothing.
using CheckReader = qcnn_status (*)(unsigned *flags);
void register_check_reader(CheckReader r);
qcnn_status collect_device_checks(unsigned *flags);
// Synchronize `st`, then turn a non-empty device-check record into
// QCNN_ERR_DEVICE_CHECK (debug builds); release builds only synchronize.
qcnn_status sync_and_check(cudaStream_t st);

// Book-keeping of launches and CUDA errors (qcnn_api.cu).
void count_launch();
qcnn_status cuda_status(cudaError_t e);
// Check the launch that was just enqueued and count it.
qcnn_status after_launch();

// Programmatic dependent launch between the kernels of one library call.
// An entry point that launches a chain of kernels opens a PdlScope; inside
// it, the first launch is a plain one (it waits for everything queued before
// it on the stream: the caller's kernels, copies, event waits) and the later
// ones are programmatic: such a kernel may be scheduled while the kernel
// before it is still running, and calls grid_dep_sync() before its first
// access to global memory.  pdl_break() makes the next launch plain again
// (after an event wait in the middle of a call).  Outside a scope every
// launch is plain.
struct PdlScope {
    PdlScope();
    ~PdlScope();
    PdlScope(const PdlScope &) = delete;
    PdlScope &operator=(const PdlScope &) = delete;
    int saved;
};
void pdl_break();
// true when the next launch may be programmatic; marks the launch as done
bool pdl_next_launch();

// Launch a kernel that calls grid_dep_sync() before touching global memory,
// programmatically when the current PdlScope allows it.  Optional cluster
// dimensions (cluster.x > 0).  Counts the launch and checks it.
template <typename... P, typename... A>
qcnn_status launch_k(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                     dim3 cluster, A &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    unsigned n = 0;
    if (pdl_next_launch()) {
        attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    if (cluster.x > 0) {
        attr[n].id = cudaLaunchAttributeClusterDimension;
        attr[n].val.clusterDim.x = cluster.x;
        attr[n].val.clusterDim.y = cluster.y;
        attr[n].val.clusterDim.z = cluster.z;
        ++n;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, static_cast<A &&>(args)...);
    count_launch();
    return cuda_status(e != cudaSuccess ? e : cudaGetLastError());
}
template <typename... P, typename... A>
qcnn_status launch_pdl(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       A &&...args) {
    return launch_k(kernel, grid, block, smem, st, dim3(0, 0, 0), static_cast<A &&>(args)...);
}

// ---------------------------------------------------------------- conv ----
struct ConvShape {
    int N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K, M, Ho, Wo;
    int bf16;  // 1: table entries rounded to bfloat16 (QCNN_LUT_BF16)
};

// Fused plan: one CTA = (image, ST consecutive output positions of the
// padded grid, CT_CTA channels).
struct ConvFusedPlan {
    bool ok = false;
    int variant = -1;   // index into the instantiated kernel table
    int P, CTW, WP;     // slots per warp, channels per warp, warps on positions
    int ST;             // output positions per tile (slots x 32 x positions per lane)
    int pitch;          // halo row pitch, max(W + pad, Wo)
    int KS;             // 32-bit words per table row (per sub-codeword; bf16:
                        // both copies, 2 x an odd word count)
    int HP;             // halo positions built: ST + (kh - 1) * pitch + kw - 1
    int ct_cta;         // channels per CTA
    int pos_tiles, ct_tiles;
    int splits = 1;     // CTAs sharing one tile's sub-spaces (small batches)
    int m_per_split;
    int cl = 1;         // splits form clusters of cl CTAs that add their partial
                        // sums in distributed shared memory; splits / cl
                        // groups are left for the split reduction (1: none)
    int sk = 0;         // stream-K schedule (large batches): sk_ctas persistent
    int sk_ctas = 0;    // CTAs over the (tile, sub-space) units, sk_base each
    int sk_base = 0, sk_extra = 0;  // (+1 for the first sk_extra)
    size_t partial_bytes = 0;  // workspace for split or stream-K partial sums
    size_t smem;        // dynamic shared memory bytes
    double score;       // estimated cost (lower is better)
};

// Clusters of C CTAs of `threads` threads and smem bytes of dynamic shared
// memory that can be resident at once (cudaOccupancyMaxActiveClusters on the
// current device, cached; with no device, the occupancy measured on a
// GB300).  0 when such a cluster cannot be launched.
int cluster_capacity(const void *kernel, int threads, int C, size_t smem);

// force >= 0: only that variant, without the planner's preference gates;
// force_cl: 0 = choose, 1 = no clusters, c > 1 = clusters of c CTAs wherever
// the tile's sub-spaces are split
ConvFusedPlan plan_conv_fused(const ConvShape &s, int force = -1, int force_cl = 0);
int conv_fused_variant_count();
void conv_fused_variant_info(int v, int info[9]);

struct ConvUnfusedPlan {
    int NB;             // images per table chunk
    int HQ, WQ;         // positions per phase (ceil(H/s), ceil(W/s))
    size_t lut_bytes;   // workspace bytes for one chunk of tables
};
ConvUnfusedPlan plan_conv_unfused(const ConvShape &s);

// Chunked plan (conv_chunked.cu): table rows of KC sub-codewords at a time.
struct ConvChunkPlan {
    bool ok = false;
    int variant = -1;
    int g_TH, KC, NCH, ct_cta, row_tiles, ct_tiles;
    size_t smem, entries_bytes, starts_bytes;
    double score;
};
ConvChunkPlan plan_conv_chunked(const ConvShape &s);
qcnn_status launch_conv_chunked(const ConvShape &s, const ConvChunkPlan &p, const float *x,
                                const float *D, const uint8_t *codes, int codes_packed,
                                const float *bias, float *y, int relu, void *ws,
                                cudaStream_t st);

// Stride-phase plan (conv_phase.cu): full table rows of one stride phase of
// a tile at a time, any stride.
struct ConvPhasePlan {
    bool ok = false;
    int variant = -1;
    int pitch, dymin, dxmin, HP, KS, ct_cta, pos_tiles, ct_tiles;
    int ST = 0;                           // output positions per tile
    int splits = 1, units_per_split = 0;  // (sub-space, phase) units per CTA
    int cl = 1;                           // cluster of splits (as ConvFusedPlan)
    size_t partial_bytes = 0;             // workspace for split partial sums
    size_t smem;
    double score;
};
ConvPhasePlan plan_conv_phase(const ConvShape &s, int force_cl = 0);
qcnn_status launch_conv_phase(const ConvShape &s, const ConvPhasePlan &p, const float *x,
                              const float *D, const uint8_t *packed, const float *bias, float *y,
                              int relu, float *partial_ws, cudaStream_t st);

size_t packed_codes_bytes(int Ct, int kk, int M);
int packed_ct(int Ct);   // Ct rounded up to a multiple of 256

qcnn_status launch_pack_codes(const uint8_t *codes, int Ct, int kk, int M, int K,
                              uint8_t *packed, cudaStream_t st);
// y = bias + sum of `splits` partial sums [splits][total] (fixed order), then ReLU
qcnn_status launch_split_reduce(const float *partial, int splits, size_t total, int Ct, int HoWo,
                                const float *bias, int relu, float *y, cudaStream_t st);
// partial_ws: p.partial_bytes of workspace (unused when p.splits == 1)
qcnn_status launch_conv_fused(const ConvShape &s, const ConvFusedPlan &p,
                              const float *x, const float *D,
                              const uint8_t *packed, const float *bias, float *y,
                              int relu, float *partial_ws, cudaStream_t st);
qcnn_status launch_conv_unfused(const ConvShape &s, const ConvUnfusedPlan &p,
                                const float *x, const float *D,
                                const uint8_t *packed, const float *bias,
                                float *y, int relu, float *lut_ws,
                                cudaStream_t st);

// ------------------------------------------------------------------ fc ----
struct FcShape {
    int N, Cs, Ct, Csp, K, M;
    int bf16;       // 1: table entries rounded to bfloat16 (QCNN_LUT_BF16)
    int code_bits;  // 0: codes [M][Ct] bytes; else bit-packed rows (bits.cu)
};

int code_bits(int K);                   // ceil(log2 K), at least 1
size_t fc_packed_pitch(int Ct, int K);  // bytes per packed FC code row
qcnn_status launch_pack_bits(const uint8_t *codes, long long row_len, long long rows,
                             long long in_pitch, long long out_pitch, int b, int K, uint8_t *out,
                             cudaStream_t st);
qcnn_status launch_unpack_bits(const uint8_t *in, long long n, int b, uint8_t *codes,
                               cudaStream_t st);
// Small batches (N <= 8, K <= 32; fc_small.cu): one thread-block cluster of C
// CTAs per output tile, the sub-spaces split over its CTAs, tables in shared
// memory read by warp shuffles, the partial sums added through distributed
// shared memory -- one kernel, no workspace.
struct FcSmallPlan {
    bool ok = false;
    int variant = -1;
    int NB, OPL, ct_cta, tiles, C, m_per, MC, crow;
    size_t smem;
};
FcSmallPlan plan_fc_small(const FcShape &s);
qcnn_status launch_fc_small(const FcShape &s, const FcSmallPlan &p, const float *x,
                            const float *D, const uint8_t *codes, const float *bias, float *y,
                            int relu, cudaStream_t st);

struct FcPlan {
    FcSmallPlan small;  // used instead of the fields below when small.ok
    int variant;        // kernel table index
    int NT, CT_CTA;     // images and outputs per CTA
    int MCH;            // sub-spaces per shared-memory chunk
    int n_chunks;       // ceil(M / MCH)
    int splits;         // CTAs along m (partial sums reduced afterwards)
    int chunks_per_split;
    int n_tiles, ct_tiles;
    size_t smem;
    size_t partial_bytes;  // workspace for split partial sums (0 if splits == 1)
};
// max_partial_bytes: no split count whose partial sums need more is chosen
// (1 split, without partial sums, always fits)
FcPlan plan_fc(const FcShape &s, size_t max_partial_bytes = ~(size_t)0);
// FC forward whose split partial sums live in caller-independent scratch of
// at most max_partial_bytes; get_scratch is asked for its device address
// only when the plan needs it (qcnn_fc_forward_noalloc)
qcnn_status fc_forward_limited(const float *x, int N, int Cs, int Ct, const float *D, int Csp,
                               int K, const uint8_t *codes, const float *bias, float *y,
                               int relu, size_t max_partial_bytes,
                               qcnn_status (*get_scratch)(void **), cudaStream_t st);
qcnn_status launch_fc(const FcShape &s, const FcPlan &p, const float *x,
                      const float *D, const uint8_t *codes, const float *bias,
                      float *y, int relu, float *partial_ws, cudaStream_t st);

// ------------------------------------------------------------ lut, pool ----
// lut: fp32 entries, or bfloat16 bit patterns when bf16 != 0
qcnn_status launch_lut_build(const float *x, int N, int Cs, int P, const float *D,
                             int Csp, int K, void *lut, int bf16, cudaStream_t st);
qcnn_status launch_maxpool(const float *x, int N, int C, int H, int W, int k,
                           int s, float *y, cudaStream_t st);

}  // namespace qcnn

// ----------------------------------------------------------- device side ----
#ifdef __CUDACC__
#include <cooperative_groups.h>
namespace qcnn {

// quantize.cu: one CTA of kSortThreads (1024) threads per label array of P
// entries: order[*] = indices grouped by label, increasing inside a group;
// starts[k] = first slot of label k, starts[K] = P.
__global__ void kmeans_order_kernel(const uint8_t *assign, int P, int K, int *order, int *starts);

// Programmatic dependent launch.  A kernel started by launch_pdl may run
// while the grid before it in the stream finishes; it calls grid_dep_sync()
// before touching global memory.  That waits until every grid this one
// depends on has completed and its writes are visible (a no-op for a kernel
// launched without the attribute), then lets the next kernel of the stream
// be scheduled; a kernel that has passed it has therefore all its inputs.
__device__ __forceinline__ void grid_dep_sync() {
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
}

__device__ __forceinline__ unsigned smem_addr(const void *p) {
    return static_cast<unsigned>(__cvta_generic_to_shared(p));
}

// 4-byte asynchronous global->shared copy; when `pred` is false nothing is
// read and the destination is filled with zeros (src-size 0).
__device__ __forceinline__ void cp_async4(void *dst, const void *src, bool pred) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(smem_addr(dst)),
                 "l"(src), "r"(pred ? 4 : 0)
                 : "memory");
}

// 16-byte asynchronous global->shared copy (both addresses 16-byte aligned).
__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(smem_addr(dst)), "l"(src)
                 : "memory");
}

__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;\n" ::: "memory");
}

template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

// Sum of the partial tiles of the CTAs of a thread-block cluster.  Every CTA
// has left its E partial sums in `red` (its own shared memory, same offset
// in every CTA); after a cluster barrier, CTA r adds elements
// [r*ceil(E/CL), ...) of all CL tiles in rank order -- a fixed order, so the
// result does not depend on the schedule -- and hands each sum to emit(e, v).
// A second barrier keeps every CTA's shared memory alive until all reads are
// done.  Every thread of every CTA of the cluster must call it.
template <typename F>
__device__ __forceinline__ void cluster_tile_reduce(const float *red, int E, F &&emit) {
    cooperative_groups::cluster_group cluster = cooperative_groups::this_cluster();
    cluster.sync();
    const int CL = (int)cluster.num_blocks(), r = (int)cluster.block_rank();
    const int per = (E + CL - 1) / CL;
    const int e1 = min(E, (r + 1) * per);
    for (int e = r * per + (int)threadIdx.x; e < e1; e += (int)blockDim.x) {
        float v = 0.f;
        for (int q = 0; q < CL; ++q) v += cluster.map_shared_rank(red, q)[e];
        emit(e, v);
    }
    cluster.sync();
}

// Byte b (0..3) of w, zero-extended.
__device__ __forceinline__ unsigned byte_of(unsigned w, int b) {
    return __byte_perm(w, 0u, 0x4440u | (unsigned)b);
}

// a += x; b += y with one packed fp32x2 add: two independent IEEE
// round-to-nearest additions, bit-identical to two scalar adds.
__device__ __forceinline__ void add2(float &a, float &b, float x, float y) {
    const float2 r = __fadd2_rn(make_float2(a, b), make_float2(x, y));
    a = r.x;
    b = r.y;
}

// a += low bfloat16 half of w, b += high half: each half widened to fp32
// (exact) and added with one round-to-nearest fp32 addition, bit-identical
// to converting first and adding in fp32.
__device__ __forceinline__ void add_bf16x2(float &a, float &b, unsigned w) {
    unsigned short lo, hi;
    asm("mov.b32 {%0, %1}, %2;" : "=h"(lo), "=h"(hi) : "r"(w));
    asm("add.rn.f32.bf16 %0, %1, %0;" : "+f"(a) : "h"(lo));
    asm("add.rn.f32.bf16 %0, %1, %0;" : "+f"(b) : "h"(hi));
}

// Two fp32 values rounded to bfloat16 (nearest, ties to even) and packed:
// lo in bits 0-15, hi in bits 16-31.
__device__ __forceinline__ unsigned pack_bf16x2(float lo, float hi) {
    unsigned r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// acc[p] += v(p) for p < P, pairing the adds where possible.
template <int P, typename F>
__device__ __forceinline__ void accumulate(float (&acc)[P], F v) {
#pragma unroll
    for (int p = 0; p + 1 < P; p += 2) add2(acc[p], acc[p + 1], v(p), v(p + 1));
    if constexpr (P % 2 == 1) acc[P - 1] += v(P - 1);
}

}  // namespace qcnn

// ------------------------------------------------------- debug-build checks
// QCNN_CHECK(cond, flag): in builds with QCNN_DEBUG_CHECKS, a kernel thread
// that finds `cond` false ORs `flag` into its translation unit's record and
// goes on (the kernels still clamp, so nothing is read out of bounds); the
// host collects the records at the next synchronizing call.  Release builds
// compile it to nothing.
#ifdef QCNN_DEBUG_CHECKS
namespace qcnn {
namespace {
__device__ unsigned g_check_flags;

qcnn_status read_clear_check_flags(unsigned *flags) {
    unsigned v = 0;
    const unsigned zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(&v, g_check_flags, sizeof v);
    if (e == cudaSuccess) e = cudaMemcpyToSymbol(g_check_flags, &zero, sizeof zero);
    *flags |= v;
    return cuda_status(e);
}
struct CheckReaderRegistration {
    CheckReaderRegistration() { register_check_reader(&read_clear_check_flags); }
} g_check_reader_registration;
}  // namespace
}  // namespace qcnn
#define QCNN_CHECK(cond, flag)                                             \
    do {                                                                   \
        if (!(cond)) atomicOr(&qcnn::g_check_flags, (unsigned)(flag));     \
    } while (0)
#else
#define QCNN_CHECK(cond, flag) \
    do {                       \
    } while (0)
#endif
#endif
