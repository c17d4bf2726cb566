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
    int xs_floats;      // floats of one input staging buffer
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
void conv_fused_variant_info(int v, int info[10]);

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
// leave_partials (fused and phase launches): a plan with several partial sums
// per output leaves them in partial_ws, without the reduction launch
qcnn_status launch_conv_phase(const ConvShape &s, const ConvPhasePlan &p, const float *x,
                              const float *D, const uint8_t *packed, const float *bias, float *y,
                              int relu, float *partial_ws, cudaStream_t st, bool early = false,
                              bool leave_partials = false);

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
                              int relu, float *partial_ws, cudaStream_t st,
                              bool early = false, bool leave_partials = false);
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
struct FcPlan {
    int variant;        // kernel table index
    int NT, CT_CTA;     // images and outputs per CTA
    int MCH;            // sub-spaces per shared-memory chunk
    int n_chunks;       // ceil(M / MCH)
    int splits;         // CTAs along m (partial sums reduced afterwards)
    int cl = 1;         // splits form clusters of cl CTAs that add their partial
                        // tiles in distributed shared memory (splits / cl
                        // partial sums per output left for the reduction)
    int chunks_per_split;
    int n_tiles, ct_tiles;
    size_t smem;
    size_t partial_bytes;  // workspace for split partial sums (0 if splits == cl)
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
// The input of a layer as the previous layer's split partial sums (that
// layer launched with leave_partials): [groups][N][Cs] for an FC layer after
// an FC layer, [groups][N][C][H][W] for a max-pool after a conv layer; the
// previous layer's bias and ReLU are applied after adding them.
struct PartialInput {
    const float *part;
    int groups;
    const float *bias;
    int relu;
};
// xin: the input comes as partial sums (x is then unused); leave_partials:
// a plan with several partial sums per output leaves them in partial_ws
// (for the next FC layer) instead of reducing them into y
qcnn_status launch_fc(const FcShape &s, const FcPlan &p, const float *x,
                      const float *D, const uint8_t *codes, const float *bias,
                      float *y, int relu, float *partial_ws, cudaStream_t st,
                      const PartialInput *xin = nullptr, bool leave_partials = false);

// ------------------------------------------------------------ lut, pool ----
// lut: fp32 entries, or bfloat16 bit patterns when bf16 != 0
qcnn_status launch_lut_build(const float *x, int N, int Cs, int P, const float *D,
                             int Csp, int K, void *lut, int bf16, cudaStream_t st);
qcnn_status launch_maxpool(const float *x, int N, int C, int H, int W, int k,
                           int s, float *y, cudaStream_t st);
// The max-pool of a conv output left in partial sums (one CTA per plane,
// staged in shared memory): planes of at most kPoolPlaneMax elements.
constexpr size_t kPoolPlaneMax = 12288;
qcnn_status launch_maxpool_partial(const PartialInput &in, int N, int C, int H, int W, int k,
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
// done.  Every thread of every CTA of the cluster (at most 16 CTAs) must
// call it.
template <typename F>
__device__ __forceinline__ void cluster_tile_reduce(const float *red, int E, F &&emit) {
    cooperative_groups::cluster_group cluster = cooperative_groups::this_cluster();
    cluster.sync();
    const int CL = (int)cluster.num_blocks(), r = (int)cluster.block_rank();
    const int per = (E + CL - 1) / CL;
    const int e1 = min(E, (r + 1) * per);
    for (int e = r * per + (int)threadIdx.x; e < e1; e += (int)blockDim.x) {
        float part[16];  // every rank's partial in flight at once, then added in order
#pragma unroll
        for (int q = 0; q < 16; ++q) part[q] = q < CL ? cluster.map_shared_rank(red, q)[e] : 0.f;
        float v = 0.f;
#pragma unroll
        for (int q = 0; q < 16; ++q)
            if (q < CL) v += part[q];
        emit(e, v);
    }
    cluster.sync();
}

// ------------------------------------------------ tcgen05 (5th-gen tensor core)
// Thin wrappers of the PTX instructions the tensor-core table build uses.

// Tensor memory: one warp allocates ncols (a power of two >= 32) columns of
// the SM's 512 and writes their base address to *dst (shared memory); the
// same warp frees them before the CTA exits.
__device__ __forceinline__ void tmem_alloc(unsigned *dst, unsigned ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(
                     smem_addr(dst)),
                 "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(unsigned taddr, unsigned ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(taddr), "r"(ncols)
                 : "memory");
}

// Shared-memory matrix descriptor of a K-major operand without swizzle: core
// matrices of 8 rows x 16 bytes stored contiguously; lbo = bytes between
// core matrices adjacent along K, sbo = bytes between groups of 8 rows.
__device__ __forceinline__ uint64_t smem_desc_kmajor(const void *p, unsigned lbo, unsigned sbo) {
    uint64_t d = 0;
    d |= (uint64_t)((smem_addr(p) >> 4) & 0x3FFFu);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;  // descriptor version of this architecture
    return d;                // base offset 0, no swizzle
}

// Instruction descriptor of kind::tf32: fp32 accumulator, tf32 A and B,
// both K-major, M x N.
__host__ __device__ constexpr uint32_t idesc_tf32(int M, int N) {
    return (1u << 4)                    // D: fp32
           | (2u << 7) | (2u << 10)     // A, B: tf32
           | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// D[tmem] (+)= A * B, issued by one thread.
__device__ __forceinline__ void mma_tf32(unsigned tmem_d, uint64_t a, uint64_t b, uint32_t idesc,
                                         bool accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(tmem_d),
        "l"(a), "l"(b), "r"(idesc), "r"((unsigned)accumulate)
        : "memory");
}

// The mbarrier at `bar` gets one arrival when every tcgen05.mma this thread
// issued so far has completed.
__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
            smem_addr(bar))
        : "memory");
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, unsigned count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(smem_addr(bar)), "r"(count)
                 : "memory");
}

// Wait until the phase with parity `parity` of the mbarrier has completed,
// polling at most max_polls times; false when it gave up.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, unsigned parity,
                                                  unsigned max_polls) {
    for (unsigned i = 0; i < max_polls; ++i) {
        unsigned done;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}\n"
            : "=r"(done)
            : "r"(smem_addr(bar)), "r"(parity)
            : "memory");
        if (done) return true;
    }
    return false;
}

__device__ __forceinline__ void tc_fence_before_sync() {
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after_sync() {
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
}
// Make this thread's generic-proxy writes to shared memory visible to the
// tensor core (async proxy).
__device__ __forceinline__ void fence_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
}

// 32 consecutive fp32 columns of the warp's TMEM lane quarter: lane i of the
// warp gets row (taddr lane field) + i, columns col .. col + 31.
__device__ __forceinline__ void tmem_ld32(unsigned taddr, float (&v)[32]) {
    unsigned r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, "
        "[%32];\n\t"
        "tcgen05.wait::ld.sync.aligned;\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// fp32 value with the 13 low mantissa bits cleared: exactly representable
// in tf32, so the tensor core reads it unchanged.
__device__ __forceinline__ float tf32_hi(float x) {
    return __uint_as_float(__float_as_uint(x) & 0xFFFFE000u);
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

// ------------------------------------------------------- device check record
// Every translation unit keeps its kernels' flags (QCNN_CHECK_* bits of
// include/qcnn.h) in a device word of its own and registers a host function
// that reads and clears it; qcnn_device_check collects them all.
//  * QCNN_CHECK(cond, flag): only in builds with QCNN_DEBUG_CHECKS, a thread
//    that finds `cond` false ORs `flag` into the record and goes on (the
//    kernels still clamp, so nothing is read out of bounds).  Release builds
//    compile it to nothing.
//  * QCNN_RECORD_IF(cond, flag): in every build (waits that gave up).
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
// Release builds read back only the units whose kernels record in every
// build (they define QCNN_UNIT_RECORDS before including this header): each
// read is a synchronous copy.
#if defined(QCNN_DEBUG_CHECKS) || defined(QCNN_UNIT_RECORDS)
struct CheckReaderRegistration {
    CheckReaderRegistration() { register_check_reader(&read_clear_check_flags); }
} g_check_reader_registration;
#endif
}  // namespace
}  // namespace qcnn
#define QCNN_RECORD_IF(cond, flag)                                         \
    do {                                                                   \
        if (cond) atomicOr(&qcnn::g_check_flags, (unsigned)(flag));        \
    } while (0)
#ifdef QCNN_DEBUG_CHECKS
#define QCNN_CHECK(cond, flag) QCNN_RECORD_IF(!(cond), flag)
#else
#define QCNN_CHECK(cond, flag) \
    do {                       \
    } while (0)
#endif
#endif
