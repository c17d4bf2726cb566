/*
 * qcnn.h -- C ABI of libqcnn, the GB300 (sm_103a) implementation of the
 * test-phase response of product-quantized (PQ) layers from
 *   J. Wu, C. Leng, Y. Wang, Q. Hu, J. Cheng, "Quantized Convolutional Neural
 *   Networks for Mobile Devices", arXiv 1512.06473 (Q-CNN).
 *
 * The method (Sec. 3.1-3.2): split the C_s input channels into M contiguous
 * sub-spaces of C'_s channels (Csp); for every input vector S^(m) and every
 * sub-codeword D^(m)_k compute the table entry <S^(m), D^(m)_k>; then every
 * output is a sum of table entries selected by stored uint8 indices
 * k_m(c_t) (FC, Eq. 5) or k_m(c_t, p_k) (conv, Eq. 7), plus a bias.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Tensors are caller-owned DEVICE pointers (cudaMalloc / torch memory),
 *    fp32 unless stated, dense and row-major in the order written in each
 *    comment ("[N][C][H][W]" = NCHW).  The only host pointers are the layer
 *    array of qcnn_net_* and the x/y buffers of qcnn_net_forward_host.
 *  - Sub-codebooks: D[m][k][j], m < M = Cs / Csp, k < K, j < Csp
 *    (the k-th column of D^(m) in the paper is row k here).
 *  - `stream` is a cudaStream_t (NULL = the legacy default stream).  Every
 *    call only enqueues work on it and returns; results are ready when the
 *    stream reaches that point.  Exception: qcnn_net_forward_host, which
 *    synchronizes the stream before returning.
 *  - Scratch memory comes from a caller-provided device workspace whose size
 *    is given by the matching *_workspace_size query.  No call allocates or
 *    frees device memory.  The workspace may be reused by the next call on
 *    the same stream; calls that run concurrently need separate workspaces.
 *  - Limits: 1 <= Csp <= 8, 1 <= K <= 256, Cs % Csp == 0, every size > 0 and
 *    every element count below 2^31.  Outside them: QCNN_ERR_INVALID_ARG,
 *    returned before any work is enqueued.
 *  - Alignment: fp32 arrays 4-byte aligned, bfloat16 tables 2-byte aligned,
 *    PACKED code arrays (conv QCNN_CODES_PACKED, and FC rows from
 *    qcnn_fc_pack_codes) 16-byte aligned; workspaces 256-byte aligned.  A
 *    misaligned array gives QCNN_ERR_INVALID_ARG (a misaligned workspace
 *    QCNN_ERR_WORKSPACE) before any work is enqueued.
 *  - Codes >= K are a caller error.  Kernels clamp every index into [0, K),
 *    so such codes never cause an out-of-bounds access, but the outputs are
 *    then unspecified.
 *  - Inputs (x, D, codes, bias) must not overlap the outputs or the
 *    workspace, and must not change while the call runs: inside one call the
 *    kernels after the first may read D and the codes before the kernel
 *    before them has finished (programmatic dependent launch).
 *  - A failed launch returns QCNN_ERR_CUDA; the CUDA error is in
 *    qcnn_last_cuda_error().  The library is stateless apart from that
 *    value, a launch counter, a cache of qcnn_net_* plans (keyed by device,
 *    batch, input shape and the layers' shapes and options) and, per device,
 *    the copy stream and events of qcnn_net_forward_host (created on its
 *    first call), and is safe to call from several threads.
 */
#ifndef QCNN_H
#define QCNN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    QCNN_OK = 0,
    QCNN_ERR_INVALID_ARG = 1, /* bad size, null pointer, limit exceeded     */
    QCNN_ERR_UNSUPPORTED = 2, /* valid request this build cannot serve      */
    QCNN_ERR_WORKSPACE = 3,   /* workspace smaller than the query asked for */
    QCNN_ERR_CUDA = 4,        /* a CUDA call or kernel launch failed        */
    QCNN_ERR_DATA = 5,        /* input data unusable (rank-deficient
                                 calibration set of qcnn_ec_quantize_fc)    */
    QCNN_ERR_DEVICE_CHECK = 6 /* debug builds: a kernel found a code >= K or
                                 an index outside its arrays (see
                                 qcnn_device_check)                         */
} qcnn_status;

typedef enum {
    QCNN_ALGO_AUTO = 0,    /* library picks: fused (stride 1), else phase,
                              else chunked, else unfused                     */
    QCNN_ALGO_FUSED = 1,   /* full table rows of a tile of output positions in
                              shared memory, stride 1 only                   */
    QCNN_ALGO_UNFUSED = 2, /* tables materialised in the workspace first      */
    QCNN_ALGO_CHUNKED = 3, /* table rows built KC sub-codewords at a time in
                              shared memory, any stride                      */
    QCNN_ALGO_PHASE = 4,   /* full table rows of one stride phase of a tile
                              at a time in shared memory, any stride (fp32
                              tables)                                        */
    QCNN_ALGO_NO_CLUSTER = 1 << 16, /* flag, OR-ed into any of the above:
                              split sub-space ranges never form thread-block
                              clusters (their partial sums all go through
                              the workspace and a reduction kernel); for
                              tests and tuning                              */
    QCNN_ALGO_FUSED_VARIANT = 256 /* + v: the fused kernel's tile variant v
                              (0 <= v < qcnn_conv_fused_variant_count()),
                              bypassing the planner's choice; for tests and
                              tuning.  QCNN_ERR_UNSUPPORTED when variant v
                              cannot serve the shape (stride, C'_s width,
                              table type, shared memory; a stream-K variant
                              also needs at least as many tiles as CTA
                              slots)                                       */
} qcnn_algo;

/*
 * The fused conv kernel's instantiated tile variants.  info receives
 * {P, CTW, WP, CSP4, NW, MINB, PIPE, BF, SK, TC}: 32-position slots per warp,
 * output channels per warp, warps along positions, C'_s register width (4
 * or 8), warps per CTA, CTAs per SM the registers are sized for, two table
 * buffers (1/0), bfloat16 tables (1/0), stream-K schedule (1/0), table build
 * on the tensor cores (1/0: tcgen05.mma kind::tf32 with the 3xTF32 split,
 * for 4 < C'_s <= 8 and K a multiple of 32).
 * QCNN_ERR_INVALID_ARG for v out of range or a NULL info.
 */
int qcnn_conv_fused_variant_count(void);
qcnn_status qcnn_conv_fused_variant_info(int v, int info[10]);

/*
 * Precision of the look-up-table entries.  FP32: each entry is the fp32 dot
 * product of Sec. 3.1 / 3.2.  BF16: each entry is that fp32 value rounded to
 * bfloat16 (round to nearest, ties to even), which halves the shared-memory
 * bytes of every look-up; the sums of Eq. 5 / Eq. 7 are still accumulated
 * in fp32.  The paper's tables are full precision; BF16 is an option of
 * this library (expected relative error around 1e-3 of the output range).
 */
typedef enum {
    QCNN_LUT_FP32 = 0,
    QCNN_LUT_BF16 = 1
} qcnn_lut_type;

typedef enum {
    QCNN_CODES_CANONICAL = 0, /* conv codes [Ct][kh*kw][M]                   */
    QCNN_CODES_PACKED = 1     /* output of qcnn_conv_pack_codes              */
} qcnn_codes_layout;

/* Human-readable name of a status value (static string, never NULL). */
const char *qcnn_status_string(qcnn_status s);

/* The last CUDA error code seen by a failing call in this process (0 if none). */
int qcnn_last_cuda_error(void);

/* Number of kernels this library has launched in this process so far. */
uint64_t qcnn_launch_count(void);

/*
 * qcnn_smem_load_rate -- the shared-memory load throughput of the current
 * GPU, in 128-byte wavefronts per SM per clock cycle: the peak of the
 * look-up stage's roofline (each look-up of Eq. 5 / Eq. 7 is one
 * shared-memory load in the fused kernels; Table 1 counts them).  One CTA
 * per SM streams conflict-free loads of vec_bytes (4 or 16) per lane from
 * shared memory and times itself with the SM's cycle counter; the rate of
 * the slowest CTA is returned, independent of the clock it ran at.
 * Synchronizes `stream`.  Allocates nothing (its per-SM cycle counts live
 * in a small array compiled into the library).  QCNN_ERR_INVALID_ARG for
 * another vec_bytes or a NULL result pointer.
 */
qcnn_status qcnn_smem_load_rate(int vec_bytes, double *wavefronts_per_sm_clk, void *stream);

/*
 * Device checks.  The library can be built with QCNN_DEBUG_CHECKS
 * (libqcnn_debug.so); its kernels then test, as they run, what the release
 * kernels only clamp:
 *   QCNN_CHECK_CODE    a code >= K was read (the codes k_m(c_t) of Eq. 5 and
 *                      k_m(c_t, p_k) of Eq. 7 index K sub-codewords);
 *   QCNN_CHECK_TABLE   a look-up-table read in shared memory fell outside
 *                      the table the kernel built;
 *   QCNN_CHECK_GLOBAL  a device-memory access fell outside its array.
 * In every build a kernel also records
 *   QCNN_CHECK_TIMEOUT a bounded wait gave up (the tensor cores did not
 *                      signal the completion of a table build in time); the
 *                      kernel went on, so its outputs are unspecified.
 * A kernel that finds one ORs its bit into a device record and carries on
 * (with the clamped value), so nothing faults or hangs.  The record is read,
 * and cleared, at the next synchronizing call: qcnn_device_check below, and
 * the calls that synchronize their stream anyway (qcnn_net_forward_host,
 * qcnn_ec_quantize_fc, qcnn_ec_quantize_conv, qcnn_model_upload), which then
 * return QCNN_ERR_DEVICE_CHECK instead of QCNN_OK.
 *
 * qcnn_debug_checks: 1 in a debug build, 0 in a release build.
 * qcnn_device_check: synchronizes `stream`; returns QCNN_ERR_DEVICE_CHECK
 *   when the record holds any bit (stored in *flags when flags is not NULL),
 *   and clears it.  The record is per process and device-wide: work on
 *   other streams since the last check is included.
 */
#define QCNN_CHECK_CODE 1u
#define QCNN_CHECK_TABLE 2u
#define QCNN_CHECK_GLOBAL 4u
#define QCNN_CHECK_TIMEOUT 8u
int qcnn_debug_checks(void);
qcnn_status qcnn_device_check(void *stream, unsigned *flags);

/*
 * qcnn_lut_build -- the look-up tables alone (Sec. 3.1, the paragraph after
 * Eq. 5; Sec. 3.2, the paragraph after Eq. 7):
 *     lut[n][m][p][k] = sum_{j < Csp} x[n][m*Csp + j][p] * D[m][k][j]
 * for every input position p = y*W + x (H = W = 1 for an FC input).
 *   x    [N][Cs][H][W]   fp32, device
 *   D    [M][K][Csp]     fp32, device
 *   lut  [N][M][H*W][K]  device, written: fp32 (lut_type QCNN_LUT_FP32) or
 *                        the bit patterns of bfloat16 values, 2 bytes each
 *                        (QCNN_LUT_BF16)
 */
qcnn_status qcnn_lut_build(const float *x, int N, int Cs, int H, int W,
                           const float *D, int Csp, int K, void *lut,
                           int lut_type, void *stream);

/*
 * qcnn_fc_forward -- PQ fully-connected layer, Eq. 5:
 *     y[n][ct] = bias[ct] + sum_{m < M} lut_n[m][codes[m][ct]]    (then ReLU if relu)
 * with lut_n the tables of x[n].  Tables are built tile by tile in shared
 * memory and never written to device memory.
 *   x      [N][Cs]   fp32       D [M][K][Csp] fp32
 *   codes  [M][Ct]   uint8      bias [Ct] fp32, or NULL for none
 *   y      [N][Ct]   fp32, written
 *   lut_type: qcnn_lut_type of the table entries
 *   workspace: at least qcnn_fc_workspace_size(...) bytes, 256-byte aligned
 *   (may be NULL when that size is 0).
 */
qcnn_status qcnn_fc_workspace_size(int N, int Cs, int Ct, int Csp, int K,
                                   int lut_type, size_t *bytes);
qcnn_status qcnn_fc_forward(const float *x, int N, int Cs, int Ct,
                            const float *D, int Csp, int K,
                            const uint8_t *codes, const float *bias, float *y,
                            int relu, int lut_type, void *workspace,
                            size_t workspace_bytes, void *stream);

/*
 * qcnn_fc_plan_info -- the plan qcnn_fc_forward (and qcnn_fc_forward_packed)
 * would run, worked out on the host.  info receives: [0] images per CTA,
 * [1] outputs per CTA, [2] CTAs sharing the sub-spaces of one tile (1: no
 * partial sums), [3] sub-spaces per shared-memory chunk, [4] CTAs of the
 * main kernel, [5] CTAs per thread-block cluster among those of [2] (1:
 * none).  A cluster adds its CTAs' partial sums in distributed shared
 * memory; only [2] / [5] partial sums per output go through the workspace
 * (none, and no second kernel, when [5] == [2]).
 * QCNN_ERR_INVALID_ARG as qcnn_fc_workspace_size, or for a NULL info.
 */
qcnn_status qcnn_fc_plan_info(int N, int Cs, int Ct, int Csp, int K,
                              int lut_type, int info[6]);

/*
 * Bit-packed codes: the storage model of Table 1 (Sec. 3.4), each code in
 * b = qcnn_code_bits(K) = ceil(log2 K) bits (at least 1).  Stream layout:
 * code i occupies stream bits [i*b, (i+1)*b), its bit t at stream bit
 * i*b + t; stream bit s is bit (s mod 8) of byte s / 8.
 *   qcnn_pack_bits / qcnn_unpack_bits: n codes <-> ceil(n*b/8) stream
 *     bytes (device buffers; packing clamps codes to 2^b - 1).
 *   qcnn_fc_pack_codes: FC codes [M][Ct] -> M rows, each packed on its own
 *     and zero-padded to a 16-byte pitch (qcnn_fc_packed_codes_bytes in
 *     all); codes >= K are clamped to K - 1.
 *   qcnn_fc_forward_packed: qcnn_fc_forward reading those rows (16-byte
 *     aligned), same result, 8/b times fewer code bytes; the workspace is
 *     the one qcnn_fc_workspace_size gives.  In a qcnn_layer, an FC layer
 *     with codes_layout QCNN_CODES_PACKED takes them too.
 */
int qcnn_code_bits(int K);
qcnn_status qcnn_pack_bits(const uint8_t *codes, long long n, int bits, uint8_t *stream,
                           void *cuda_stream);
qcnn_status qcnn_unpack_bits(const uint8_t *stream, long long n, int bits, uint8_t *codes,
                             void *cuda_stream);
size_t qcnn_fc_packed_codes_bytes(int M, int Ct, int K);
qcnn_status qcnn_fc_pack_codes(const uint8_t *codes, int M, int Ct, int K, uint8_t *packed,
                               void *stream);
qcnn_status qcnn_fc_forward_packed(const float *x, int N, int Cs, int Ct, const float *D,
                                   int Csp, int K, const uint8_t *packed, const float *bias,
                                   float *y, int relu, int lut_type, void *workspace,
                                   size_t workspace_bytes, void *stream);

/*
 * qcnn_fc_forward_noalloc -- the FC response of qcnn_fc_forward, for callers
 * that cannot hand the library any device memory: code running inside
 * another runtime's execution step, where that runtime owns all device
 * memory and forbids allocation, or a foreign-function caller with no device
 * allocator.  The paper has no counterpart; it is a deployment convenience.
 *   Scratch: a fixed array of QCNN_FC_NOALLOC_SCRATCH_BYTES compiled into
 *   the library, held in the memory of every GPU that loads it until the
 *   process exits.  The call allocates nothing.  The first call on each
 *   device looks up the array's device address (cudaGetSymbolAddress), so
 *   make that first call before any stream capture.  The address is kept
 *   per device together with the id of the CUDA context it belongs to; if
 *   that context is replaced (cudaDeviceReset, or any teardown of the
 *   primary context), the next call looks it up again, and that call too
 *   must then come before any stream capture.
 *   Plan: that of qcnn_fc_forward, except that no split count is used
 *   whose partial sums would exceed QCNN_FC_NOALLOC_SCRATCH_BYTES (one
 *   split needs none), so every size runs; where qcnn_fc_forward would
 *   split further, this call is slower and its sums are added in another
 *   order (a difference within fp32 rounding; identical plans give
 *   bit-identical results).
 *   All calls share the array: calls that overlap on the GPU (different
 *   streams or host threads without ordering) race and give wrong results.
 *   Nothing in it needs clearing: each call writes what it reads back.
 * Arguments, layouts and other errors are those of qcnn_fc_forward with
 * lut_type QCNN_LUT_FP32.
 */
#define QCNN_FC_NOALLOC_SCRATCH_BYTES (16u << 20)
qcnn_status qcnn_fc_forward_noalloc(const float *x, int N, int Cs, int Ct,
                                    const float *D, int Csp, int K,
                                    const uint8_t *codes, const float *bias,
                                    float *y, int relu, void *stream);

/*
 * qcnn_conv_pack_codes -- re-layout conv codes once, at model-load time,
 * for the fused kernels: packed[m][pk][ct] (ct padded with code 0 to a
 * multiple of 256), every code clamped into [0, K).
 *   codes  [Ct][kh*kw][M] uint8, device;  packed: qcnn_conv_packed_codes_bytes
 */
size_t qcnn_conv_packed_codes_bytes(int Ct, int kh, int kw, int M);
qcnn_status qcnn_conv_pack_codes(const uint8_t *codes, int Ct, int kh, int kw,
                                 int M, int K, uint8_t *packed, void *stream);

/*
 * qcnn_conv_forward -- PQ convolutional layer, Eq. 7:
 *     y[n][ct][oy][ox] = bias[ct] + sum_{ky<kh, kx<kw} sum_{m<M}
 *                        lut_n[m][iy*W + ix][codes[ct][ky*kw + kx][m]]
 * with iy = oy*stride - pad + ky, ix = ox*stride - pad + kx; a position
 * outside the map contributes 0 (zero padding); then ReLU if relu.
 * Output size Ho = (H + 2 pad - kh) / stride + 1 (floor), same for Wo.
 *   x      [N][Cs][H][W]   fp32         D [M][K][Csp] fp32
 *   codes  [Ct][kh*kw][M]  uint8 (codes_layout CANONICAL) or the output of
 *          qcnn_conv_pack_codes (PACKED)
 *   bias   [Ct] or NULL;   y [N][Ct][Ho][Wo] fp32, written
 *   algo:  QCNN_ALGO_FUSED (and QCNN_ALGO_FUSED_VARIANT + v) needs stride
 *          1, else QCNN_ERR_UNSUPPORTED.
 *   lut_type: qcnn_lut_type of the table entries; QCNN_LUT_BF16 is served
 *          by the fused and chunked algorithms (UNFUSED returns
 *          QCNN_ERR_UNSUPPORTED).
 *   workspace: at least qcnn_conv_workspace_size(...) bytes, 256-byte aligned.
 */
qcnn_status qcnn_conv_workspace_size(int N, int Cs, int H, int W, int Ct,
                                     int kh, int kw, int stride, int pad,
                                     int Csp, int K, int codes_layout,
                                     int algo, int lut_type, size_t *bytes);
qcnn_status qcnn_conv_forward(const float *x, int N, int Cs, int H, int W,
                              int Ct, int kh, int kw, int stride, int pad,
                              const float *D, int Csp, int K,
                              const uint8_t *codes, int codes_layout,
                              const float *bias, float *y, int relu, int algo,
                              int lut_type, void *workspace,
                              size_t workspace_bytes, void *stream);

/*
 * qcnn_conv_plan_info -- the launch plan qcnn_conv_forward would run for
 * these arguments, worked out on the host like every plan (no work is
 * enqueued and no device memory is touched).  It is for tests, tuning and
 * logs.  info receives:
 *   [0] the algorithm run: QCNN_ALGO_FUSED, _PHASE, _CHUNKED or _UNFUSED;
 *   [1] its kernel variant (FUSED: the index of
 *       qcnn_conv_fused_variant_info), -1 for UNFUSED;
 *   [2] output positions per tile (FUSED, PHASE; else 0);
 *   [3] output channels per CTA (0 for UNFUSED);
 *   [4] CTAs sharing the sub-spaces of one tile (1: no partial sums);
 *   [5] 1 when the FUSED kernel runs the stream-K schedule, else 0;
 *   [6] CTAs of the main kernel (0 for UNFUSED);
 *   [7] CTAs per thread-block cluster among those of [4]: they add their
 *       partial sums in distributed shared memory, so only [4] / [7] partial
 *       sums per output go through the workspace (none, and no second
 *       kernel, when [7] == [4]); 1 for no cluster.
 * Errors are those of qcnn_conv_workspace_size, plus QCNN_ERR_INVALID_ARG
 * for a NULL info.
 */
qcnn_status qcnn_conv_plan_info(int N, int Cs, int H, int W, int Ct, int kh,
                                int kw, int stride, int pad, int Csp, int K,
                                int codes_layout, int algo, int lut_type,
                                int info[8]);

/*
 * qcnn_maxpool -- k x k max-pool, stride s, no padding, floor output size
 * (the pooling between the layers of the whole-network experiments,
 * Sec. 4.2.3).  x [N][C][H][W] -> y [N][C][Ho][Wo], Ho = (H - k) / s + 1.
 */
qcnn_status qcnn_maxpool(const float *x, int N, int C, int H, int W, int k,
                         int s, float *y, void *stream);

/*
 * Whole network: a stack of PQ conv / PQ FC / max-pool layers (Sec. 4.2.3,
 * Table 8).  An FC layer that follows a conv or pool layer reads its input
 * flattened in C*H*W order.  The input channel count of each layer is the
 * output channel count of the layer before it.  Each layer runs the plan of
 * its single-layer call (qcnn_conv_forward with the layer's algo,
 * qcnn_fc_forward, qcnn_maxpool), with one launch fewer where a layer's
 * split partial sums go straight to the next layer instead of a reduction:
 *   - a conv layer to the max-pool after it (planes of at most 12288
 *     elements): the pool adds them in split order, then the bias and ReLU,
 *     as the reduction does, so the output is bit-identical;
 *   - an FC layer to the FC layer after it (batches of at most 8): the next
 *     layer adds them in split order while staging its input, which may
 *     round differently from the single call's reduction.
 */
typedef enum { QCNN_LAYER_CONV = 0, QCNN_LAYER_FC = 1, QCNN_LAYER_MAXPOOL = 2 } qcnn_layer_kind;

typedef struct {
    int kind;           /* qcnn_layer_kind                                   */
    int Ct;             /* CONV / FC: output channels                        */
    int kh, kw;         /* CONV: kernel size; MAXPOOL: window (kh == kw)     */
    int stride, pad;    /* CONV: stride, zero padding; MAXPOOL: stride       */
    int Csp, K;         /* CONV / FC: sub-space dimension, sub-codewords     */
    int relu;           /* CONV / FC: 1 = ReLU after the bias                */
    int algo;           /* CONV: qcnn_algo, optionally | QCNN_ALGO_NO_CLUSTER */
    int codes_layout;   /* CONV: qcnn_codes_layout of `codes`; FC: CANONICAL
                           ([M][Ct] bytes) or PACKED (qcnn_fc_pack_codes)   */
    int lut_type;       /* CONV / FC: qcnn_lut_type of the table entries     */
    const float *D;     /* CONV / FC: [M][K][Csp], device                    */
    const uint8_t *codes; /* CONV: see qcnn_conv_forward; FC: [M][Ct]; device */
    const float *bias;  /* [Ct] or NULL, device                              */
} qcnn_layer;

/*
 * Quantizer: learning D and the codes from dense weights by k-means in
 * every sub-space (Sec. 3.1, Eq. 4 for FC; Sec. 3.2, Eq. 6 for conv), all
 * sub-spaces at once.  Lloyd's algorithm from caller-supplied initial
 * centroids: `iters` rounds of (assign every point to its nearest centroid;
 * move every centroid to the mean of its points), then a last assignment
 * against the final centroids gives the codes.
 *   - distances: sum_j (x_j - c_j)^2 in binary32, term by term (each
 *     subtraction, square and sum rounded, no fused multiply-add); ties go
 *     to the smallest index;
 *   - means: coordinates summed in double in point-index order, divided by
 *     the count, rounded to binary32; a centroid without points keeps its
 *     value.
 * Both rules are fixed, so the results are reproducible bit for bit.
 *
 * qcnn_kmeans: generic form.
 *   points [M][P][Csp] fp32, init [M][K][Csp] fp32 (device)
 *   D      [M][K][Csp] fp32, written;  assign [M][P] uint8, written
 * qcnn_pq_quantize: a layer's weights.
 *   kind QCNN_LAYER_FC:   W [Ct][Cs] (one weight vector per row; kh, kw
 *                         ignored); codes [M][Ct] (qcnn_fc_forward layout)
 *   kind QCNN_LAYER_CONV: W [Ct][Cs][kh][kw]; sub-space m pools the m-th
 *                         sub-vectors of every kernel at every offset, point
 *                         p = c_t * kh*kw + p_k; codes [Ct][kh*kw][M]
 *                         (qcnn_conv_forward canonical layout)
 *   init [M][K][Csp]; D [M][K][Csp] written.
 * Limits as for the forward calls (1 <= Csp <= 8, 1 <= K <= 256,
 * Cs % Csp == 0), iters >= 0.  Workspace from the matching query,
 * 256-byte aligned.
 */
qcnn_status qcnn_kmeans_workspace_size(int M, int P, int Csp, int K, size_t *bytes);
qcnn_status qcnn_kmeans(const float *points, int M, int P, int Csp, int K,
                        const float *init, int iters, float *D, uint8_t *assign,
                        void *workspace, size_t workspace_bytes, void *stream);
qcnn_status qcnn_pq_quantize_workspace_size(int kind, int Ct, int Cs, int kh, int kw,
                                            int Csp, int K, size_t *bytes);
qcnn_status qcnn_pq_quantize(int kind, const float *W, int Ct, int Cs, int kh, int kw,
                             int Csp, int K, const float *init, int iters, float *D,
                             uint8_t *codes, void *workspace, size_t workspace_bytes,
                             void *stream);

/*
 * qcnn_ec_quantize_fc -- quantization with error correction of an FC layer
 * (Sec. 3.3.1, Eq. 8-12): minimises
 *     sum_n || T_n - sum_m (D^(m) B^(m))^T S_n^(m) ||^2
 * over N calibration vectors (S_n: the layer input in the quantized
 * network, T_n: the response of the original layer), by block coordinate
 * descent over the sub-spaces m = 0..M-1, `outer` sweeps.  For each m the
 * residual of Eq. 9 is held fixed and `inner` alternations run, each a
 * codeword update (Eq. 11: per-codeword least squares, solved with the
 * Cholesky factor of G = sum_n S_n^(m) S_n^(m)T; a codeword assigned to no
 * output keeps its value) followed by an assignment update (Eq. 12, ties
 * to the smallest index).  Arithmetic in double.
 *   S [N][Cs] fp32, T [N][Ct] fp32 (device)
 *   D [M][K][Csp] fp32, codes [M][Ct] uint8: the starting point on entry
 *     (e.g. from qcnn_pq_quantize), the result on return
 * Synchronizes `stream` before returning.  Returns QCNN_ERR_DATA when some
 * G is not positive definite (fewer than Csp independent calibration
 * sub-vectors); D and codes are then unspecified.
 */
qcnn_status qcnn_ec_quantize_fc_workspace_size(int N, int Cs, int Ct, int Csp, int K,
                                               size_t *bytes);

/*
 * qcnn_ec_quantize_conv -- quantization with error correction of a conv
 * layer (Sec. 3.3.2, Appendix B): minimises
 *     sum_{n,p_t} || sum_{(p_k,p_s)} sum_m (D^(m) B_pk^(m))^T S_{n,p_s}^(m) - T_{n,p_t} ||^2
 * by block coordinate descent over the sub-spaces m = 0..M-1, `outer`
 * sweeps, `inner` alternations per sub-space, each
 *   - a pass over the codewords k = 0..K-1 in order: D_k becomes the
 *     least-squares fit (Eq. B.6) of what the other codewords leave, in the
 *     sum of the input sub-vectors at the offsets assigned to k; a codeword
 *     assigned nowhere keeps its value;
 *   - a pass over the kernel offsets p_k = 0..kh*kw-1 in order: every
 *     channel's code at p_k becomes the best single codeword for what the
 *     other offsets leave (Eq. B.8), ties to the smallest index.
 * Arithmetic in double; zero padding as in qcnn_conv_forward.
 *   S [N][Cs][H][W] fp32 (layer input), T [N][Ct][Ho][Wo] fp32 (response of
 *     the original layer before its bias); device
 *   D [M][K][Csp] fp32, codes [Ct][kh*kw][M] uint8: the starting point on
 *     entry (codes >= K are clamped), the result on return
 * Synchronizes `stream` before returning.  Returns QCNN_ERR_DATA when a
 * least-squares problem or some G is singular; D and codes are then
 * unspecified.
 */
qcnn_status qcnn_ec_quantize_conv_workspace_size(int N, int Cs, int H, int W, int Ct, int kh,
                                                 int kw, int stride, int pad, int Csp, int K,
                                                 size_t *bytes);
qcnn_status qcnn_ec_quantize_conv(const float *S, const float *T, int N, int Cs, int H, int W,
                                  int Ct, int kh, int kw, int stride, int pad, int Csp, int K,
                                  float *D, uint8_t *codes, int outer, int inner, void *workspace,
                                  size_t workspace_bytes, void *stream);
qcnn_status qcnn_ec_quantize_fc(const float *S, const float *T, int N, int Cs, int Ct,
                                int Csp, int K, float *D, uint8_t *codes, int outer,
                                int inner, void *workspace, size_t workspace_bytes,
                                void *stream);

/*
 * Model blob: a whole stack in one byte string, codes stored in
 * ceil(log2 K) bits (the storage model of Table 1) -- 4 Cs K bytes of
 * sub-codebooks plus kh kw M Ct log2(K) / 8 bytes of codes per layer, and
 * the biases.  Layout (little-endian, arrays 16-byte aligned):
 *   header   32 B: "QCNNMDL1", u32 version 1, u32 n_layers, u32 C, H, W,
 *                  u32 0
 *   records  80 B per layer: u32 kind, Ct, kh, kw, stride, pad, Csp, K,
 *                  relu, bits, has_bias, Cs; u64 off_D, off_codes,
 *                  off_bias, 0 (offsets from the end of the records)
 *   payload  D [M][K][Csp] fp32; codes, one bit stream (qcnn_pack_bits
 *            layout) in the canonical order (FC [M][Ct], conv
 *            [Ct][kh*kw][M]); bias [Ct] fp32
 * qcnn_model_serialize: `layers` hold HOST pointers (D, canonical codes,
 *   bias or NULL) for the input C x H x W; writes the blob to host memory
 *   `out` (NULL: only sets *bytes_needed).  QCNN_ERR_WORKSPACE when
 *   out_bytes is too small.
 * qcnn_model_info: validates a blob in host memory (every size, offset and
 *   the layer chain) and gives its layer count, input shape and the device
 *   bytes qcnn_model_upload needs.
 * qcnn_model_upload: copies the blob's arrays into `device_buffer` (256-byte
 *   aligned, at least that size), lays the codes out for the kernels and
 *   fills layers[n_layers] with device pointers into it (codes_layout
 *   PACKED, algo AUTO, lut_type FP32), ready for qcnn_net_forward.
 *   Synchronizes `stream` before returning.
 */
qcnn_status qcnn_model_serialize(const qcnn_layer *layers, int n_layers, int C, int H, int W,
                                 void *out, size_t out_bytes, size_t *bytes_needed);
qcnn_status qcnn_model_info(const void *blob, size_t bytes, int *n_layers, int *C, int *H,
                            int *W, size_t *device_bytes);
qcnn_status qcnn_model_upload(const void *blob, size_t bytes, void *device_buffer,
                              size_t device_bytes, qcnn_layer *layers, void *stream);

/* Output shape of the stack for one image (C, H, W; H = W = 1 after an FC). */
qcnn_status qcnn_net_output_shape(const qcnn_layer *layers, int n_layers,
                                  int C, int H, int W, int *out_C, int *out_H,
                                  int *out_W);

/*
 * qcnn_net_workspace_size: bytes of workspace for qcnn_net_forward
 * (host_io = 0) or qcnn_net_forward_host (host_io = 1, which also stages
 * the input and output in the workspace).
 */
qcnn_status qcnn_net_workspace_size(const qcnn_layer *layers, int n_layers,
                                    int N, int C, int H, int W, int host_io,
                                    size_t *bytes);

/*
 * qcnn_net_plan_info -- where qcnn_net_forward (host_io = 0) or
 * qcnn_net_forward_host (host_io = 1) hands split partial sums from one
 * layer to the next instead of a reduction launch, worked out on the host
 * (no GPU work; the plan is the one those calls cache).  info has
 * 2 * n_layers ints: info[2i] = 1 when layer i leaves its partial sums to
 * layer i + 1, info[2i + 1] = 1 when layer i takes its input as layer
 * i - 1's partial sums.  Errors are those of qcnn_net_workspace_size, plus
 * QCNN_ERR_INVALID_ARG for a NULL info.
 */
qcnn_status qcnn_net_plan_info(const qcnn_layer *layers, int n_layers, int N, int C, int H,
                               int W, int host_io, int *info);

/* x [N][C][H][W] device -> y [N][out_C][out_H][out_W] device. */
qcnn_status qcnn_net_forward(const qcnn_layer *layers, int n_layers,
                             const float *x, int N, int C, int H, int W,
                             float *y, void *workspace, size_t workspace_bytes,
                             void *stream);

/*
 * qcnn_net_forward_host -- the same, with x and y in HOST memory (pinned
 * memory gives the fastest copies).  Copies x to the device, runs the
 * stack, copies y back, and synchronizes `stream` before returning.  When
 * N is a multiple of 2 or 4 with at least 8 images per slice, x is copied
 * in 2 or 4 slices on a separate copy stream of the library, and the first
 * layer runs on each slice as soon as it has arrived.  Calls of this
 * function on one device are serialized.
 */
qcnn_status qcnn_net_forward_host(const qcnn_layer *layers, int n_layers,
                                  const float *x_host, int N, int C, int H,
                                  int W, float *y_host, void *workspace,
                                  size_t workspace_bytes, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* QCNN_H */
