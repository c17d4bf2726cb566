// fc_small.cu -- PQ fully-connected layer response (Sec. 3.1, Eq. 5) for
// small batches (up to 8 images) and K <= 32 sub-codewords:
//   y[n][ct] = bias[ct] + sum_m LUT_n[m][k_m(ct)],  LUT_n[m][k] = <x_n^(m), D^(m)_k>
//
// At small batches the layer is a stream of code bytes (one per output and
// sub-space) and each table entry is read only a few times, so the plan is
// chosen to spread the code bytes over the whole GPU and to need no second
// kernel:
//  * A thread-block cluster of C CTAs owns CT_CTA outputs (one output tile);
//    CTA rank r of the cluster takes the sub-spaces [r*m_per, (r+1)*m_per).
//  * A CTA copies its share to shared memory with cp.async: its slice of
//    the inputs, and per sub-space its sub-codebook and the tile's slice of
//    the code row (bytes or ceil(log2 K)-bit packed).  When the whole share
//    fits it is fetched at once (one memory latency per CTA); otherwise in
//    chunks of MC sub-spaces, one chunk ahead.  The tables of a chunk for
//    the tile's images are built by all threads into shared memory,
//    T[mm][n][k].
//  * Gather by warp shuffle: for sub-space mm and image n, lane l loads
//    T[mm][n][l] (one conflict-free load per warp) and every lane fetches the
//    entries its outputs' codes name with __shfl_sync -- one shuffle serves
//    the 32 lanes' look-ups whatever the codes are, where a shared-memory
//    gather of random codes would serialize on bank conflicts.
//  * The C partial sums of each output are added through distributed shared
//    memory: every CTA leaves its sums in its own shared memory, the cluster
//    synchronizes, and CTA r adds the r-th slice of the tile's outputs from
//    all C CTAs in rank order (a fixed order: results are reproducible bit
//    for bit), adds the bias, applies ReLU and writes y.
#include "qcnn_internal.cuh"

#include <cooperative_groups.h>

#include <algorithm>
#include <cmath>

namespace cg = cooperative_groups;

namespace qcnn {

struct FcSmallArgs {
    const float *x;  // usually the output of the kernel before
    const float *__restrict__ D;
    const uint8_t *__restrict__ codes;
    const float *__restrict__ bias;
    float *__restrict__ y;
    int N, Cs, Ct, Csp, K, M;
    int C, m_per, MC, relu;
    int cvec;     // bytes per code copy (16, 8 or 4; 0: byte by byte)
    int cbits;    // 0: byte codes [M][Ct]; else packed rows of cbits-bit codes
    int cpitch;   // bytes per code row in device memory
    int crow;     // bytes of the tile's slice of a code row (a multiple of 16)
};

// staged code rows are crow + 16 bytes apart: the word after a packed slice
// is read (and ignored) by the last lane's funnel shift
__host__ __device__ inline int fc_small_cstride(int crow) { return crow + 16; }

constexpr int kSmallThreads = 256;
constexpr int kSmallWarps = kSmallThreads / 32;
constexpr int kTC = 32;  // sub-spaces per table build (the tables of a staged chunk
                         // are built and gathered kTC sub-spaces at a time)

// shared memory carve-up (byte offsets, 16-aligned); nbuf = 1 when the
// CTA's whole share is one chunk (MC = m_per), else 2 (double buffered)
struct FcSmallSmem {
    size_t xs, ts, ds, cs, red, total;
    int nbuf;
};
__host__ __device__ inline FcSmallSmem fc_small_layout(int NB, int m_per, int Csp, int K, int MC,
                                                       int crow, int ct_cta) {
    FcSmallSmem L;
    L.nbuf = MC >= m_per ? 1 : 2;
    L.xs = 0;                                                         // [NB][m_per * Csp]
    L.ts = L.xs + ((size_t)NB * m_per * Csp * 4 + 15) / 16 * 16;      // [kTC][NB][32]
    L.ds = L.ts + (size_t)kTC * NB * 32 * 4;                          // [nbuf][MC][K][Csp]
    L.cs = L.ds + ((size_t)L.nbuf * MC * K * Csp * 4 + 15) / 16 * 16;  // [nbuf][MC][cstride]
    L.red = L.cs + (size_t)L.nbuf * MC * fc_small_cstride(crow);       // [ct_cta][NB]
    L.total = L.red + (size_t)ct_cta * NB * 4;
    return L;
}

// NB: images per CTA (a power of two, 1..8); OPL: consecutive outputs per
// lane (1, 2 or 4), so a CTA's tile is CT_CTA = 256 * OPL outputs.
template <int NB, int OPL, bool BF>
__global__ void __launch_bounds__(kSmallThreads, 1) fc_small_kernel(const FcSmallArgs a) {
    constexpr int CT_CTA = kSmallThreads * OPL;
    extern __shared__ __align__(16) unsigned char smem[];
    const FcSmallSmem L = fc_small_layout(NB, a.m_per, a.Csp, a.K, a.MC, a.crow, CT_CTA);
    float *xs = reinterpret_cast<float *>(smem + L.xs);
    float *ts = reinterpret_cast<float *>(smem + L.ts);
    float *ds = reinterpret_cast<float *>(smem + L.ds);
    uint8_t *cs = smem + L.cs;
    float *red = reinterpret_cast<float *>(smem + L.red);
    cg::cluster_group cluster = cg::this_cluster();
    grid_dep_sync();

    const int tid = threadIdx.x, lane = tid & 31;
    const int rank = (int)cluster.block_rank();
    const int tile = blockIdx.x / a.C;
    const int ct0 = tile * CT_CTA;
    const int n0 = blockIdx.y * NB;
    const int mb = rank * a.m_per, me = min(a.M, mb + a.m_per);
    const int nm = max(0, me - mb);
    const int n_chunks = (nm + a.MC - 1) / a.MC;
    const int lane_ct = tid * OPL;  // first output of this lane in the tile

    // x slice of the CTA's sub-spaces, every image of the tile (zeros past N)
    const int xw = nm * a.Csp;
    for (int e = tid; e < NB * xw; e += kSmallThreads) {
        const int n = e / xw, j = e - n * xw;
        const bool ok = n0 + n < a.N;
        cp_async4(xs + n * a.m_per * a.Csp + j,
                  ok ? a.x + (size_t)(n0 + n) * a.Cs + (size_t)mb * a.Csp + j : a.x, ok);
    }
    // chunk c -> buffer b: sub-codebooks D[m0 .. m0 + mc) (contiguous) and
    // the code rows' slices of this tile
    const int cstride = fc_small_cstride(a.crow);
    const int dch = a.MC * a.K * a.Csp;  // floats of one D buffer
    auto stage_codes = [&](int c, int b) {
        const int m0 = mb + c * a.MC, mc = min(a.MC, me - m0);
        const float *dsrc = a.D + (size_t)m0 * a.K * a.Csp;
        float *db = ds + (size_t)b * dch;
        for (int e = tid; e < mc * a.K * a.Csp; e += kSmallThreads) cp_async4(db + e, dsrc + e, true);
        uint8_t *cb = cs + (size_t)b * a.MC * cstride;
        const size_t off0 = a.cbits ? (size_t)tile * a.crow : (size_t)ct0;
        const size_t row_end = a.cbits ? (size_t)a.cpitch : (size_t)a.Ct;
        if (a.cvec == 0) {  // rows not 4-byte aligned: byte by byte, zeros past the row
            for (int e = tid; e < mc * a.crow; e += kSmallThreads) {
                const int mm = e / a.crow, q = e - mm * a.crow;
                const size_t byte = off0 + q;
                cb[mm * cstride + q] =
                    byte < row_end ? a.codes[(size_t)(m0 + mm) * a.cpitch + byte] : (uint8_t)0;
            }
            return;
        }
        const int per_row = a.crow / a.cvec;
        for (int e = tid; e < mc * per_row; e += kSmallThreads) {
            const int mm = e / per_row, q = e - mm * per_row;
            const size_t byte = off0 + (size_t)q * a.cvec;
            const bool ok = byte < row_end;  // whole copies: Ct (or the pitch) is a multiple
            const uint8_t *src = ok ? a.codes + (size_t)(m0 + mm) * a.cpitch + byte : a.codes;
            const unsigned d = smem_addr(cb + mm * cstride + q * a.cvec);
            const int sz = ok ? a.cvec : 0;
            if (a.cvec == 16)
                asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d), "l"(src),
                             "r"(sz)
                             : "memory");
            else if (a.cvec == 8)
                asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;\n" ::"r"(d), "l"(src),
                             "r"(sz)
                             : "memory");
            else
                asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(d), "l"(src),
                             "r"(sz)
                             : "memory");
        }
    };
    if (n_chunks > 0) stage_codes(0, 0);
    cp_async_commit();

    float acc[OPL][NB];
#pragma unroll
    for (int o = 0; o < OPL; ++o)
#pragma unroll
        for (int n = 0; n < NB; ++n) acc[o][n] = 0.f;
    const unsigned kmax = (unsigned)(a.K - 1);
    const int bit0 = lane_ct * a.cbits;
    const unsigned cmask = (1u << a.cbits) - 1u;

    for (int c = 0; c < n_chunks; ++c) {
        const int b = L.nbuf == 1 ? 0 : c & 1;
        const int m0 = mb + c * a.MC, mc = min(a.MC, me - m0);
        cp_async_wait<0>();
        __syncthreads();  // chunk c (and the x slice) staged; gather of c-1 done
        if (c + 1 < n_chunks) stage_codes(c + 1, b ^ 1);
        cp_async_commit();
        const float *db = ds + (size_t)b * dch;
        const uint8_t *cb = cs + (size_t)b * a.MC * cstride;
        for (int t0 = 0; t0 < mc; t0 += kTC) {
            const int tc = min(kTC, mc - t0);
            if (t0 > 0) __syncthreads();  // gather of the previous tables done
            // tables: ts[i][n][k] = <x_n^(m), D[m][k]>, m = m0 + t0 + i (k < K;
            // rows padded to 32 with the entry of K - 1, never selected)
            for (int e = tid; e < tc * NB * 32; e += kSmallThreads) {
                const int k = e & 31, r = e >> 5, n = r % NB, i = r / NB;
                const int kk = min(k, a.K - 1);
                const float *dp = db + ((t0 + i) * a.K + kk) * a.Csp;
                const float *xp = xs + n * a.m_per * a.Csp + (m0 - mb + t0 + i) * a.Csp;
                float v = 0.f;
                for (int j = 0; j < a.Csp; ++j) v = fmaf(xp[j], dp[j], v);
                if constexpr (BF) v = __bfloat162float(__float2bfloat16_rn(v));
                ts[e] = v;
            }
            __syncthreads();
            for (int i = 0; i < tc; ++i) {
                const int mm = t0 + i;
                // this lane's OPL codes of sub-space m0 + mm
                unsigned w;
                if (a.cbits) {
                    const unsigned *cw = reinterpret_cast<const unsigned *>(cb + mm * cstride);
                    const unsigned v =
                        __funnelshift_r(cw[bit0 >> 5], cw[(bit0 >> 5) + 1], bit0 & 31);
                    w = 0;
#pragma unroll
                    for (int o = 0; o < OPL; ++o) w |= ((v >> (o * a.cbits)) & cmask) << (8 * o);
                } else if constexpr (OPL == 4) {
                    w = *reinterpret_cast<const unsigned *>(cb + mm * cstride + lane_ct);
                } else if constexpr (OPL == 2) {
                    w = *reinterpret_cast<const unsigned short *>(cb + mm * cstride + lane_ct);
                } else {
                    w = cb[mm * cstride + lane_ct];
                }
                const float *tr = ts + (size_t)i * NB * 32 + lane;
#pragma unroll
                for (int n = 0; n < NB; ++n) {
                    const float t = tr[n * 32];
#pragma unroll
                    for (int o = 0; o < OPL; ++o) {
                        const unsigned code = byte_of(w, o);
                        QCNN_CHECK(code <= kmax, QCNN_CHECK_CODE);
                        acc[o][n] += __shfl_sync(0xffffffffu, t, (int)min(code, kmax));
                    }
                }
            }
        }
    }

    // ---- cluster reduction of the C partial sums (fixed rank order)
#pragma unroll
    for (int o = 0; o < OPL; ++o)
#pragma unroll
        for (int n = 0; n < NB; ++n) red[(lane_ct + o) * NB + n] = acc[o][n];
    cluster.sync();
    const int E = CT_CTA * NB;
    const int per = (E + a.C - 1) / a.C;
    const int e0 = rank * per, e1 = min(E, e0 + per);
    for (int e = e0 + tid; e < e1; e += kSmallThreads) {
        float v = 0.f;
        for (int q = 0; q < a.C; ++q) v += cluster.map_shared_rank(red, q)[e];
        const int o = e / NB, n = e - o * NB;
        const int ct = ct0 + o;
        if (ct < a.Ct && n0 + n < a.N) {
            if (a.bias) v += a.bias[ct];
            if (a.relu) v = fmaxf(v, 0.f);
            QCNN_CHECK((size_t)(n0 + n) * a.Ct + ct < (size_t)a.N * a.Ct, QCNN_CHECK_GLOBAL);
            a.y[(size_t)(n0 + n) * a.Ct + ct] = v;
        }
    }
    cluster.sync();  // no CTA leaves while its sums may still be read
}

struct FcSmallVariant {
    int NB, OPL, BF;
    void (*fn)(FcSmallArgs);
};
#define QCNN_FCS(NB, OPL) {NB, OPL, 0, fc_small_kernel<NB, OPL, false>}, \
                          {NB, OPL, 1, fc_small_kernel<NB, OPL, true>}
static const FcSmallVariant kFcSmall[] = {
    QCNN_FCS(1, 1), QCNN_FCS(1, 2), QCNN_FCS(1, 4), QCNN_FCS(2, 1), QCNN_FCS(2, 2),
    QCNN_FCS(2, 4), QCNN_FCS(4, 1), QCNN_FCS(4, 2), QCNN_FCS(4, 4), QCNN_FCS(8, 1),
    QCNN_FCS(8, 2), QCNN_FCS(8, 4)};
#undef QCNN_FCS
constexpr int kNumFcSmall = sizeof(kFcSmall) / sizeof(kFcSmall[0]);
constexpr int kMaxCluster = 16;

// The plan: among the variants for the batch (images per CTA) and the
// cluster sizes 2..16, the one with the least estimated time, in SM cycles:
// per CTA the larger of its load streams (the tile's code rows from HBM at
// about 40 B per cycle, its sub-codebooks from L2 at about 64 B per cycle)
// and its shared-memory and shuffle instructions (per sub-space and image:
// one table load and OPL shuffles per warp), plus a fixed cost for launch
// and the two cluster barriers; times the waves of co-resident clusters.
FcSmallPlan plan_fc_small(const FcShape &s) {
    FcSmallPlan best;
    if (s.N > 8 || s.K > 32) return best;
    const int sms = num_sms();
    const int NB = s.N <= 1 ? 1 : s.N <= 2 ? 2 : s.N <= 4 ? 4 : 8;
    double best_t = 1e300;
    for (int v = 0; v < kNumFcSmall; ++v) {
        const FcSmallVariant &fv = kFcSmall[v];
        if (fv.NB != NB || fv.BF != s.bf16) continue;
        const int ct_cta = kSmallThreads * fv.OPL;
        const int tiles = cdiv(s.Ct, ct_cta);
        // packed codes: the tile's slice of a row, a whole number of 16-byte pieces
        const int crow = s.code_bits ? ct_cta * s.code_bits / 8 : ct_cta;
        if (crow % 16 != 0) continue;
        for (int C = 2; C <= kMaxCluster; C *= 2) {
            const int m_per = cdiv(s.M, C);
            // the whole share in one stage when it fits, else chunks of 32
            int MC = m_per;
            FcSmallSmem L = fc_small_layout(NB, m_per, s.Csp, s.K, MC, crow, ct_cta);
            if (L.total > 200 * 1024) {
                MC = std::min(m_per, 32);
                L = fc_small_layout(NB, m_per, s.Csp, s.K, MC, crow, ct_cta);
            }
            if (L.total > 200 * 1024) continue;
            const int active = cluster_capacity(reinterpret_cast<const void *>(fv.fn),
                                                kSmallThreads, C, L.total);
            if (active < 1) continue;
            const double waves = std::ceil((double)tiles / active);
            // CTAs of a wave that share one SM share its pipes and bandwidth
            const double per_sm = std::ceil((double)std::min(tiles, active) * C / sms);
            const double t_load = std::max((double)m_per * crow / 40.0,
                                           (double)m_per * s.K * s.Csp * 4.0 / 64.0);
            const double t_comp = (double)m_per * NB * kSmallWarps * (fv.OPL + 1) +
                                  (double)m_per * NB * 32 * s.Csp / kSmallThreads;
            const double t = waves * (per_sm * std::max(t_load, t_comp) + 3000.0);
            if (t < best_t) {
                best_t = t;
                best.ok = true;
                best.variant = v;
                best.NB = NB;
                best.OPL = fv.OPL;
                best.ct_cta = ct_cta;
                best.tiles = tiles;
                best.C = C;
                best.m_per = m_per;
                best.MC = MC;
                best.crow = crow;
                best.smem = L.total;
            }
        }
    }
    return best;
}

qcnn_status launch_fc_small(const FcShape &s, const FcSmallPlan &p, const float *x,
                            const float *D, const uint8_t *codes, const float *bias, float *y,
                            int relu, cudaStream_t st) {
    const FcSmallVariant &fv = kFcSmall[p.variant];
    FcSmallArgs a;
    a.x = x;
    a.D = D;
    a.codes = codes;
    a.bias = bias;
    a.y = y;
    a.N = s.N;
    a.Cs = s.Cs;
    a.Ct = s.Ct;
    a.Csp = s.Csp;
    a.K = s.K;
    a.M = s.M;
    a.C = p.C;
    a.m_per = p.m_per;
    a.MC = p.MC;
    a.relu = relu;
    a.cbits = s.code_bits;
    a.cpitch = s.code_bits ? (int)fc_packed_pitch(s.Ct, s.K) : s.Ct;
    a.crow = p.crow;
    const uintptr_t base = reinterpret_cast<uintptr_t>(codes);
    if (s.code_bits) {
        a.cvec = 16;  // packed rows: 16-byte pitch, 16-byte aligned array
    } else {
        a.cvec = (s.Ct % 16 == 0 && base % 16 == 0) ? 16
                 : (s.Ct % 8 == 0 && base % 8 == 0) ? 8
                 : (s.Ct % 4 == 0 && base % 4 == 0) ? 4
                                                     : 0;
    }
    cudaError_t e = cudaFuncSetAttribute(fv.fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(fv.fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem);
    if (e != cudaSuccess) return cuda_status(e);
    const dim3 grid(p.tiles * p.C, cdiv(s.N, p.NB), 1);
    return launch_k(fv.fn, grid, dim3(kSmallThreads), p.smem, st, dim3(p.C, 1, 1), a);
}

}  // namespace qcnn
