// fc.cu -- PQ fully-connected layer response (Sec. 3.1, Eq. 5):
//   y[n][ct] = bias[ct] + sum_m LUT_n[m][k_m(ct)],  LUT_n[m][k] = <x_n^(m), D^(m)_k>
//
// One CTA owns NT images, CT_CTA outputs and a range of sub-spaces.  It walks
// that range in chunks of MCH sub-spaces: the chunk's tables for its NT
// images are built in shared memory, layout lut[mm][k][n] with an odd row
// pitch NTP, then every lane -- which owns CPL = 4 consecutive outputs and
// NW images -- adds lut[mm][code][n] for its codes.  Lanes of a warp hold
// different codes for the same (mm, n): with the odd pitch, distinct codes
// below 32 land in distinct banks and equal codes broadcast, so the gather is
// conflict free for K <= 32.  The chunk's codes, inputs and sub-codebooks are
// copied to shared memory with cp.async one chunk ahead (double buffered), so
// their device-memory latency overlaps the previous chunk's gather; each
// code then serves NW images.
// bfloat16 tables (BF): a 32-bit table word holds the entries of two images
// (2i, 2i+1) for the same (mm, k) -- both use the same code -- so one load
// serves two look-ups; the word pitch of a row is odd as above.  Tiles of a
// single image per lane keep 2-byte entries (pitch NT | 1 halves).
// Codes can also come bit-packed (b = ceil(log2 K) bits each, every [M][Ct]
// row padded to a 16-byte pitch): a CTA's slice of a row is then b * CT_CTA
// / 8 bytes, staged with 16-byte copies, and a lane takes its 4 codes from one
// funnel shift of two 32-bit words -- 8/b times fewer code bytes from HBM.
// When the sub-space range is split over several CTAs (to fill the GPU),
// the partial sums go to the workspace and a second kernel adds them in a
// fixed order (deterministic), then applies bias and ReLU.  With many splits
// of small image tiles, clusters of CTAs first add their partial tiles in
// distributed shared memory (rank order), so fewer partial sums per output
// reach the workspace.
#include "qcnn_internal.cuh"

#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <type_traits>

namespace qcnn {

struct FcArgs {
    const float *__restrict__ x;
    const float *__restrict__ D;
    const uint8_t *__restrict__ codes;  // [M][Ct]
    const float *__restrict__ bias;
    float *__restrict__ y;
    float *__restrict__ partial;  // [splits][N][Ct] when splits > 1
    int N, Cs, Ct, Csp, K, M;
    int NT, CT_CTA, MCH, n_chunks, chunks_per_split, splits, relu;
    int cl;  // the splits of a tile form clusters of cl CTAs (1: none)
    int cvec;    // bytes per code copy: 16, 8 or 4 (0: byte copies)
    int cbits;   // 0: one byte per code; else bits per code (packed rows)
    int cpitch;  // packed: bytes per code row (multiple of 16)
    int crb;     // bytes per staged code row in shared memory (CT_CTA + 16)
    int cch_log2;  // log2 of MCH * Csp rounded up to a power of two
    int dvec16;    // 1: sub-codebooks staged in 16-byte pieces (K * Csp % 4 == 0, D 16-aligned)
    // xgroups > 0: the input is the previous FC layer's output still as
    // partial sums, x[n][c] = act(xbias[c] + sum_g xpart[g][n][c]) (act: ReLU
    // when xrelu), added in g order while staging -- that layer's reduction
    // kernel is not run.  (Written by the kernel before: coherent loads.)
    const float *xpart;
    const float *xbias;
    int xgroups, xrelu;
    int k_log2;    // log2 K when K is a power of two, else -1
    // 1: D and the codes are constants of the caller (no kernel of the same
    // call writes them): the first chunk's are staged before the wait on the
    // previous kernel (programmatic dependent launch), only x after it
    int early;
};

constexpr int kFcThreads = 256;
constexpr int kCPL = 4;       // outputs per lane
constexpr int kMchMax = 16;   // sub-spaces per chunk, at most

struct FcSmem {
    size_t lut, xs, ds, cs, total;
};
// row_bytes: bytes of one table row (NTP entries or words); code rows are
// staged at a stride of CT_CTA + 16 bytes (byte codes, or a packed slice plus
// the word the last lane's shift reads past it)
__host__ __device__ inline FcSmem fc_smem_layout(int MCH, int K, int row_bytes, int NTX,
                                                 int Csp, int CT_CTA) {
    FcSmem s;
    s.lut = 0;
    s.xs = ((size_t)MCH * K * row_bytes + 15) / 16 * 16;
    s.ds = s.xs + ((size_t)2 * MCH * Csp * NTX * 4 + 15) / 16 * 16;
    s.cs = s.ds + ((size_t)2 * MCH * K * Csp * 4 + 15) / 16 * 16;
    s.total = s.cs + (size_t)2 * MCH * (CT_CTA + 16);
    return s;
}

// bytes of one table row
__host__ __device__ inline int fc_row_bytes(int NT, int NTP, bool bf16) {
    return bf16 && NT % 2 != 0 ? (NTP * 2 + 3) / 4 * 4 : NTP * 4;
}

// a += the bfloat16 value h, widened to fp32 (exact), one fp32 rounding
__device__ __forceinline__ void add_bf16(float &a, unsigned short h) {
    asm("add.rn.f32.bf16 %0, %1, %0;" : "+f"(a) : "h"(h));
}

// NW : images per lane;  WN : warps along images (8 / WN along outputs)
// MINB : CTAs per SM the register budget is sized for
// BF : bfloat16 tables
template <int NW, int WN, int MINB, bool BF>
__global__ void __launch_bounds__(kFcThreads, MINB) fc_fused_kernel(const FcArgs a) {
    constexpr int CT_CTA = (8 / WN) * 32 * kCPL;
    constexpr int kCtCtaLog2 = CT_CTA == 1024 ? 10 : (CT_CTA == 512 ? 9 : 8);
    static_assert((1 << kCtCtaLog2) == CT_CTA, "output tile must be 256, 512 or 1024");
    constexpr int NT = NW * WN;  // images per CTA (== a.NT)
    constexpr bool PAIRS = BF && NW % 2 == 0;  // bf16 words of two images
    static_assert(!BF || NW % 2 == 0 || NW == 1, "bf16 tiles: even NW or NW == 1");
    // odd row pitches (compile-time, so row addresses fold): the table's
    // (fp32: floats >= NT; bf16 pairs: words >= NT/2; bf16 singles: halves
    // >= NT) and the staged x's (>= NT)
    constexpr int NTP = (BF && NT % 2 == 0 ? NT / 2 : NT) | 1;
    constexpr int NTX = NT | 1;
    extern __shared__ __align__(16) unsigned char smem[];
    const FcSmem L = fc_smem_layout(a.MCH, a.K, fc_row_bytes(NT, NTP, BF), NTX, a.Csp, CT_CTA);
    float *lut = reinterpret_cast<float *>(smem + L.lut);
    float *xs = reinterpret_cast<float *>(smem + L.xs);
    float *ds = reinterpret_cast<float *>(smem + L.ds);
    uint8_t *cs = smem + L.cs;
    if (!a.early) grid_dep_sync();

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int wn = warp % WN, wc = warp / WN;
    const int ct0 = blockIdx.x * CT_CTA;
    const int n0 = blockIdx.y * a.NT;
    const int split = blockIdx.z;
    const int c_begin = split * a.chunks_per_split;
    const int c_end = min(a.n_chunks, c_begin + a.chunks_per_split);
    const int lane_ct = (wc * 32 + lane) * kCPL;  // first output of this lane in the tile
    const int nbase = wn * NW;
    const int CCH = a.MCH * a.Csp;  // staged x floats per image
    const unsigned kmax4 = (unsigned)(a.K - 1) * 0x01010101u;

    auto stage_x = [&](int c, int b) {
        const int m0 = c * a.MCH;
        const int mch = min(a.MCH, a.M - m0);
        float *xb = xs + (size_t)b * CCH * NTX;
        // (image nn, float cc) with cc on a power-of-two stride: no division
        const int cmask = (1 << a.cch_log2) - 1;
        if (a.xgroups > 0) {  // sums of the previous layer's partials, in group order
            const size_t plane = (size_t)a.N * a.Cs;
            for (int e = tid; e < (NT << a.cch_log2); e += kFcThreads) {
                const int cc = e & cmask, nn = e >> a.cch_log2;
                if (cc >= CCH) continue;
                float v = 0.f;
                if (cc < mch * a.Csp && n0 + nn < a.N) {
                    const size_t c = (size_t)m0 * a.Csp + cc;
                    const float *src = a.xpart + (size_t)(n0 + nn) * a.Cs + c;
                    for (int g = 0; g < a.xgroups; ++g) v += src[g * plane];
                    if (a.xbias) v += a.xbias[c];
                    if (a.xrelu) v = fmaxf(v, 0.f);
                }
                xb[cc * NTX + nn] = v;
            }
            return;
        }
        for (int e = tid; e < (NT << a.cch_log2); e += kFcThreads) {
            const int cc = e & cmask, nn = e >> a.cch_log2;
            if (cc >= CCH) continue;
            const bool ok = cc < mch * a.Csp && n0 + nn < a.N;
            const float *src = ok ? a.x + (size_t)(n0 + nn) * a.Cs + (size_t)m0 * a.Csp + cc : a.x;
            cp_async4(xb + cc * NTX + nn, src, ok);
        }
    };
    auto stage_w = [&](int c, int b) {  // sub-codebooks and codes of chunk c
        const int m0 = c * a.MCH;
        const int mch = min(a.MCH, a.M - m0);
        float *db = ds + (size_t)b * a.MCH * a.K * a.Csp;
        const int dn = a.MCH * a.K * a.Csp, dv = mch * a.K * a.Csp;
        const float *dsrc = a.D + (size_t)m0 * a.K * a.Csp;
        if (a.dvec16) {  // 16-byte pieces (the build reads only the chunk's mch sub-spaces)
            for (int e = tid * 4; e < dv; e += kFcThreads * 4) cp_async16(db + e, dsrc + e);
        } else {
            for (int e = tid; e < dn; e += kFcThreads) cp_async4(db + e, e < dv ? dsrc + e : a.D, e < dv);
        }
        // codes[m0 + mm][ct0 .. ct0 + CT_CTA) -> cs[b][mm][.]; zero outside
        uint8_t *cb = cs + (size_t)b * a.MCH * a.crb;
        // Each thread copies one column q of the rows mm = mm_first,
        // mm_first + rows_step, ...: its source and destination advance by a
        // fixed step (no per-copy index arithmetic)
        if (a.cbits) {  // packed rows: this CTA's slice, whole 16-byte copies
            const int slice = (CT_CTA * a.cbits) >> 3;
            const int nq = slice >> 4;  // copies per row (<= 64)
            const int rows_step = kFcThreads / nq;
            if (tid < rows_step * nq) {
                const int mm_first = tid / nq, qq = tid - mm_first * nq;
                const size_t byte = (size_t)blockIdx.x * slice + (size_t)qq * 16;
                const bool col_ok = byte < (size_t)a.cpitch;
                const uint8_t *src = a.codes + (size_t)(m0 + mm_first) * a.cpitch + byte;
                const size_t src_step = (size_t)rows_step * a.cpitch;
                unsigned d = smem_addr(cb + mm_first * a.crb + qq * 16);
                const unsigned d_step = (unsigned)(rows_step * a.crb);
                for (int mm = mm_first; mm < a.MCH; mm += rows_step, src += src_step, d += d_step) {
                    const bool ok = col_ok && mm < mch;
                    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d),
                                 "l"(ok ? src : a.codes), "r"(ok ? 16 : 0)
                                 : "memory");
                }
            }
        } else if (a.cvec > 0) {
            // copies of V bytes (the row's alignment), V fixed per loop
            auto copy_rows = [&](auto vc) {
                constexpr int V = decltype(vc)::value;
                constexpr int row_log2 = kCtCtaLog2 - (V == 16 ? 4 : V == 8 ? 3 : 2);
                constexpr int per_row = 1 << row_log2;  // copies per code row (<= 256)
                constexpr int rows_step = kFcThreads / per_row;
                const int mm_first = tid >> row_log2, q = tid & (per_row - 1);
                const int ct = ct0 + q * V;
                const bool col_ok = ct < a.Ct;  // Ct % V == 0: all or nothing
                const uint8_t *src = a.codes + (size_t)(m0 + mm_first) * a.Ct + ct;
                const size_t src_step = (size_t)rows_step * a.Ct;
                unsigned d = smem_addr(cb + mm_first * a.crb + q * V);
                const unsigned d_step = (unsigned)(rows_step * a.crb);
                for (int mm = mm_first; mm < a.MCH; mm += rows_step, src += src_step, d += d_step) {
                    const bool ok = col_ok && mm < mch;
                    const uint8_t *s = ok ? src : a.codes;
                    const int sz = ok ? V : 0;
                    if constexpr (V == 16)
                        asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d), "l"(s), "r"(sz) : "memory");
                    else if constexpr (V == 8)
                        asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;\n" ::"r"(d), "l"(s), "r"(sz) : "memory");
                    else
                        asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(d), "l"(s), "r"(sz) : "memory");
                }
            };
            if (a.cvec == 16) copy_rows(std::integral_constant<int, 16>());
            else if (a.cvec == 8) copy_rows(std::integral_constant<int, 8>());
            else copy_rows(std::integral_constant<int, 4>());
        } else {  // rows not 4-byte aligned: plain byte copies
            for (int e = tid; e < a.MCH * CT_CTA; e += kFcThreads) {
                const int mm = e / CT_CTA, q = e % CT_CTA;
                const int ct = ct0 + q;
                cb[mm * a.crb + q] = (mm < mch && ct < a.Ct) ? a.codes[(size_t)(m0 + mm) * a.Ct + ct] : 0;
            }
        }
    };
    auto stage = [&](int c, int b) {
        stage_x(c, b);
        stage_w(c, b);
    };

    float acc[kCPL][NW];
#pragma unroll
    for (int c = 0; c < kCPL; ++c)
#pragma unroll
        for (int i = 0; i < NW; ++i) acc[c][i] = 0.f;

    if (c_begin < c_end) stage_w(c_begin, 0);
    if (a.early) grid_dep_sync();
    if (c_begin < c_end) stage_x(c_begin, 0);
    cp_async_commit();
    for (int c = c_begin; c < c_end; ++c) {
        const int b = (c - c_begin) & 1;
        const int mch = min(a.MCH, a.M - c * a.MCH);
        cp_async_wait<0>();
        __syncthreads();  // chunk c staged; gather of c-1 finished
        if (c + 1 < c_end) {
            stage(c + 1, b ^ 1);
            cp_async_commit();
        }

        // build lut[mm][k][nn] = <x(nn, mm), D[m0 + mm][k]>; (k, nn) with nn
        // fastest over the compile-time image tile: no division
        {
            const float *xb = xs + (size_t)b * CCH * NTX;
            const float *db = ds + (size_t)b * a.MCH * a.K * a.Csp;
            for (int mm = 0; mm < mch; ++mm) {
                if constexpr (PAIRS) {
                    constexpr int NP = NT / 2;  // image pairs
                    unsigned *lw = reinterpret_cast<unsigned *>(lut);
                    for (int e = tid; e < a.K * NP; e += kFcThreads) {
                        const int np = e % NP, k = e / NP;
                        const float *xp = xb + mm * a.Csp * NTX + 2 * np;
                        const float *dp = db + (mm * a.K + k) * a.Csp;
                        float v0 = 0.f, v1 = 0.f;
#pragma unroll
                        for (int j = 0; j < kMaxCsp; ++j) {
                            if (j < a.Csp) {
                                v0 = fmaf(xp[j * NTX], dp[j], v0);
                                v1 = fmaf(xp[j * NTX + 1], dp[j], v1);
                            }
                        }
                        lw[(mm * a.K + k) * NTP + np] = pack_bf16x2(v0, v1);
                    }
                } else if constexpr (BF) {
                    for (int e = tid; e < a.K * NT; e += kFcThreads) {
                        const int nn = e % NT, k = e / NT;
                        const float *xp = xb + mm * a.Csp * NTX + nn;
                        const float *dp = db + (mm * a.K + k) * a.Csp;
                        float v = 0.f;
#pragma unroll
                        for (int j = 0; j < kMaxCsp; ++j)
                            if (j < a.Csp) v = fmaf(xp[j * NTX], dp[j], v);
                        reinterpret_cast<unsigned short *>(lut)[(mm * a.K + k) * NTP + nn] =
                            (unsigned short)(pack_bf16x2(v, 0.f) & 0xffffu);
                    }
                }
            }
            if constexpr (!BF) {
                // fp32: the chunk's (mm, k, nn) entries, flat over the block
                // (several sub-spaces side by side when K * NT < the block);
                // r = mm * K + k is the table row
                const int kl = a.k_log2;
                // 16-image tiles: a warp's 32 entries are 16 images of two rows;
                // rows r and r + 16 (odd pitch 17: bank offsets 16 apart) instead
                // of r and r + 1 (whose banks overlap in one) keep its stores
                // conflict free, when the rows come in whole groups of 32
                const bool rows16 = NT == 16 && ((mch * a.K) & 31) == 0;
                for (int e = tid; e < mch * a.K * NT; e += kFcThreads) {
                    const int nn = e % NT;
                    int r = e / NT;
                    if (rows16) {
                        const int q = e >> 5;
                        r = ((q >> 4) << 5) + (q & 15) + (((e >> 4) & 1) << 4);
                    }
                    const int mm = kl >= 0 ? r >> kl : r / a.K;
                    const float *xp = xb + mm * a.Csp * NTX + nn;
                    const float *dp = db + r * a.Csp;
                    float v = 0.f;
                    if (a.Csp == 4) {  // one 16-byte load of the sub-codeword
                        const float4 d = *reinterpret_cast<const float4 *>(dp);
                        v = fmaf(xp[0], d.x, v);
                        v = fmaf(xp[NTX], d.y, v);
                        v = fmaf(xp[2 * NTX], d.z, v);
                        v = fmaf(xp[3 * NTX], d.w, v);
                    } else {
#pragma unroll
                        for (int j = 0; j < kMaxCsp; ++j)
                            if (j < a.Csp) v = fmaf(xp[j * NTX], dp[j], v);
                    }
                    lut[r * NTP + nn] = v;
                }
            }
        }
        __syncthreads();

        // gather: the lane's 4 codes of sub-space mm, as the bytes of w
        const uint8_t *cb = cs + (size_t)b * a.MCH * a.crb;
        auto gather_mm = [&](int mm, unsigned w) {
                QCNN_CHECK(__vcmpgtu4(w, kmax4) == 0u, QCNN_CHECK_CODE);
                w = __vminu4(w, kmax4);
#pragma unroll
                for (int q = 0; q < kCPL; ++q) {
                    const int code = (int)byte_of(w, q);
                    QCNN_CHECK((mm * a.K + code + 1) * NTP <= a.MCH * a.K * NTP,
                               QCNN_CHECK_TABLE);
                    if constexpr (PAIRS) {
                        const unsigned *row = reinterpret_cast<const unsigned *>(lut) +
                                              (mm * a.K + code) * NTP + nbase / 2;
#pragma unroll
                        for (int i = 0; i < NW / 2; ++i)
                            add_bf16x2(acc[q][2 * i], acc[q][2 * i + 1], row[i]);
                    } else if constexpr (BF) {
                        const unsigned short *row = reinterpret_cast<const unsigned short *>(lut) +
                                                    (mm * a.K + code) * NTP + nbase;
#pragma unroll
                        for (int i = 0; i < NW; ++i) add_bf16(acc[q][i], row[i]);
                    } else {
                        const float *row = lut + (mm * a.K + code) * NTP + nbase;
                        accumulate<NW>(acc[q], [&](int i) { return row[i]; });
                    }
                }
        };
        // (unrolled by 4, not over all kMchMax sub-spaces: the straight-line
        // code of a full unroll missed the instruction cache -- fc6 at batch
        // 1: 13.5 -> 9.4 us under ncu, 1,042 -> 973 instructions per warp)
        if (a.cbits) {  // packed rows: 4 codes of b bits from one funnel shift
            const int cbits = a.cbits, bit0 = lane_ct * cbits;
            const unsigned cmask = (1u << cbits) - 1u;
#pragma unroll 4
            for (int mm = 0; mm < mch; ++mm) {
                const unsigned *cw = reinterpret_cast<const unsigned *>(cb + mm * a.crb);
                const unsigned v = __funnelshift_r(cw[bit0 >> 5], cw[(bit0 >> 5) + 1], bit0 & 31);
                gather_mm(mm, (v & cmask) | (((v >> cbits) & cmask) << 8) |
                                  (((v >> (2 * cbits)) & cmask) << 16) |
                                  (((v >> (3 * cbits)) & cmask) << 24));
            }
        } else {
#pragma unroll 4
            for (int mm = 0; mm < mch; ++mm)
                gather_mm(mm, *reinterpret_cast<const unsigned *>(cb + mm * a.crb + lane_ct));
        }
    }

    // epilogue
    const int ct_lane = ct0 + lane_ct;
    if (a.cl > 1) {
        // the cluster's CTAs (consecutive splits of this tile) add their
        // partial tiles in distributed shared memory, in rank order; with
        // more splits than one cluster, each cluster's sum is a partial for
        // the split reduction
        __syncthreads();  // every warp is done with the table
        float *red = reinterpret_cast<float *>(smem);  // [NT][CT_CTA]
#pragma unroll
        for (int i = 0; i < NW; ++i)
#pragma unroll
            for (int q = 0; q < kCPL; ++q) red[(nbase + i) * CT_CTA + lane_ct + q] = acc[q][i];
        const int group = split / a.cl, groups = a.splits / a.cl;
        cluster_tile_reduce(red, NT * CT_CTA, [&](int e, float v) {
            const int n = n0 + (e >> kCtCtaLog2), ct = ct0 + (e & (CT_CTA - 1));
            if (n >= a.N || ct >= a.Ct) return;
            if (groups > 1) {
                a.partial[((size_t)group * a.N + n) * a.Ct + ct] = v;
            } else {
                v += a.bias ? a.bias[ct] : 0.f;
                if (a.relu) v = fmaxf(v, 0.f);
                a.y[(size_t)n * a.Ct + ct] = v;
            }
        });
        return;
    }
#pragma unroll
    for (int i = 0; i < NW; ++i) {
        const int n = n0 + nbase + i;
        if (n >= a.N) continue;
#pragma unroll
        for (int q = 0; q < kCPL; ++q) {
            const int ct = ct_lane + q;
            if (ct >= a.Ct) continue;
            if (a.splits == 1) {
                float v = acc[q][i] + (a.bias ? a.bias[ct] : 0.f);
                if (a.relu) v = fmaxf(v, 0.f);
                a.y[(size_t)n * a.Ct + ct] = v;
            } else {
                a.partial[((size_t)split * a.N + n) * a.Ct + ct] = acc[q][i];
            }
        }
    }
}

__global__ void fc_reduce_kernel(const float *partial, int splits, int N, int Ct,
                                 const float *__restrict__ bias, int relu, float *__restrict__ y) {
    grid_dep_sync();
    const size_t total = (size_t)N * Ct;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (size_t)gridDim.x * blockDim.x) {
        float v = 0.f;
        // (unrolled: the loads of up to 16 splits in flight at once, added in order)
#pragma unroll 16
        for (int s = 0; s < splits; ++s) v += partial[(size_t)s * total + i];
        if (bias) v += bias[i % Ct];
        if (relu) v = fmaxf(v, 0.f);
        y[i] = v;
    }
}

// Few outputs, many splits (batch 1): one warp per output; lane l adds the
// splits l, l + 32, ... in order, then a fixed butterfly adds the lanes.
__global__ void fc_reduce_warp_kernel(const float *partial, int splits, int N, int Ct,
                                      const float *__restrict__ bias, int relu,
                                      float *__restrict__ y) {
    grid_dep_sync();
    const size_t total = (size_t)N * Ct;
    const int lane = threadIdx.x & 31;
    for (size_t i = ((size_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < total;
         i += ((size_t)gridDim.x * blockDim.x) >> 5) {
        float v = 0.f;
        for (int s = lane; s < splits; s += 32) v += partial[(size_t)s * total + i];
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0) {
            if (bias) v += bias[i % Ct];
            if (relu) v = fmaxf(v, 0.f);
            y[i] = v;
        }
    }
}

// eff: measured gather throughput relative to the (NW 4, WN 1) tile (GB300,
// AlexNet fc6-fc8 at batch 128).  The (16, 1) tile -- 16 images per lane
// across all 1024 outputs of the CTA, so each code and each staged code row
// serves 16 images -- runs fc6 / fc7 1.3x / 1.2x faster than (4, 1).
struct FcVariant {
    int NW, WN, MINB, BF;
    double eff;
    void (*fn)(FcArgs);
};
#define QCNN_FC(NW, WN, MB, EFF) {NW, WN, MB, 0, EFF, fc_fused_kernel<NW, WN, MB, false>}
#define QCNN_FC_BF(NW, WN, MB, EFF) {NW, WN, MB, 1, EFF, fc_fused_kernel<NW, WN, MB, true>}
static const FcVariant kFcVariants[] = {
    QCNN_FC(16, 2, 2, 0.8),   QCNN_FC(8, 2, 3, 0.84),   QCNN_FC(8, 4, 3, 0.6),
    QCNN_FC(4, 1, 3, 1.0),    QCNN_FC(1, 1, 3, 0.5),    QCNN_FC_BF(16, 2, 2, 0.8),
    QCNN_FC_BF(8, 2, 3, 0.84), QCNN_FC_BF(8, 4, 3, 0.6), QCNN_FC_BF(4, 1, 3, 1.0),
    QCNN_FC_BF(1, 1, 3, 0.5), QCNN_FC(16, 1, 2, 1.2),  QCNN_FC_BF(16, 1, 2, 1.2),
};
#undef QCNN_FC_BF
#undef QCNN_FC
constexpr int kNumFc = sizeof(kFcVariants) / sizeof(kFcVariants[0]);

// odd table-row pitch in the unit the kernel indexes (see FcArgs::NTP)
static int fc_ntp(int NT, int bf16) { return (bf16 && NT % 2 == 0 ? NT / 2 : NT) | 1; }

FcPlan plan_fc(const FcShape &s, size_t max_partial_bytes) {
    FcPlan best{};
    double best_t = 1e300;
    const int sms = num_sms();
    const size_t sm_bytes = 228 * 1024;
#ifdef QCNN_TUNING  // tuning builds only: force a variant, split count, chunk or cluster
    const char *force_env = getenv("QCNN_FC_VARIANT");
    const int force = force_env ? atoi(force_env) : -1;
    const char *sp_env = getenv("QCNN_FC_SPLITS");
    const char *mch_env = getenv("QCNN_FC_MCH");
    const char *cl_env = getenv("QCNN_FC_CLUSTER");
#endif
    for (int v = 0; v < kNumFc; ++v) {
#ifdef QCNN_TUNING
        if (force >= 0 && v != force) continue;
#endif
        const FcVariant &fv = kFcVariants[v];
        if (fv.BF != s.bf16) continue;
        const int NT = fv.NW * fv.WN;
        const int CT_CTA = (8 / fv.WN) * 32 * kCPL;
        const int NTP = fc_ntp(NT, fv.BF), NTX = NT | 1;
        const int row_bytes = fc_row_bytes(NT, NTP, fv.BF);
        // largest chunk that lets MINB CTAs share an SM
        int MCH = std::min(kMchMax, std::max(1, 512 / s.K));
#ifdef QCNN_TUNING
        if (mch_env) MCH = std::max(1, std::min(kMchMax, atoi(mch_env)));
#endif
        while (MCH > 1 &&
               (fc_smem_layout(MCH, s.K, row_bytes, NTX, s.Csp, CT_CTA).total + 1024) *
                       fv.MINB > sm_bytes)
            --MCH;
        const size_t smem = fc_smem_layout(MCH, s.K, row_bytes, NTX, s.Csp, CT_CTA).total;
        if (smem > 200 * 1024) continue;
        const int cps_sm = std::max(1, std::min(fv.MINB, (int)(sm_bytes / (smem + 1024))));
        const int n_chunks = cdiv(s.M, MCH);
        const int n_tiles = cdiv(s.N, NT), ct_tiles = cdiv(s.Ct, CT_CTA);
        const int tiles = n_tiles * ct_tiles;
        const int target = 2 * sms * cps_sm;
        int splits = std::max(1, std::min(n_chunks, (int)std::lround((double)target / tiles)));
        // 16-image tiles: at least two chunks per CTA (measured: fc8 at batch
        // 128, 64 chunks, 32 splits 39.6 us against 47.8 us with 64; at batch
        // 64 37.6 against 41.6 us).  Single-image tiles keep one chunk per CTA
        // (fc6-8 at batch 1 are fastest with every chunk on its own CTA).
        if (NT >= 16) splits = std::min(splits, std::max(1, n_chunks / 2));
#ifdef QCNN_TUNING
        if (sp_env) splits = std::max(1, std::min(n_chunks, atoi(sp_env)));
#endif
        // at most max_partial_bytes of partial sums [splits][N][Ct]
        const size_t per_split = (size_t)s.N * s.Ct * sizeof(float);
        const size_t cap = max_partial_bytes / per_split;
        if (splits > 1 && (size_t)splits > cap) splits = cap >= 2 ? (int)cap : 1;
        const int cpsplit = cdiv(n_chunks, splits);
        splits = cdiv(n_chunks, cpsplit);
        // Many splits of several tiles of few images: clusters of 8 CTAs add
        // their partial tiles in distributed shared memory, so an eighth of
        // the partial sums goes through the workspace.  Measured (clusters /
        // none): fc6 batch 1 (144 splits, 4 tiles) 17.0 / 19.5 us, fc6 batch
        // 8 36.9 / 39.0 us, fc7 batch 8 24.0 / 27.8 us; no change for fc7
        // batch 1 and fc8 batch 8.  With a single tile (fc8 batch 1: 12.6 /
        // 11.2 us), fewer splits (fc7 batch 64, 32 splits: 70.7 / 68.1 us) or
        // 16-image tiles (64 KB of partial sums per CTA through distributed
        // shared memory; fc8 batch 128: 46.8 / 43.0 us in the whole step) the
        // cluster's scheduling constraint, barriers and remote reads cost
        // more than the partial sums they save.
        int cl = 1;
        if (splits >= 64 && tiles >= 2 && NT <= 4 && (size_t)NT * CT_CTA * sizeof(float) <= smem) {
            for (int c = 8; c >= 2 && cl == 1; c /= 2)
                if (splits % c == 0 &&
                    cluster_capacity(reinterpret_cast<const void *>(fv.fn), kFcThreads, c, smem) >= 1)
                    cl = c;
        }
#ifdef QCNN_TUNING
        if (cl_env) {
            const int c = atoi(cl_env);
            if (c < 1 || splits % c != 0 ||
                (c > 1 && ((size_t)NT * CT_CTA * sizeof(float) > smem ||
                           cluster_capacity(reinterpret_cast<const void *>(fv.fn), kFcThreads, c,
                                            smem) < 1)))
                continue;
            cl = c;
        }
#endif
        double slots = (double)cps_sm * sms;
        if (cl > 1)
            slots = std::min(slots, (double)cl * cluster_capacity(reinterpret_cast<const void *>(fv.fn),
                                                                   kFcThreads, cl, smem));
        const double ctas = (double)tiles * splits;
        const double waves = std::ceil(ctas / slots);
        // one CTA: shared-memory wavefronts (gather + build) per chunk; a wave
        // of cps_sm co-resident CTAs shares one SM
        const double per_chunk = (double)MCH * NT * CT_CTA / (fv.BF && fv.NW % 2 == 0 ? 64.0 : 32.0) +
                                 (double)MCH * s.K * NT / 32.0 * 2;
        const double t_smem = waves * cpsplit * per_chunk * cps_sm / 1.2e9 / fv.eff;
        // (byte codes counted for both code layouts, so that packed and
        // unpacked calls make the same plan and share one workspace query)
        const int parts = splits / cl;
        const double bytes = (double)s.M * s.Ct * n_tiles + 4.0 * s.N * s.Cs * ct_tiles +
                             (parts > 1 ? 8.0 * parts * s.N * s.Ct : 0.0);
        const double t = std::max(t_smem, bytes / 6.0e12) + (parts > 1 ? 3e-6 : 0.0);
        if (t < best_t) {
            best_t = t;
            best.variant = v;
            best.NT = NT;
            best.CT_CTA = CT_CTA;
            best.MCH = MCH;
            best.n_chunks = n_chunks;
            best.splits = splits;
            best.cl = cl;
            best.chunks_per_split = cpsplit;
            best.n_tiles = n_tiles;
            best.ct_tiles = ct_tiles;
            best.smem = smem;
            best.partial_bytes = parts > 1 ? (size_t)parts * per_split : 0;
        }
    }
    return best;
}

qcnn_status launch_fc(const FcShape &s, const FcPlan &p, const float *x, const float *D,
                      const uint8_t *codes, const float *bias, float *y, int relu,
                      float *partial_ws, cudaStream_t st, const PartialInput *xin,
                      bool leave_partials) {
    const FcVariant &fv = kFcVariants[p.variant];
    FcArgs a;
    a.x = x;
    a.D = D;
    a.codes = codes;
    a.bias = bias;
    a.y = y;
    a.partial = partial_ws;
    a.N = s.N;
    a.Cs = s.Cs;
    a.Ct = s.Ct;
    a.Csp = s.Csp;
    a.K = s.K;
    a.M = s.M;
    a.NT = p.NT;
    a.CT_CTA = p.CT_CTA;
    a.MCH = p.MCH;
    a.n_chunks = p.n_chunks;
    a.chunks_per_split = p.chunks_per_split;
    a.splits = p.splits;
    a.relu = relu;
    const uintptr_t base = reinterpret_cast<uintptr_t>(codes);
    a.cvec = (s.Ct % 16 == 0 && base % 16 == 0) ? 16
             : (s.Ct % 8 == 0 && base % 8 == 0) ? 8
             : (s.Ct % 4 == 0 && base % 4 == 0) ? 4
                                                 : 0;
    a.cbits = s.code_bits;
    a.cpitch = s.code_bits ? (int)fc_packed_pitch(s.Ct, s.K) : 0;
    a.crb = p.CT_CTA + 16;
    a.cch_log2 = 0;
    while ((1 << a.cch_log2) < p.MCH * s.Csp) ++a.cch_log2;
    a.early = 1;  // no kernel of a library call writes D or the codes
    a.xpart = xin ? xin->part : nullptr;
    a.xbias = xin ? xin->bias : nullptr;
    a.xgroups = xin ? xin->groups : 0;
    a.xrelu = xin ? xin->relu : 0;
    a.dvec16 = (s.K * s.Csp) % 4 == 0 && reinterpret_cast<uintptr_t>(D) % 16 == 0;
    a.k_log2 = -1;
    for (int b = 0; b < 9; ++b)
        if (s.K == 1 << b) a.k_log2 = b;
    a.cl = p.cl;
    cudaError_t e =
        cudaFuncSetAttribute(fv.fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem);
    if (e == cudaSuccess && p.cl > 8)
        e = cudaFuncSetAttribute(fv.fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return cuda_status(e);
    const dim3 grid(p.ct_tiles, p.n_tiles, p.splits);
    const dim3 cluster = p.cl > 1 ? dim3(1, 1, p.cl) : dim3(0, 0, 0);
    qcnn_status rc = launch_k(fv.fn, grid, dim3(kFcThreads), p.smem, st, cluster, a);
    const int groups = p.splits / p.cl;  // partial sums per output left
    if (rc != QCNN_OK || groups == 1 || leave_partials) return rc;
    const size_t total = (size_t)s.N * s.Ct;
    const int blocks = (int)std::min<size_t>((total + 255) / 256, (size_t)num_sms() * 8);
    if (total < 65536 && groups >= 16) {
        const int wblocks = (int)std::min<size_t>((total * 32 + 255) / 256, (size_t)num_sms() * 16);
        return launch_pdl(fc_reduce_warp_kernel, dim3(wblocks), dim3(256), 0, st,
                          static_cast<const float *>(partial_ws), groups, s.N, s.Ct, bias, relu,
                          y);
    }
    return launch_pdl(fc_reduce_kernel, dim3(blocks), dim3(256), 0, st,
                      static_cast<const float *>(partial_ws), groups, s.N, s.Ct, bias, relu, y);
}

}  // namespace qcnn
