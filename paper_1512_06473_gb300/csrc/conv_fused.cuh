// conv_fused.cuh -- the fused stride-1 conv kernel (Sec. 3.2, Eq. 7) and its
// tile-variant table entries, shared by the units that instantiate the
// variants (conv_fused_*.cu, compiled in parallel) and by conv.cu, which
// plans and launches them.  See conv.cu for the algorithm.
#pragma once

#include "qcnn_internal.cuh"

namespace qcnn {

// ==================================================================== fused
struct ConvFusedArgs {
    const float *__restrict__ x;
    const float *__restrict__ D;
    const uint8_t *__restrict__ codes;  // packed [M][kk][CtP]
    const float *__restrict__ bias;
    float *__restrict__ y;
    int N, Cs, H, W, Ct, kh, kw, pad, Csp, K, M, Ho, Wo;
    int pitch, ST, KS, HP, CtP, relu;  // ST: output positions per tile
    int xs_floats;  // floats of one x staging buffer (HP rounded up, times CSP4)
    int splits, m_per_split;    // sub-space ranges over several CTAs (small batches)
    int cl;                     // the splits of a tile form clusters of cl CTAs (1: none)
    float *__restrict__ partial;  // [splits / cl][N][Ct][Ho][Wo] when splits > cl
    // stream-K schedule (large batches): CTA c takes the (tile, sub-space)
    // units [u0, u1), u = tile * M + m, sk_base units each plus one for the
    // first sk_extra CTAs; tile = (n * ct_tiles + ct_tile) * pos_tiles + pos.
    // A tile whose units fall to several CTAs leaves one partial piece per
    // CTA, [CT_CTA][ST] over the tile's positions: partial[c][1] from the
    // CTA that began it (its head), partial[c][0] from each later one (a
    // middle part or its tail)
    int sk, sk_base, sk_extra, pos_tiles, ct_tiles;
    // 1: D and the packed codes are the caller's and no kernel of the same
    // call writes them, so the first sub-space's D and codes are staged
    // before the wait on the previous kernel (programmatic dependent launch),
    // their fetch overlapping that kernel's tail; only x waits
    int early;
};

// Shared memory carve-up of the fused kernel (byte offsets, 16-aligned);
// nlut = 2 table buffers when the sub-spaces are software pipelined.  With
// the tensor-core build (tc_rows > 0: halo positions rounded up to whole
// 128-row MMA tiles), the staging buffers hold the operands in the tensor
// core's K-major layout, plus the low halves of the 3xTF32 split (alo,
// blo), the mbarrier of the MMAs and the tensor-memory address.
struct FusedSmem {
    size_t lut, xs, ds, cs, alo, blo, bar, total;
};
__host__ __device__ inline FusedSmem fused_smem_layout(int K, int KS, int xs_floats, int csp4,
                                                       int kk, int ct_cta, int nlut,
                                                       int tc_rows = 0) {
    FusedSmem s;
    s.lut = 0;
    s.xs = ((size_t)nlut * K * KS * 4 + 15) / 16 * 16;
    s.ds = s.xs + (size_t)2 * xs_floats * 4;
    s.cs = s.ds + (size_t)2 * K * csp4 * 4;
    s.alo = s.cs + ((size_t)2 * kk * ct_cta + 15) / 16 * 16;
    s.blo = s.alo + (size_t)tc_rows * csp4 * 4;
    s.bar = s.blo + (tc_rows ? (size_t)K * csp4 * 4 : 0);
    s.total = s.bar + (tc_rows ? 16 : 0);
    return s;
}

// Offset (in floats) of element j of row r of a K-major tf32 operand with
// 8 elements per row, in the tensor core's layout without swizzle: core
// matrices of 8 rows x 4 elements (128 bytes), the two along K 128 bytes
// apart, groups of 8 rows 256 bytes apart.
__host__ __device__ inline int tc_off(int r, int j) {
    return ((r >> 3) * 2 + (j >> 2)) * 32 + (r & 7) * 4 + (j & 3);
}

// Load CTW consecutive code bytes (16-byte aligned in shared memory).
template <int CTW>
__device__ __forceinline__ void load_code_words(const uint8_t *p, unsigned (&w)[CTW / 4]) {
    if constexpr (CTW % 16 == 0) {
#pragma unroll
        for (int i = 0; i < CTW / 16; ++i) {
            const uint4 v = reinterpret_cast<const uint4 *>(p)[i];
            w[4 * i + 0] = v.x;
            w[4 * i + 1] = v.y;
            w[4 * i + 2] = v.z;
            w[4 * i + 3] = v.w;
        }
    } else if constexpr (CTW == 8) {
        const uint2 v = *reinterpret_cast<const uint2 *>(p);
        w[0] = v.x;
        w[1] = v.y;
    } else {
        static_assert(CTW == 4, "CTW must be 4, 8 or a multiple of 16");
        w[0] = *reinterpret_cast<const unsigned *>(p);
    }
}

// P     : 32-position slots per warp
// CTW   : output channels per warp
// WP    : warps along positions (NW / WP warps along channels)
// CSP4  : C'_s rounded up to 4 or 8 (register width of one sub-vector)
// NW    : warps per CTA (8, 16 or 32)
// MINB  : CTAs per SM the register budget is sized for
// PIPE  : two table buffers; sub-space m+1's table is built while m is
//         gathered, with one barrier per sub-space instead of two
// BF    : bfloat16 pair tables; a slot is then 64 positions (2 per lane)
// SK    : stream-K schedule (a persistent grid over (tile, sub-space) units)
// TC    : table build on the tensor cores (tcgen05.mma kind::tf32, 3xTF32):
//         positions x C'_s times C'_s x K per sub-space, accumulators in
//         tensor memory, stored to the table by all warps
template <int P, int CTW, int WP, int CSP4, int NW, int MINB, bool PIPE, bool BF, bool SK,
          bool TC = false>
__global__ void __launch_bounds__(NW * 32, MINB) conv_fused_kernel(const ConvFusedArgs a) {
    static_assert(!SK || !PIPE, "the stream-K schedule has one table buffer");
    static_assert(!TC || (CSP4 == 8 && !PIPE && !BF),
                  "tensor-core build: fp32 tables, C'_s width 8, one table buffer");
    constexpr int NT = NW * 32;
    constexpr int E = BF ? 2 : 1;  // positions per lane and slot
    constexpr int CT_CTA = (NW / WP) * CTW;
    constexpr int Q16 = CT_CTA / 16;
    constexpr int ST = WP * P * 32 * E;  // output positions per tile
    // sub-codewords per lane per build pass (fewer under a 64-register budget)
    constexpr int QB = (NW * MINB >= 32 ? 8 : 16) / CSP4;
    static_assert(CT_CTA % 16 == 0, "channel tile must be a multiple of 16");
    extern __shared__ __align__(16) unsigned char smem[];
    const int kk = a.kh * a.kw;
    const int K = a.K, KS = a.KS, HP = a.HP, pitch = a.pitch;
    const int tc_rows = TC ? a.xs_floats / CSP4 : 0;  // whole 128-row MMA tiles
    const FusedSmem L =
        fused_smem_layout(K, KS, a.xs_floats, CSP4, kk, CT_CTA, PIPE ? 2 : 1, tc_rows);
    float *lut0 = reinterpret_cast<float *>(smem + L.lut);
    float *xs = reinterpret_cast<float *>(smem + L.xs);
    float *ds = reinterpret_cast<float *>(smem + L.ds);
    uint8_t *cs = smem + L.cs;
    // (the tensor-core variants allocate tensor memory, which the kernel
    // before may still hold: they wait first)
    const bool early = !TC && a.early;
    if (!early) grid_dep_sync();

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int wp = warp % WP, wc = warp / WP;
    const int split = SK ? 0 : blockIdx.z % a.splits;
    // tile being staged (sn, sl0, sct0) and tile being computed (cn, cl0, cct0):
    // image, first output position, first channel
    int sn = blockIdx.z / a.splits, sl0 = blockIdx.x * ST, sct0 = blockIdx.y * CT_CTA;
    const int HW = a.H * a.W;

    // stream-K unit uu -> its tile: image n, first position l0, first channel ct0
    auto tile_of = [&](long long uu, int &n, int &l0, int &ct0) {
        const long long t = uu / a.M;
        n = (int)(t / ((long long)a.ct_tiles * a.pos_tiles));
        const int rest = (int)(t - (long long)n * a.ct_tiles * a.pos_tiles);
        ct0 = (rest / a.pos_tiles) * CT_CTA;
        l0 = (rest % a.pos_tiles) * ST;
    };
    long long u = 0, u1 = 0;  // stream-K unit range
    if constexpr (SK) {
        const int c = blockIdx.x;
        u = (long long)c * a.sk_base + min(c, a.sk_extra);
        u1 = u + a.sk_base + (c < a.sk_extra ? 1 : 0);
        tile_of(u, sn, sl0, sct0);
    }
    int cn = sn, cl0 = sl0, cct0 = sct0;
    if (a.Csp < CSP4) {
        for (int e = tid; e < 2 * a.xs_floats; e += NT) xs[e] = 0.f;
        for (int e = tid; e < 2 * K * CSP4; e += NT) ds[e] = 0.f;
    }
    // tensor-core build: tensor memory for the accumulators of every
    // 128-position tile (K columns each), one mbarrier for the MMAs
    uint64_t *tc_bar = reinterpret_cast<uint64_t *>(smem + L.bar);
    unsigned *tc_slot = reinterpret_cast<unsigned *>(smem + L.bar + 8);
    if constexpr (TC) {
        if (warp == 0) tmem_alloc(tc_slot, 512u);
        if (tid == 0) {
            mbar_init(tc_bar, 1);
            asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
        }
    }
    __syncthreads();

    // ---- asynchronous staging (callers commit) --------------------------
    // Inputs of sub-space m for the halo of the tile (image n, first
    // position l0): halo position h is input (iy, ix) = (r - pad, c - pad)
    // with l0 + h = r*pitch + c, zero-filled where that falls in the padding;
    // sub-vector slots j >= C'_s stay zero.
    auto stage_x = [&](int m, int b, int n, int l0) {
        float *xb = xs + b * a.xs_floats;
        const float *xn = a.x + ((size_t)n * a.Cs + (size_t)m * a.Csp) * HW;
        for (int h = tid; h < HP; h += NT) {
            const int g = l0 + h, r = g / pitch, c = g - r * pitch;
            const int iy = r - a.pad, ix = c - a.pad;
            const bool ok = iy >= 0 && iy < a.H && ix >= 0 && ix < a.W;
            const float *src = ok ? xn + iy * a.W + ix : a.x;
            for (int j = 0; j < a.Csp; ++j)
                cp_async4(xb + (TC ? tc_off(h, j) : h * CSP4 + j),
                          ok ? src + (size_t)j * HW : a.x, ok);
        }
    };
    auto stage_d = [&](int m, int b) {
        float *db = ds + b * K * CSP4;
        const float *dm = a.D + (size_t)m * K * a.Csp;
        for (int k = tid; k < K; k += NT)
            for (int j = 0; j < a.Csp; ++j)
                cp_async4(db + (TC ? tc_off(k, j) : k * CSP4 + j), dm + k * a.Csp + j, true);
    };
    auto stage_xd = [&](int m, int b, int n, int l0) {
        stage_x(m, b, n, l0);
        stage_d(m, b);
    };
    // codes of sub-space m, channels ct0 ..; 16-byte pieces past the packed
    // row (CtP, a multiple of 256, may be short of the last tile) are zeros
    auto stage_codes = [&](int m, int b, int ct0) {
        uint8_t *cb = cs + (size_t)b * kk * CT_CTA;
        const uint8_t *cm = a.codes + (size_t)m * kk * a.CtP + ct0;
        for (int e = tid; e < kk * Q16; e += NT) {
            const int pk = e / Q16, q = e % Q16;
            if (ct0 + q * 16 < a.CtP)
                cp_async16(cb + pk * CT_CTA + q * 16, cm + (size_t)pk * a.CtP + q * 16);
            else
                *reinterpret_cast<uint4 *>(cb + pk * CT_CTA + q * 16) = make_uint4(0, 0, 0, 0);
        }
    };
    // first stage of the CTA (sub-space m, and m+1's D and x when m2 is
    // set): the constants first, then the wait on the previous kernel
    auto stage_first = [&](int m, bool m2, int n, int l0, int ct0) {
        stage_d(m, 0);
        if (m2) stage_d(m + 1, 1);
        stage_codes(m, 0, ct0);
        if (early) grid_dep_sync();
        stage_x(m, 0, n, l0);
        if (m2) stage_x(m + 1, 1, n, l0);
        cp_async_commit();
    };

    // ---- build: lut[k][h] = <x(h), D[m][k]>; lanes on k, warps on h -------
    const int hpw = cdiv(HP, NW);
    const int h0 = warp * hpw, h1 = min(HP, h0 + hpw);
    auto build = [&](int b, float *lut) {
        const float *xb = xs + b * a.xs_floats;
        const float *db = ds + b * K * CSP4;
        for (int q0 = 0; q0 < K; q0 += 32 * QB) {
            float dk[QB][CSP4];
#pragma unroll
            for (int i = 0; i < QB; ++i) {
                const int k = min(q0 + 32 * i + lane, K - 1);
#pragma unroll
                for (int j = 0; j < CSP4; j += 4) {
                    const float4 v = *reinterpret_cast<const float4 *>(db + k * CSP4 + j);
                    dk[i][j] = v.x;
                    dk[i][j + 1] = v.y;
                    dk[i][j + 2] = v.z;
                    dk[i][j + 3] = v.w;
                }
            }
            for (int h = h0; h < h1; ++h) {
                float xv[CSP4];
#pragma unroll
                for (int j = 0; j < CSP4; j += 4) {
                    const float4 v = *reinterpret_cast<const float4 *>(xb + h * CSP4 + j);
                    xv[j] = v.x;
                    xv[j + 1] = v.y;
                    xv[j + 2] = v.z;
                    xv[j + 3] = v.w;
                }
#pragma unroll
                for (int i = 0; i < QB; ++i) {
                    const int k = q0 + 32 * i + lane;
                    float v = 0.f;
#pragma unroll
                    for (int j = 0; j < CSP4; ++j) v = fmaf(xv[j], dk[i][j], v);
                    if (k < K) lut[k * KS + h] = v;
                }
            }
        }
    };
    // bfloat16 pair tables: a lane walks its warp's positions in order and,
    // at position h, writes the word (t[h-1], t[h]) into copy (h-1) & 1.  The
    // walk starts one position early (the left neighbour of the range) and
    // the last range runs one past HP with a zero entry, so every pair
    // (q, q+1), 0 <= q < HP, is written exactly once.
    auto build_bf16 = [&](int b, float *lut) {
        if (h0 >= HP) return;
        const float *xb = xs + b * a.xs_floats;
        const float *db = ds + b * K * CSP4;
        unsigned *w = reinterpret_cast<unsigned *>(lut);
        const int RW = KS >> 1;  // words per row of one copy (odd)
        const int hs = max(h0 - 1, 0), he = h1 == HP ? HP + 1 : h1;
        for (int q0 = 0; q0 < K; q0 += 32 * QB) {
            float dk[QB][CSP4];
#pragma unroll
            for (int i = 0; i < QB; ++i) {
                const int k = min(q0 + 32 * i + lane, K - 1);
#pragma unroll
                for (int j = 0; j < CSP4; j += 4) {
                    const float4 v = *reinterpret_cast<const float4 *>(db + k * CSP4 + j);
                    dk[i][j] = v.x;
                    dk[i][j + 1] = v.y;
                    dk[i][j + 2] = v.z;
                    dk[i][j + 3] = v.w;
                }
            }
            float prev[QB];
            for (int h = hs; h < he; ++h) {
                float xv[CSP4];
#pragma unroll
                for (int j = 0; j < CSP4; j += 4) {
                    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (h < HP) v = *reinterpret_cast<const float4 *>(xb + h * CSP4 + j);
                    xv[j] = v.x;
                    xv[j + 1] = v.y;
                    xv[j + 2] = v.z;
                    xv[j + 3] = v.w;
                }
                const int q = h - 1;
                unsigned *wq = w + (q & 1) * K * RW + (q >> 1);
#pragma unroll
                for (int i = 0; i < QB; ++i) {
                    const int k = q0 + 32 * i + lane;
                    float v = 0.f;
#pragma unroll
                    for (int j = 0; j < CSP4; ++j) v = fmaf(xv[j], dk[i][j], v);
                    if (h > hs && k < K) wq[k * RW] = pack_bf16x2(prev[i], v);
                    prev[i] = v;
                }
            }
        }
    };

    // ---- tensor-core build (TC): T[h][k] = sum_j x(h)[j] D[m][k][j] as the
    // product of the positions x C'_s operand A and the C'_s x K operand B
    // (3xTF32: A_hi B_hi + A_hi B_lo + A_lo B_hi, each tf32 product exact,
    // accumulated in fp32 -- the fp32 accuracy of the FFMA build), one MMA of
    // 128 positions x K codewords per tile and term; then every warp moves
    // its tensor-memory lane quarter to the table, lut[k][h].
    unsigned tc_phase = 0;
    bool tc_failed = false;  // a wait gave up: no further MMAs or waits (bounded time)
    auto build_tc = [&](int b, float *lut) {
        float *ab = xs + b * a.xs_floats;  // raw fp32 A, split in place to A_hi
        float *bb = ds + b * K * CSP4;     // raw fp32 B -> B_hi
        float *al = reinterpret_cast<float *>(smem + L.alo);
        float *bl = reinterpret_cast<float *>(smem + L.blo);
        for (int e = tid; e < tc_rows * CSP4; e += NT) {
            const float v = ab[e], hi = tf32_hi(v);
            ab[e] = hi;
            al[e] = v - hi;  // exact
        }
        for (int e = tid; e < K * CSP4; e += NT) {
            const float v = bb[e], hi = tf32_hi(v);
            bb[e] = hi;
            bl[e] = v - hi;
        }
        fence_async_smem();
        tc_fence_before_sync();
        __syncthreads();
        const unsigned tbase = *tc_slot;
        const int n_mt = tc_rows / 128;
        if (tid == 0 && !tc_failed) {
            tc_fence_after_sync();
            const uint32_t idesc = idesc_tf32(128, K);
            const uint64_t bh = smem_desc_kmajor(bb, 128, 256), blw = smem_desc_kmajor(bl, 128, 256);
            for (int t = 0; t < n_mt; ++t) {
                const uint64_t ah = smem_desc_kmajor(ab + t * 128 * CSP4, 128, 256);
                const uint64_t alw = smem_desc_kmajor(al + t * 128 * CSP4, 128, 256);
                const unsigned d = tbase + (unsigned)(t * K);
                mma_tf32(d, ah, bh, idesc, false);
                mma_tf32(d, ah, blw, idesc, true);
                mma_tf32(d, alw, bh, idesc, true);
            }
            mma_commit(tc_bar);
        }
        if (!tc_failed) {
            const bool done = mbar_wait_bounded(tc_bar, tc_phase, 1u << 20);
            tc_phase ^= 1u;
            // the same decision in every thread of the CTA
            tc_failed = __syncthreads_or(!done) != 0;
            if (tid == 0) QCNN_RECORD_IF(tc_failed, QCNN_CHECK_TIMEOUT);
        }
        tc_fence_after_sync();
        const int q = warp & 3, chunks = K / 32;
        for (int u = warp >> 2; u < n_mt * chunks; u += NW / 4) {
            const int t = u / chunks, c0 = (u - t * chunks) * 32;
            const int h = t * 128 + q * 32 + lane;
            float v[32];
            tmem_ld32(tbase + ((unsigned)(q * 32) << 16) + (unsigned)(t * K + c0), v);
            if (h < HP) {
#pragma unroll
                for (int j = 0; j < 32; ++j) lut[(c0 + j) * KS + h] = v[j];
            }
        }
        tc_fence_before_sync();
    };

    // ---- gather: acc[c][p] += lut[code(c, pk)][pos(p) + ky*pitch + kx] -----
    float acc[CTW][P * E];
#pragma unroll
    for (int c = 0; c < CTW; ++c)
#pragma unroll
        for (int p = 0; p < P * E; ++p) acc[c][p] = 0.f;
    // byte offset of the lane's first word (fp32: position; bf16: pair)
    const int lane_off4 = (wp * P * 32 + lane) * 4;
    const int KS4 = (BF ? KS >> 1 : KS) * 4;  // bytes between rows k and k+1
    const unsigned kmax4 = (unsigned)(K - 1) * 0x01010101u;  // clamp codes into [0, K)
    auto gather = [&](int b, const float *lut) {
        const unsigned char *lutb = reinterpret_cast<const unsigned char *>(lut);
        const uint8_t *cb = cs + (size_t)b * kk * CT_CTA + wc * CTW;
        for (int ky = 0; ky < a.kh; ++ky) {
            for (int kx = 0; kx < a.kw; ++kx) {
                const int pk = ky * a.kw + kx;
                unsigned w[CTW / 4];
                load_code_words<CTW>(cb + pk * CT_CTA, w);
#pragma unroll
                for (int i = 0; i < CTW / 4; ++i) {
                    QCNN_CHECK(__vcmpgtu4(w[i], kmax4) == 0u, QCNN_CHECK_CODE);
                    w[i] = __vminu4(w[i], kmax4);
                }
                const int off = ky * pitch + kx;
                const int base4 =
                    BF ? lane_off4 + (off >> 1) * 4 + (off & 1) * K * KS4 : lane_off4 + off * 4;
#pragma unroll
                for (int c = 0; c < CTW; ++c) {
                    const unsigned code = byte_of(w[c >> 2], c & 3);
                    QCNN_CHECK((int)code * KS4 + base4 + (P - 1) * 128 + 4 <= K * KS * 4,
                               QCNN_CHECK_TABLE);
                    const unsigned char *row = lutb + (int)code * KS4 + base4;
                    if constexpr (BF) {
#pragma unroll
                        for (int p = 0; p < P; ++p)
                            add_bf16x2(acc[c][2 * p], acc[c][2 * p + 1],
                                       *reinterpret_cast<const unsigned *>(row + p * 128));
                    } else {
                        accumulate<P>(acc[c], [&](int p) {
                            return *reinterpret_cast<const float *>(row + p * 128);
                        });
                    }
                }
            }
        }
    };

    // ---- epilogue: bias, ReLU, store; or raw partial sums (mode 1: split-M
    // slice `split`; mode 2: stream-K piece `slot` of boundary `bnd`)
    auto store = [&](int mode, int bnd, int slot) {
#pragma unroll
        for (int c = 0; c < CTW; ++c) {
            const int ct = cct0 + wc * CTW + c;
            if (ct >= a.Ct) continue;
            const float bv = a.bias ? a.bias[ct] : 0.f;
#pragma unroll
            for (int p = 0; p < P * E; ++p) {
                const int l = BF ? (wp * P + (p >> 1)) * 64 + 2 * lane + (p & 1)
                                 : (wp * P + p) * 32 + lane;
                const int g = cl0 + l, oy = g / pitch, col = g - oy * pitch;
                if (col < a.Wo && oy < a.Ho) {
                    const size_t o = (((size_t)cn * a.Ct + ct) * a.Ho + oy) * a.Wo + col;
                    QCNN_CHECK(o < (size_t)a.N * a.Ct * a.Ho * a.Wo, QCNN_CHECK_GLOBAL);
                    if (mode == 1) {
                        a.partial[(size_t)split * a.N * a.Ct * a.Ho * a.Wo + o] = acc[c][p];
                    } else if (mode == 2) {
                        const size_t piece = (size_t)CT_CTA * ST;
                        a.partial[((size_t)bnd * 2 + slot) * piece +
                                  (size_t)(wc * CTW + c) * ST + l] = acc[c][p];
                    } else {
                        float v = acc[c][p] + bv;
                        if (a.relu) v = fmaxf(v, 0.f);
                        a.y[o] = v;
                    }
                }
            }
        }
    };

    // sub-spaces [mb, me) of this CTA (all of them unless M is split)
    const int mb = split * a.m_per_split, me = min(a.M, mb + a.m_per_split);
    if constexpr (SK) {
        // ---- stream-K: units [u, u1) in order, u = tile * M + m; the first
        // and last tile of the range may be cut (partial pieces)
        int m = (int)(u % a.M);
        int piece_m0 = m;  // first sub-space of the current piece
        stage_first(m, false, sn, sl0, sct0);
        for (int b = 0;; b ^= 1) {
            cp_async_wait<0>();
            __syncthreads();  // unit u staged; gather of the previous unit finished
            const bool last_of_tile = m == a.M - 1, last_of_range = u + 1 == u1;
            if (!last_of_range) {
                if (last_of_tile) tile_of(u + 1, sn, sl0, sct0);  // the next unit opens a new tile
                const int mn = last_of_tile ? 0 : m + 1;
                stage_xd(mn, b ^ 1, sn, sl0);
                stage_codes(mn, b ^ 1, sct0);
                cp_async_commit();
            }
            if constexpr (TC) build_tc(b, lut0);
            else if constexpr (BF) build_bf16(b, lut0);
            else build(b, lut0);
            __syncthreads();
            gather(b, lut0);
            if (last_of_tile || last_of_range) {
                // whole tile -> y; head of a tile cut at the range end ->
                // piece 1 of this CTA; a middle part or the tail of a tile
                // begun by an earlier CTA -> piece 0 of this CTA
                const bool whole = piece_m0 == 0 && last_of_tile;
                store(whole ? 0 : 2, blockIdx.x, piece_m0 == 0 ? 1 : 0);
                if (last_of_range) break;
#pragma unroll
                for (int c = 0; c < CTW; ++c)
#pragma unroll
                    for (int p = 0; p < P * E; ++p) acc[c][p] = 0.f;
                cn = sn;
                cl0 = sl0;
                cct0 = sct0;
                piece_m0 = 0;
            }
            ++u;
            m = last_of_tile ? 0 : m + 1;
        }
        if constexpr (TC) {
            __syncthreads();  // every warp's last tensor-memory load has completed
            if (warp == 0) tmem_dealloc(*tc_slot, 512u);
        }
        return;
    } else if constexpr (!PIPE) {
        stage_first(mb, false, sn, sl0, sct0);
        for (int m = mb; m < me; ++m) {
            const int b = (m - mb) & 1;
            cp_async_wait<0>();
            __syncthreads();  // stage m visible; gather of m-1 finished everywhere
            if (m + 1 < me) {
                stage_xd(m + 1, b ^ 1, sn, sl0);
                stage_codes(m + 1, b ^ 1, sct0);
                cp_async_commit();
            }
            if constexpr (TC) build_tc(b, lut0);
            else if constexpr (BF) build_bf16(b, lut0);
            else build(b, lut0);
            __syncthreads();
            gather(b, lut0);
        }
    } else {
        float *lut1 = lut0 + (size_t)K * KS;
        stage_first(mb, mb + 1 < me, sn, sl0, sct0);
        cp_async_wait<0>();
        __syncthreads();
        if constexpr (BF) build_bf16(0, lut0);
        else build(0, lut0);
        __syncthreads();
        // Iteration m (b = (m - mb) & 1): table m ready in buffer b, codes m in
        // code buffer b, inputs of m+1 in staging buffer b^1.
        for (int m = mb; m < me; ++m) {
            const int b = (m - mb) & 1;
            if (m + 2 < me) stage_xd(m + 2, b, sn, sl0);
            if (m + 1 < me) stage_codes(m + 1, b ^ 1, sct0);
            cp_async_commit();
            // even warps build first, odd warps gather first: the latency-bound
            // table build of one half overlaps the other half's gather
            auto build_next = [&]() {
                if (m + 1 >= me) return;
                if constexpr (BF) build_bf16(b ^ 1, b ? lut0 : lut1);
                else build(b ^ 1, b ? lut0 : lut1);
            };
            // (one loop of two steps, so that the gather and the build are
            // each inlined once: the two orders as straight code doubled the
            // loop and missed the instruction cache)
#pragma unroll 1
            for (int step = 0; step < 2; ++step) {
                if ((step ^ warp) & 1) gather(b, b ? lut1 : lut0);
                else build_next();
            }
            cp_async_wait<0>();
            __syncthreads();
        }
    }

    if constexpr (!SK) {
        if (a.cl > 1) {
            // the cluster's CTAs (the splits of this tile) add their partial
            // tiles in distributed shared memory; with more splits than one
            // cluster, each cluster's sum is a partial for the split reduction
            __syncthreads();  // every warp is done with the table
            float *red = reinterpret_cast<float *>(smem);  // [CT_CTA][ST]
#pragma unroll
            for (int c = 0; c < CTW; ++c)
#pragma unroll
                for (int p = 0; p < P * E; ++p) {
                    const int l = BF ? (wp * P + (p >> 1)) * 64 + 2 * lane + (p & 1)
                                     : (wp * P + p) * 32 + lane;
                    red[(wc * CTW + c) * ST + l] = acc[c][p];
                }
            const size_t plane = (size_t)a.N * a.Ct * a.Ho * a.Wo;
            const int group = split / a.cl, groups = a.splits / a.cl;
            cluster_tile_reduce(red, CT_CTA * ST, [&](int e, float v) {
                const int ch = e / ST, l = e - ch * ST;
                const int ct = cct0 + ch;
                const int g = cl0 + l, oy = g / pitch, col = g - oy * pitch;
                if (ct >= a.Ct || col >= a.Wo || oy >= a.Ho) return;
                const size_t o = (((size_t)cn * a.Ct + ct) * a.Ho + oy) * a.Wo + col;
                QCNN_CHECK(o < plane, QCNN_CHECK_GLOBAL);
                if (groups > 1) {
                    a.partial[(size_t)group * plane + o] = v;
                } else {
                    v += a.bias ? a.bias[ct] : 0.f;
                    if (a.relu) v = fmaxf(v, 0.f);
                    a.y[o] = v;
                }
            });
        } else {
            store(a.splits > 1 ? 1 : 0, 0, 0);
        }
        if constexpr (TC) {
            __syncthreads();  // every warp's last tensor-memory load has completed
            if (warp == 0) tmem_dealloc(*tc_slot, 512u);
        }
    }
}


// ---------------------------------------------------------- variant table --
// eff: measured gather throughput of the variant relative to the best one
// (GB300, AlexNet conv2-5 and VGG-16 conv3-5 shapes, all lanes counted);
// build: share of the table-build time left exposed (1 = not overlapped).
struct FusedVariant {
    int P, CTW, WP, CSP4, NW, MINB, PIPE, BF, SK;
    double eff, build;
    void (*fn)(ConvFusedArgs);
    int TC = 0;  // table build on the tensor cores
};

#define QCNN_FUSED(P, CTW, WP, C4, NW, MB, PIPE, EFF, BLD) \
    {P, CTW, WP, C4, NW, MB, PIPE, 0, 0, EFF, BLD,          \
     conv_fused_kernel<P, CTW, WP, C4, NW, MB, PIPE, false, false>}
#define QCNN_FUSED_BF(P, CTW, WP, C4, NW, MB, PIPE, EFF, BLD) \
    {P, CTW, WP, C4, NW, MB, PIPE, 1, 0, EFF, BLD,             \
     conv_fused_kernel<P, CTW, WP, C4, NW, MB, PIPE, true, false>}
#define QCNN_FUSED_SK(P, CTW, WP, C4, NW, MB, EFF, BLD) \
    {P, CTW, WP, C4, NW, MB, 0, 0, 1, EFF, BLD,         \
     conv_fused_kernel<P, CTW, WP, C4, NW, MB, false, false, true>}
#define QCNN_FUSED_BF_SK(P, CTW, WP, C4, NW, MB, EFF, BLD) \
    {P, CTW, WP, C4, NW, MB, 0, 1, 1, EFF, BLD,            \
     conv_fused_kernel<P, CTW, WP, C4, NW, MB, false, true, true>}
// tensor-core table build (C'_s 5..8): the build's FMAs leave the SM's FMA
// pipe; its stores to the table remain
#define QCNN_FUSED_TC(P, CTW, WP, NW, EFF, BLD)                                     \
    {P, CTW, WP, 8, NW, 1, 0, 0, 0, EFF, BLD,                                       \
     conv_fused_kernel<P, CTW, WP, 8, NW, 1, false, false, false, true>, 1}
#define QCNN_FUSED_TC_SK(P, CTW, WP, NW, EFF, BLD)                                  \
    {P, CTW, WP, 8, NW, 1, 0, 0, 1, EFF, BLD,                                       \
     conv_fused_kernel<P, CTW, WP, 8, NW, 1, false, false, true, true>, 1}
#define QCNN_FUSED_SET(C4)                                                                       \
    QCNN_FUSED(4, 8, 2, C4, 8, 2, false, 0.45, 1.0), /* small tiles for small batches */        \
    QCNN_FUSED(4, 16, 1, C4, 16, 1, false, 1.0, 1.0), /* 16 warps, 128 registers */             \
    QCNN_FUSED(7, 8, 1, C4, 16, 1, false, 1.0, 1.0),                                             \
    QCNN_FUSED(6, 8, 1, C4, 16, 1, false, 1.0, 1.0), /* a whole 13x13 map (pitch 14) */         \
    QCNN_FUSED(5, 8, 1, C4, 16, 1, false, 1.0, 1.0), /* 27x27 maps in 5 tiles (pitch 29) */     \
    QCNN_FUSED(5, 16, 1, C4, 16, 1, false, 1.0, 1.0),                                            \
    QCNN_FUSED(6, 16, 1, C4, 12, 1, false, 1.0, 1.0), /* 12 warps: 192 channels */              \
    QCNN_FUSED(4, 8, 1, C4, 16, 2, false, 0.83, 1.0), /* 2 x 16 warps, 64 registers */          \
    QCNN_FUSED(8, 4, 1, C4, 32, 1, false, 0.82, 1.0), /* 32 warps, 64 registers */              \
    QCNN_FUSED(7, 4, 1, C4, 32, 1, false, 0.89, 1.0),                                            \
    QCNN_FUSED(4, 8, 1, C4, 32, 1, false, 0.98, 1.0),                                            \
    QCNN_FUSED(2, 32, 1, C4, 16, 1, true, 0.75, 0.3), /* pipelined: two table buffers */         \
    QCNN_FUSED(4, 16, 1, C4, 16, 1, true, 0.85, 0.3),                                             \
    QCNN_FUSED(2, 16, 2, C4, 16, 1, true, 0.7, 0.3),                                             \
    QCNN_FUSED(4, 8, 1, C4, 16, 1, true, 0.8, 0.3)
// bfloat16 tables: slots of 64 positions, so half the slots of the fp32
// tiles cover the same band.  Measured (same shapes): the pair-table build
// costs about 1.3x the fp32 build; pipelined tiles never win (32-warp tiles,
// slower still and short of registers, are not instantiated).
#define QCNN_FUSED_BF_SET(C4)                                                      \
    QCNN_FUSED_BF(2, 8, 2, C4, 8, 2, false, 0.45, 1.3),                            \
    QCNN_FUSED_BF(4, 8, 1, C4, 16, 1, false, 1.0, 1.3),                            \
    QCNN_FUSED_BF(2, 16, 1, C4, 16, 1, false, 0.97, 1.3),                          \
    QCNN_FUSED_BF(4, 8, 1, C4, 16, 1, true, 0.6, 0.4),                             \
    QCNN_FUSED_BF(2, 16, 1, C4, 16, 1, true, 0.6, 0.4)
// stream-K schedules of the tiles that win on grids with a short last wave
// (AlexNet's 27x27 and 13x13 layers), fp32 and bf16 tables
#define QCNN_FUSED_SK_SET(C4)                      \
    QCNN_FUSED_SK(4, 16, 1, C4, 16, 1, 1.0, 1.0),  \
    QCNN_FUSED_SK(7, 8, 1, C4, 16, 1, 1.0, 1.0),   \
    QCNN_FUSED_SK(6, 8, 1, C4, 16, 1, 1.0, 1.0),   \
    QCNN_FUSED_SK(5, 16, 1, C4, 16, 1, 1.0, 1.0),  \
    QCNN_FUSED_SK(6, 16, 1, C4, 12, 1, 1.0, 1.0),  \
    QCNN_FUSED_BF_SK(3, 16, 1, C4, 12, 1, 1.0, 1.3), /* bf16: a whole 13x13 map */ \
    QCNN_FUSED_BF_SK(3, 8, 1, C4, 16, 1, 1.0, 1.3),                               \
    QCNN_FUSED_BF_SK(2, 16, 1, C4, 16, 1, 1.0, 1.3),                              \
    QCNN_FUSED_BF_SK(4, 8, 1, C4, 16, 1, 1.0, 1.3)
// The variant table is assembled from the units in this order (the index of
// a variant is part of the ABI: QCNN_ALGO_FUSED_VARIANT + v).
const FusedVariant *fused_variants_plain(int *n);  // conv_fused_plain.cu
const FusedVariant *fused_variants_bf16(int *n);   // conv_fused_bf16.cu
const FusedVariant *fused_variants_sk(int *n);     // conv_fused_sk.cu
const FusedVariant *fused_variants_tc(int *n);     // conv_fused_tc.cu
const FusedVariant *fused_variants_tc_sk(int *n);  // conv_fused_tc_sk.cu
const FusedVariant *fused_variants_narrow(int *n);  // conv_fused_plain.cu (64-channel tiles)

}  // namespace qcnn
