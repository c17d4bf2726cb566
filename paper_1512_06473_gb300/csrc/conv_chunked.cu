// conv_chunked.cu -- PQ conv response (Eq. 7) for layers whose table rows do
// not fit shared memory whole: any stride, any kernel size, K up to 256.
// Built for AlexNet conv1 (11x11, stride 4, one sub-space of C'_s = 3,
// K = 128), where the K-entry table of every input position of a band of
// output rows would need ~1.5 MB.
//
// One CTA owns an image, a band of TH output rows (all columns) and CT_CTA
// output channels.  For each sub-space m and each chunk of KC sub-codewords
// [k0, k0 + KC) it
//   1. builds the chunk's table of every input position the band reads, in
//      a stride-phase-split layout  lut[kl][ay][ax][r][c]  with
//      iy = (oy0 + r + dymin)*s + ay,  ix = (c + dxmin)*s + ax,
//      so that for a fixed kernel offset the 32 lanes of a warp (consecutive
//      output columns) read 32 consecutive words: conflict free;
//   2. gathers only the (c_t, p_k) pairs whose code lies in the chunk.  Those
//      pairs come from per-(m, c_t) entry lists, counting-sorted by chunk in
//      the workspace by a small prep kernel, each entry being the ready
//      byte offset  4 * (kl*SK + phase*PS + (dy - dymin)*PW + (dx - dxmin)).
// A lane owns P positions of the band's output grid of pitch PW
// (l = r*PW + c, columns c >= Wo are discarded) and CTW channels; its input
// sub-vectors (QPT positions x CSPT channels) stay in registers across the
// chunks of a sub-space.
// bfloat16 tables (BF): a row holds 2-byte entries twice, copy 0 as built
// and copy 1 shifted left by one entry, both SKW words long.  A lane takes
// two neighbouring output columns (2 P positions) and reads one 32-bit word
// per look-up pair: for an entry whose row offset e is even the word
// (e/2 + lane) of copy 0, for an odd e the same word of copy 1.  The prep
// kernel folds the copy choice into the entry's byte offset.
#include "qcnn_internal.cuh"

#include <algorithm>
#include <cmath>

namespace qcnn {

constexpr int kChunkThreads = 512;

struct ChunkGeom {
    int s, pad, kh, kw, TH, PR, PW, PS, SK, NQ, dymin, dymax, dxmin, dxmax, KC, NCH;
    int bf;   // bfloat16 tables
    int SKW;  // bf16: words of one row copy (entries SK <= 2 SKW)
};

// Byte offset of entry e of row kl inside a chunk table.
__host__ __device__ inline unsigned chunk_entry_bytes(const ChunkGeom &g, int kl, int e) {
    if (!g.bf) return 4u * (unsigned)(kl * g.SK + e);
    return 4u * (unsigned)(((e & 1) * g.KC + kl) * g.SKW + (e >> 1));
}

__host__ __device__ inline int floor_div(int a, int b) {
    return (a >= 0) ? a / b : -((-a + b - 1) / b);
}

// Offset (in floats) of kernel offset (ky, kx) inside one table row.
__host__ __device__ inline int chunk_phase_off(const ChunkGeom &g, int ky, int kx) {
    const int ty = ky - g.pad, tx = kx - g.pad;
    const int dy = floor_div(ty, g.s), dx = floor_div(tx, g.s);
    const int ay = ty - dy * g.s, ax = tx - dx * g.s;
    return (ay * g.s + ax) * g.PS + (dy - g.dymin) * g.PW + (dx - g.dxmin);
}

// ------------------------------------------------------------------ prep --
// One CTA per (m, ct), one thread per kernel offset p_k (kk <= kMaxPrepKK):
// entries[m][ct][*] = byte offsets grouped by chunk, in p_k order inside a
// chunk (a stable counting sort, so the gather order -- and the rounding --
// is the same on every call); starts[m][ct][c] = first entry of chunk c.
constexpr int kMaxPrepKK = 1024;

__global__ void chunk_prep_kernel(const uint8_t *__restrict__ codes, int packed, int CtP,
                                  int Ct, int kk, int M, int K, ChunkGeom g,
                                  uint32_t *__restrict__ entries, int *__restrict__ starts) {
    extern __shared__ int psh[];  // wcount[NW][NCH], bstart[NCH + 1]
    grid_dep_sync();
    const int nw = blockDim.x / 32;
    int *wcount = psh, *bstart = psh + nw * g.NCH;
    const int i = blockIdx.x;
    const int m = i / Ct, ct = i % Ct;
    const int pk = threadIdx.x, lane = pk & 31, warp = pk >> 5;
    int code = 0, b = -1;
    if (pk < kk) {
        code = packed ? codes[((size_t)m * kk + pk) * CtP + ct] : codes[((size_t)ct * kk + pk) * M + m];
        QCNN_CHECK(code < K, QCNN_CHECK_CODE);
        code = min(code, K - 1);
        b = code / g.KC;
    }
    for (int e = threadIdx.x; e < nw * g.NCH; e += blockDim.x) wcount[e] = 0;
    __syncthreads();
    const unsigned same = __match_any_sync(0xffffffffu, b);  // lanes of this warp in chunk b
    const int rank = __popc(same & ((1u << lane) - 1u));
    if (b >= 0 && rank == 0) wcount[warp * g.NCH + b] = __popc(same);
    __syncthreads();
    if (threadIdx.x == 0) {  // exclusive prefix over (chunk, warp)
        int run = 0;
        for (int c = 0; c < g.NCH; ++c) {
            bstart[c] = run;
            for (int w = 0; w < nw; ++w) {
                const int v = wcount[w * g.NCH + c];
                wcount[w * g.NCH + c] = run;
                run += v;
            }
        }
        bstart[g.NCH] = run;
    }
    __syncthreads();
    if (b >= 0) {
        const int pos = wcount[warp * g.NCH + b] + rank;
        const int ky = pk / g.kw, kx = pk % g.kw;
        entries[(size_t)i * kk + pos] =
            chunk_entry_bytes(g, code - b * g.KC, chunk_phase_off(g, ky, kx));
    }
    for (int c = threadIdx.x; c <= g.NCH; c += blockDim.x)
        starts[(size_t)i * (g.NCH + 1) + c] = bstart[c];
}

// ---------------------------------------------------------------- kernel --
struct ChunkArgs {
    const float *x;  // usually the output of the kernel before: coherent loads
    const float *__restrict__ D;
    const uint32_t *entries;  // written by chunk_prep_kernel just before
    const int *starts;
    const float *__restrict__ bias;
    float *__restrict__ y;
    int N, Cs, H, W, Ct, Csp, K, M, Ho, Wo, kk, ct_cta, relu;
    ChunkGeom g;
};

template <int P, int CTW, int QPT, int CSPT, bool BF>
__global__ void __launch_bounds__(kChunkThreads, 1) conv_chunked_kernel(const ChunkArgs a) {
    constexpr int E = BF ? 2 : 1;  // positions per lane and slot
    extern __shared__ __align__(16) float csm[];
    const ChunkGeom &g = a.g;
    float *lut = csm;  // fp32 [KC][SK]; bf16 [2][KC][SKW] words
    float *ds = csm + (BF ? (size_t)2 * g.KC * g.SKW : (size_t)g.KC * g.SK);  // [K][CSPT]
    grid_dep_sync();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int oy0 = blockIdx.x * g.TH;
    const int ct0 = blockIdx.y * a.ct_cta;
    const int n = blockIdx.z;
    const int ctw0 = ct0 + warp * CTW;

    float acc[CTW][P * E];
#pragma unroll
    for (int c = 0; c < CTW; ++c)
#pragma unroll
        for (int p = 0; p < P * E; ++p) acc[c][p] = 0.f;

    float xr[QPT][CSPT];  // input sub-vectors of positions tid + qi * 512

    // rows [kl] of chunk ch: lut[kl][q] = <x(q), D[m][k0 + kl]>; every thread
    // writes its QPT positions (SK >= QPT * 512, positions past NQ hold 0)
    auto build = [&](int ch, float *L) {
        const int k0 = ch * g.KC, kc = min(g.KC, a.K - k0);
        if constexpr (BF) {
            // entry q of row kl -> copy 0 at q, copy 1 at q - 1 (2-byte slots)
            unsigned short *h0 = reinterpret_cast<unsigned short *>(L);
            unsigned short *h1 = h0 + (size_t)2 * g.KC * g.SKW;
            for (int kl = 0; kl < kc; ++kl) {
                float dk[CSPT];
#pragma unroll
                for (int j = 0; j < CSPT; ++j) dk[j] = ds[(k0 + kl) * CSPT + j];
                const int rb = 2 * kl * g.SKW + tid;
#pragma unroll
                for (int qi = 0; qi + 1 < QPT; qi += 2) {
                    float2 v = make_float2(0.f, 0.f);
#pragma unroll
                    for (int j = 0; j < CSPT; ++j)
                        v = __ffma2_rn(make_float2(xr[qi][j], xr[qi + 1][j]),
                                       make_float2(dk[j], dk[j]), v);
                    const unsigned w = pack_bf16x2(v.x, v.y);
                    const int q0 = rb + qi * kChunkThreads, q1 = q0 + kChunkThreads;
                    h0[q0] = (unsigned short)(w & 0xffffu);
                    h0[q1] = (unsigned short)(w >> 16);
                    if (qi > 0 || tid > 0) h1[q0 - 1] = (unsigned short)(w & 0xffffu);
                    h1[q1 - 1] = (unsigned short)(w >> 16);
                }
                if constexpr (QPT % 2 == 1) {
                    float v = 0.f;
#pragma unroll
                    for (int j = 0; j < CSPT; ++j) v = fmaf(xr[QPT - 1][j], dk[j], v);
                    const unsigned short hv = (unsigned short)(pack_bf16x2(v, 0.f) & 0xffffu);
                    const int q = rb + (QPT - 1) * kChunkThreads;
                    h0[q] = hv;
                    if (QPT > 1 || tid > 0) h1[q - 1] = hv;
                }
            }
        } else {
            for (int kl = 0; kl < kc; ++kl) {
                float dk[CSPT];
#pragma unroll
                for (int j = 0; j < CSPT; ++j) dk[j] = ds[(k0 + kl) * CSPT + j];
                float *row = L + kl * g.SK + tid;
#pragma unroll
                for (int qi = 0; qi + 1 < QPT; qi += 2) {
                    float2 v = make_float2(0.f, 0.f);
#pragma unroll
                    for (int j = 0; j < CSPT; ++j)
                        v = __ffma2_rn(make_float2(xr[qi][j], xr[qi + 1][j]),
                                       make_float2(dk[j], dk[j]), v);
                    row[qi * kChunkThreads] = v.x;
                    row[(qi + 1) * kChunkThreads] = v.y;
                }
                if constexpr (QPT % 2 == 1) {
                    float v = 0.f;
#pragma unroll
                    for (int j = 0; j < CSPT; ++j) v = fmaf(xr[QPT - 1][j], dk[j], v);
                    row[(QPT - 1) * kChunkThreads] = v;
                }
            }
        }
    };

    // the (c_t, p_k) pairs of this warp's channels whose code is in chunk ch
    auto gather = [&](int m, int ch, const float *L) {
        const unsigned char *lb = reinterpret_cast<const unsigned char *>(L) + lane * 4;
#pragma unroll
        for (int c = 0; c < CTW; ++c) {
            const int ct = ctw0 + c;
            if (ct < a.Ct) {
                const size_t row = (size_t)m * a.Ct + ct;
                const int e0 = a.starts[row * (g.NCH + 1) + ch];
                const int e1 = a.starts[row * (g.NCH + 1) + ch + 1];
                const uint32_t *ep = a.entries + row * a.kk;
                auto look = [&](const unsigned char *b) {
                    QCNN_CHECK(b + (P - 1) * 128 + 4 <=
                                   reinterpret_cast<const unsigned char *>(L) + 4 * g.KC * g.SK,
                               QCNN_CHECK_TABLE);
                    if constexpr (BF) {
#pragma unroll
                        for (int p = 0; p < P; ++p)
                            add_bf16x2(acc[c][2 * p], acc[c][2 * p + 1],
                                       *reinterpret_cast<const unsigned *>(b + p * 128));
                    } else {
                        accumulate<P>(acc[c], [&](int p) {
                            return *reinterpret_cast<const float *>(b + p * 128);
                        });
                    }
                };
                int e = e0;
                for (; e + 1 < e1; e += 2) {
                    const unsigned o0 = ep[e], o1 = ep[e + 1];
                    look(lb + o0);
                    look(lb + o1);
                }
                if (e < e1) look(lb + ep[e]);
            }
        }
    };

    for (int m = 0; m < a.M; ++m) {
        __syncthreads();  // previous sub-space finished with ds and the tables
        for (int e = tid; e < a.K * CSPT; e += kChunkThreads) {
            const int k = e / CSPT, j = e % CSPT;
            ds[e] = j < a.Csp ? __ldg(a.D + ((size_t)m * a.K + k) * a.Csp + j) : 0.f;
        }
#pragma unroll
        for (int qi = 0; qi < QPT; ++qi) {
            const int q = tid + qi * kChunkThreads;
            const int phase = q / g.PS, rem = q - phase * g.PS;
            const int r = rem / g.PW, c = rem - r * g.PW;
            const int ay = phase / g.s, ax = phase - ay * g.s;
            const int iy = (oy0 + r + g.dymin) * g.s + ay, ix = (c + g.dxmin) * g.s + ax;
            const bool ok = q < g.NQ && iy >= 0 && iy < a.H && ix >= 0 && ix < a.W;
            const float *xp = a.x + (((size_t)n * a.Cs + (size_t)m * a.Csp) * a.H +
                                     (ok ? iy : 0)) * a.W + (ok ? ix : 0);
#pragma unroll
            for (int j = 0; j < CSPT; ++j) {
                const float v = xp[(size_t)min(j, a.Csp - 1) * a.H * a.W];
                xr[qi][j] = (ok && j < a.Csp) ? v : 0.f;
            }
        }
        __syncthreads();  // ds ready

        for (int ch = 0; ch < g.NCH; ++ch) {
            build(ch, lut);
            __syncthreads();
            gather(m, ch, lut);
            __syncthreads();  // table rows free for the next chunk
        }
    }

    // ---- epilogue
#pragma unroll
    for (int c = 0; c < CTW; ++c) {
        const int ct = ctw0 + c;
        if (ct >= a.Ct) continue;
        const float bv = a.bias ? a.bias[ct] : 0.f;
#pragma unroll
        for (int p = 0; p < P * E; ++p) {
            const int l = BF ? (p >> 1) * 64 + 2 * lane + (p & 1) : p * 32 + lane;
            const int r = l / g.PW, col = l - r * g.PW;
            const int oy = oy0 + r;
            if (r < g.TH && col < a.Wo && oy < a.Ho) {
                float v = acc[c][p] + bv;
                if (a.relu) v = fmaxf(v, 0.f);
                a.y[(((size_t)n * a.Ct + ct) * a.Ho + oy) * a.Wo + col] = v;
            }
        }
    }
}

struct ChunkVariant {
    int P, CTW, QPT, CSPT, BF;
    void (*fn)(ChunkArgs);
};
#define QCNN_CHUNK(P, CTW, QPT, C) {P, CTW, QPT, C, 0, conv_chunked_kernel<P, CTW, QPT, C, false>}
#define QCNN_CHUNK_BF(P, CTW, QPT, C) {P, CTW, QPT, C, 1, conv_chunked_kernel<P, CTW, QPT, C, true>}
static const ChunkVariant kChunk[] = {
    QCNN_CHUNK(8, 6, 11, 3),  // AlexNet conv1: 4 rows of 57, 96 channels per CTA
    QCNN_CHUNK(8, 1, 11, 3),  // same band, 16 channels per CTA: small batches
    QCNN_CHUNK(8, 8, 6, 4),
    QCNN_CHUNK(4, 8, 4, 8),
    // bfloat16 tables: slots of 64 positions
    QCNN_CHUNK_BF(4, 6, 11, 3),
    QCNN_CHUNK_BF(4, 1, 11, 3),
    QCNN_CHUNK_BF(4, 8, 6, 4),
    QCNN_CHUNK_BF(2, 8, 4, 8),
};
#undef QCNN_CHUNK_BF
#undef QCNN_CHUNK
constexpr int kNumChunk = sizeof(kChunk) / sizeof(kChunk[0]);

static ChunkGeom chunk_geom(const ConvShape &s, int TH, int KC, int P, int QPT, int bf) {
    ChunkGeom g;
    g.bf = bf;
    g.s = s.stride;
    g.pad = s.pad;
    g.kh = s.kh;
    g.kw = s.kw;
    g.TH = TH;
    g.dymin = floor_div(-s.pad, s.stride);
    g.dymax = floor_div(s.kh - 1 - s.pad, s.stride);
    g.dxmin = floor_div(-s.pad, s.stride);
    g.dxmax = floor_div(s.kw - 1 - s.pad, s.stride);
    g.PR = TH + g.dymax - g.dymin;
    g.PW = s.Wo + g.dxmax - g.dxmin;
    g.PS = g.PR * g.PW;
    g.NQ = s.stride * s.stride * g.PS;
    // entries of a row: the largest entry offset plus the lanes' reach
    int sk = (s.stride * s.stride - 1) * g.PS + (g.dymax - g.dymin) * g.PW + (g.dxmax - g.dxmin) +
             P * 32 * (bf ? 2 : 1) + (bf ? 1 : 0);
    sk = std::max(sk, QPT * kChunkThreads);  // every thread's positions fit a row
    if (bf) {
        g.SKW = (sk + 1) / 2;
        g.SK = 2 * g.SKW;
    } else {
        while (sk % 32 != 1) ++sk;
        g.SK = sk;
        g.SKW = 0;
    }
    g.KC = KC;
    g.NCH = cdiv(s.K, KC);
    return g;
}

ConvChunkPlan plan_conv_chunked(const ConvShape &s) {
    ConvChunkPlan best;
    const int sms = num_sms();
    int dev = 0, smem_optin = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
            cudaSuccess || smem_optin <= 0) {
        cudaGetLastError();
        smem_optin = 227 * 1024;
    }
#ifdef QCNN_TUNING  // tuning builds only: force a variant from the environment
    const char *force_env = getenv("QCNN_CHUNK_VARIANT");
    const int force = force_env ? atoi(force_env) : -1;
#endif
    for (int v = 0; v < kNumChunk; ++v) {
#ifdef QCNN_TUNING
        if (force >= 0 && v != force) continue;
#endif
        const ChunkVariant &cv = kChunk[v];
        if (cv.BF != s.bf16 || s.Csp > cv.CSPT || s.kh * s.kw > kMaxPrepKK) continue;
        const int ct_cta = 16 * cv.CTW;
        const int E = cv.BF ? 2 : 1;
        // largest band that the variant's lanes and registers cover
        for (int TH = std::min(s.Ho, 64); TH >= 1; --TH) {
            const ChunkGeom g0 = chunk_geom(s, TH, 1, cv.P, cv.QPT, cv.BF);
            if (TH * g0.PW > cv.P * 32 * E) continue;
            if (g0.NQ > cv.QPT * kChunkThreads) continue;
            const int row_tiles = cdiv(s.Ho, TH);
            const int th = cdiv(s.Ho, row_tiles);  // balance the bands
            for (int KC : {16, 8, 4, 2, 1}) {
                if (KC > s.K) continue;
                const ChunkGeom g = chunk_geom(s, th, KC, cv.P, cv.QPT, cv.BF);
                // fp32: KC rows of SK floats; bf16: two copies of KC x SKW words
                const size_t smem = ((size_t)KC * g.SK + (size_t)s.K * cv.CSPT) * sizeof(float);
                if (smem > (size_t)smem_optin) continue;
                const int ct_tiles = cdiv(s.Ct, ct_cta);
                const double ctas = (double)s.N * row_tiles * ct_tiles;
                const double waves = std::ceil(ctas / sms);
                // per CTA and sub-space: gather wavefronts + table stores + a
                // barrier cost per chunk
                const double gather = (double)cv.P * ct_cta * s.kh * s.kw;
                const double build = (double)g.NQ * s.K / 32.0 * (cv.BF ? 2.0 : 1.0);
                const double sync = (double)g.NCH * 1200.0;
                const double score = waves * (gather + build + sync) * s.M;
                if (!best.ok || score < best.score) {
                    best.ok = true;
                    best.variant = v;
                    best.g_TH = th;
                    best.KC = KC;
                    best.ct_cta = ct_cta;
                    best.row_tiles = row_tiles;
                    best.ct_tiles = ct_tiles;
                    best.smem = smem;
                    best.score = score;
                }
                break;  // largest KC that fits
            }
            break;  // largest TH that fits
        }
    }
    if (best.ok) {
        const ChunkVariant &cv = kChunk[best.variant];
        const ChunkGeom g = chunk_geom(s, best.g_TH, best.KC, cv.P, cv.QPT, cv.BF);
        best.NCH = g.NCH;
        best.entries_bytes = align_up((size_t)s.M * s.Ct * s.kh * s.kw * 4, kWsAlign);
        best.starts_bytes = align_up((size_t)s.M * s.Ct * (g.NCH + 1) * 4, kWsAlign);
    }
    return best;
}

qcnn_status launch_conv_chunked(const ConvShape &s, const ConvChunkPlan &p, const float *x,
                                const float *D, const uint8_t *codes, int codes_packed,
                                const float *bias, float *y, int relu, void *ws,
                                cudaStream_t st) {
    const ChunkVariant &cv = kChunk[p.variant];
    const ChunkGeom g = chunk_geom(s, p.g_TH, p.KC, cv.P, cv.QPT, cv.BF);
    uint32_t *entries = static_cast<uint32_t *>(ws);
    int *starts = reinterpret_cast<int *>(static_cast<uint8_t *>(ws) + p.entries_bytes);
    const int kk = s.kh * s.kw;
    const int pthreads = cdiv(kk, 32) * 32;
    const size_t psmem = ((size_t)(pthreads / 32) * g.NCH + g.NCH + 1) * sizeof(int);
    qcnn_status rc = launch_pdl(chunk_prep_kernel, dim3(s.M * s.Ct), dim3(pthreads), psmem, st,
                                codes, codes_packed, packed_ct(s.Ct), s.Ct, kk, s.M, s.K, g,
                                entries, starts);
    if (rc != QCNN_OK) return rc;
    ChunkArgs a;
    a.x = x;
    a.D = D;
    a.entries = entries;
    a.starts = starts;
    a.bias = bias;
    a.y = y;
    a.N = s.N;
    a.Cs = s.Cs;
    a.H = s.H;
    a.W = s.W;
    a.Ct = s.Ct;
    a.Csp = s.Csp;
    a.K = s.K;
    a.M = s.M;
    a.Ho = s.Ho;
    a.Wo = s.Wo;
    a.kk = kk;
    a.ct_cta = p.ct_cta;
    a.relu = relu;
    a.g = g;
    cudaError_t e =
        cudaFuncSetAttribute(cv.fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem);
    if (e != cudaSuccess) return cuda_status(e);
    dim3 grid(p.row_tiles, p.ct_tiles, s.N);
    return launch_pdl(cv.fn, grid, dim3(kChunkThreads), p.smem, st, a);
}

}  // namespace qcnn
