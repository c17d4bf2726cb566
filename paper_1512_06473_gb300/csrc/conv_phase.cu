// conv_phase.cu -- PQ conv response (Sec. 3.2, Eq. 7) of strided layers, one
// stride phase at a time.
//
// With stride s and padding p, kernel row ky reads input row oy*s - p + ky.
// Writing ky - p = dy*s + ay (0 <= ay < s) that row is (oy + dy)*s + ay: for
// a fixed phase (ay, ax) the layer is a stride-1 correlation of the phase
// plane X_{ay,ax}[py][px] = x[py*s + ay][px*s + ax] with the kernel offsets
// (dy, dx) of that phase.  Every phase plane is laid out on one padded grid
// of pitch Wo + dxmax - dxmin (dx ranging over [dxmin, dxmax]): output
// (oy, ox) is position oy*pitch + ox, and it reads grid position
// (oy + dy - dymin)*pitch + (ox + dx - dxmin), a plain shift per offset.
//
// One CTA owns an image, a tile of ST consecutive output positions and
// CT_CTA output channels.  For each (sub-space m, phase) unit it builds, in
// shared memory, the table of the ST + reach grid positions the tile reads --
// all K sub-codewords, layout lut[k][h] with lanes on consecutive positions,
// as in the stride-1 fused kernel -- and gathers the offsets of that phase:
// for one (c_t, p_k) the whole warp shares one code and reads 32
// consecutive words of one table row (conflict free).  AlexNet conv1 (11x11,
// stride 4): 16 phases of 3x3, 3x2, 2x3 or 2x2 offsets.
// Units are split over several CTAs for small batches (partial sums through
// the workspace, added in a fixed order by launch_split_reduce).
#include "qcnn_internal.cuh"

#include <algorithm>
#include <cmath>

namespace qcnn {

struct PhaseArgs {
    const float *__restrict__ x;
    const float *__restrict__ D;
    const uint8_t *__restrict__ codes;  // packed [M][kk][CtP]
    const float *__restrict__ bias;
    float *__restrict__ y;
    float *__restrict__ partial;  // [splits / cl][N][Ct][Ho][Wo] when splits > cl
    int N, Cs, H, W, Ct, kh, kw, s, pad, Csp, K, M, Ho, Wo;
    int pitch, dymin, dxmin, HP, KS, CtP, relu, xs_floats;
    int splits, units_per_split;
    int cl;  // the splits of a tile form clusters of cl CTAs (1: none)
    // 1: D and the packed codes are constants of the caller (no kernel of the
    // same call writes them): the first sub-space's are staged before the
    // wait on the previous kernel
    int early;
};

struct PhaseSmem {
    size_t lut, xs, ds, cs, total;
};
__host__ __device__ inline PhaseSmem phase_smem_layout(int K, int KS, int xs_floats, int csp4,
                                                       int kk, int ct_cta) {
    PhaseSmem L;
    L.lut = 0;
    L.xs = ((size_t)K * KS * 4 + 15) / 16 * 16;
    L.ds = L.xs + (size_t)2 * xs_floats * 4;
    L.cs = L.ds + (size_t)2 * K * csp4 * 4;
    L.total = L.cs + ((size_t)2 * kk * ct_cta + 15) / 16 * 16;
    return L;
}

// P: 32-position slots per warp; CTW: channels per warp (even);
// CSP4: C'_s register width (4 or 8); CSPE: C'_s itself when the variant is
// made for one value (the build then skips the zero slots), else CSP4;
// NW: warps per CTA.
template <int P, int CTW, int CSP4, int CSPE, int NW>
__global__ void __launch_bounds__(NW * 32, 1) conv_phase_kernel(const PhaseArgs a) {
    static_assert(CSPE >= 1 && CSPE <= CSP4, "C'_s width");
    constexpr int NT = NW * 32;
    constexpr int ST = P * 32;
    constexpr int CT_CTA = NW * CTW;
    constexpr int Q16 = CT_CTA / 16;
    constexpr int QB = 16 / CSP4;  // sub-codewords per lane per build pass
    static_assert(CT_CTA % 16 == 0 && CTW % 2 == 0, "channel tile");
    extern __shared__ __align__(16) unsigned char smem[];
    const int kk = a.kh * a.kw, K = a.K, KS = a.KS, HP = a.HP, pitch = a.pitch, s = a.s;
    const int S2 = s * s;
    const PhaseSmem L = phase_smem_layout(K, KS, a.xs_floats, CSP4, kk, CT_CTA);
    float *lut = reinterpret_cast<float *>(smem + L.lut);
    float *xs = reinterpret_cast<float *>(smem + L.xs);
    float *ds = reinterpret_cast<float *>(smem + L.ds);
    uint8_t *cs = smem + L.cs;
    if (!a.early) grid_dep_sync();

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int l0 = blockIdx.x * ST, ct0 = blockIdx.y * CT_CTA;
    const int n = blockIdx.z / a.splits, split = blockIdx.z % a.splits;
    const int HW = a.H * a.W;
    const int U = a.M * S2;
    const int ub = split * a.units_per_split, ue = min(U, ub + a.units_per_split);

    if (a.Csp < CSP4) {  // sub-vector slots j >= C'_s stay zero
        for (int e = tid; e < 2 * a.xs_floats; e += NT) xs[e] = 0.f;
        for (int e = tid; e < 2 * K * CSP4; e += NT) ds[e] = 0.f;
    }
    __syncthreads();

    // ---- staging (callers commit) ----------------------------------------
    // grid position l0 + h = r*pitch + c is phase-plane point
    // (r + dymin, c + dxmin), i.e. input (iy, ix) = ((r + dymin)*s + ay,
    // (c + dxmin)*s + ax); zero outside the map
    auto stage_x = [&](int u, int b) {
        const int m = u / S2, ph = u - m * S2, ay = ph / s, ax = ph - ay * s;
        float *xb = xs + b * a.xs_floats;
        const float *xn = a.x + ((size_t)n * a.Cs + (size_t)m * a.Csp) * HW;
        for (int h = tid; h < HP; h += NT) {
            const int g = l0 + h, r = g / pitch, c = g - r * pitch;
            const int iy = (r + a.dymin) * s + ay, ix = (c + a.dxmin) * s + ax;
            const bool ok = iy >= 0 && iy < a.H && ix >= 0 && ix < a.W;
            const float *src = ok ? xn + iy * a.W + ix : a.x;
            for (int j = 0; j < a.Csp; ++j)
                cp_async4(xb + h * CSP4 + j, ok ? src + (size_t)j * HW : a.x, ok);
        }
    };
    auto stage_m = [&](int m) {  // sub-codebook and codes of sub-space m, buffer m & 1
        float *db = ds + (m & 1) * K * CSP4;
        const float *dm = a.D + (size_t)m * K * a.Csp;
        for (int k = tid; k < K; k += NT)
            for (int j = 0; j < a.Csp; ++j) cp_async4(db + k * CSP4 + j, dm + k * a.Csp + j, true);
        uint8_t *cb = cs + (size_t)(m & 1) * kk * CT_CTA;
        const uint8_t *cm = a.codes + (size_t)m * kk * a.CtP + ct0;
        for (int e = tid; e < kk * Q16; e += NT) {  // zeros past the packed row
            const int pk = e / Q16, q = e % Q16;
            if (ct0 + q * 16 < a.CtP)
                cp_async16(cb + pk * CT_CTA + q * 16, cm + (size_t)pk * a.CtP + q * 16);
            else
                *reinterpret_cast<uint4 *>(cb + pk * CT_CTA + q * 16) = make_uint4(0, 0, 0, 0);
        }
    };

    // ---- build: lut[k][h] = <x(h), D[m][k]>; lanes on k, warps on h -------
    const int hpw = cdiv(HP, NW);
    const int h0 = warp * hpw, h1 = min(HP, h0 + hpw);
    auto build = [&](int b, int m) {
        const float *xb = xs + b * a.xs_floats;
        const float *db = ds + (m & 1) * K * CSP4;
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
                    for (int j = 0; j < CSPE; ++j) v = fmaf(xv[j], dk[i][j], v);
                    if (k < K) lut[k * KS + h] = v;
                }
            }
        }
    };

    // ---- gather: the offsets (ky, kx) of phase (ay, ax) --------------------
    float acc[CTW][P];
#pragma unroll
    for (int c = 0; c < CTW; ++c)
#pragma unroll
        for (int p = 0; p < P; ++p) acc[c][p] = 0.f;
    const unsigned char *lutb = reinterpret_cast<const unsigned char *>(lut) + lane * 4;
    const int KS4 = KS * 4;
    const unsigned kmax4 = (unsigned)(K - 1) * 0x01010101u;  // clamp codes into [0, K)
    auto gather = [&](int u) {
        const int m = u / S2, ph = u - m * S2, ay = ph / s, ax = ph - ay * s;
        const uint8_t *cb = cs + (size_t)(m & 1) * kk * CT_CTA + warp * CTW;
        // first kernel row / column of the phase: (ky - pad) % s == ay; the
        // offset (dy, dx) then steps by one with each further row / column
        const int ky0 = (ay + a.pad) % s, kx0 = (ax + a.pad) % s;
        const int dy0 = (ky0 - a.pad - ay) / s, dx0 = (kx0 - a.pad - ax) / s;  // exact
        for (int ky = ky0, dy = dy0; ky < a.kh; ky += s, ++dy) {
            for (int kx = kx0, dx = dx0; kx < a.kw; kx += s, ++dx) {
                const int pk = ky * a.kw + kx;
                // the warp's CTW codes: 32-bit words, or 16-bit pairs when
                // CTW is not a multiple of 4; clamped into [0, K)
                unsigned w[(CTW + 3) / 4];
                if constexpr (CTW % 4 == 0) {
#pragma unroll
                    for (int i = 0; i < CTW / 4; ++i)
                        w[i] = *reinterpret_cast<const unsigned *>(cb + pk * CT_CTA + 4 * i);
                } else {
                    const unsigned short *h =
                        reinterpret_cast<const unsigned short *>(cb + pk * CT_CTA);
#pragma unroll
                    for (int i = 0; i < (CTW + 3) / 4; ++i)
                        w[i] = (unsigned)h[2 * i] | (2 * i + 1 < CTW / 2 ? (unsigned)h[2 * i + 1] << 16 : 0u);
                }
#pragma unroll
                for (int i = 0; i < (CTW + 3) / 4; ++i) {
                    QCNN_CHECK(__vcmpgtu4(w[i], kmax4) == 0u, QCNN_CHECK_CODE);
                    w[i] = __vminu4(w[i], kmax4);
                }
                const int off4 = ((dy - a.dymin) * pitch + (dx - a.dxmin)) * 4;
#pragma unroll
                for (int c = 0; c < CTW; ++c) {
                    QCNN_CHECK((int)byte_of(w[c >> 2], c & 3) * KS4 + off4 + lane * 4 +
                                       (P - 1) * 128 + 4 <= K * KS4,
                               QCNN_CHECK_TABLE);
                    const unsigned char *row = lutb + (int)byte_of(w[c >> 2], c & 3) * KS4 + off4;
                    accumulate<P>(acc[c], [&](int p) {
                        return *reinterpret_cast<const float *>(row + p * 128);
                    });
                }
            }
        }
    };

    // ---- units [ub, ue): one table buffer, two barriers per unit ----------
    stage_m(ub / S2);
    if (a.early) grid_dep_sync();
    stage_x(ub, 0);
    cp_async_commit();
    for (int u = ub, b = 0; u < ue; ++u, b ^= 1) {
        cp_async_wait<0>();
        __syncthreads();  // unit u staged; gather of unit u - 1 finished
        if (u + 1 < ue) {
            stage_x(u + 1, b ^ 1);
            if ((u + 1) / S2 != u / S2) stage_m((u + 1) / S2);
            cp_async_commit();
        }
        build(b, u / S2);
        __syncthreads();
        gather(u);
    }
    cp_async_wait<0>();

    if (a.cl > 1) {
        // the splits of this tile (one cluster) add their partial tiles in
        // distributed shared memory; with more splits than one cluster, each
        // cluster's sum is a partial for the split reduction
        __syncthreads();  // every warp is done with the table
        float *red = reinterpret_cast<float *>(smem);  // [CT_CTA][ST]
#pragma unroll
        for (int c = 0; c < CTW; ++c)
#pragma unroll
            for (int p = 0; p < P; ++p) red[(warp * CTW + c) * ST + p * 32 + lane] = acc[c][p];
        const size_t plane = (size_t)a.N * a.Ct * a.Ho * a.Wo;
        const int group = split / a.cl, groups = a.splits / a.cl;
        cluster_tile_reduce(red, CT_CTA * ST, [&](int e, float v) {
            const int ch = e / ST, l = e - ch * ST;
            const int ct = ct0 + ch;
            const int g = l0 + l, oy = g / pitch, ox = g - oy * pitch;
            if (ct >= a.Ct || ox >= a.Wo || oy >= a.Ho) return;
            const size_t o = (((size_t)n * a.Ct + ct) * a.Ho + oy) * a.Wo + ox;
            QCNN_CHECK(o < plane, QCNN_CHECK_GLOBAL);
            if (groups > 1) {
                a.partial[(size_t)group * plane + o] = v;
            } else {
                v += a.bias ? a.bias[ct] : 0.f;
                if (a.relu) v = fmaxf(v, 0.f);
                a.y[o] = v;
            }
        });
        return;
    }

    // ---- epilogue: bias, ReLU, store; or raw partial sums -------------------
#pragma unroll
    for (int c = 0; c < CTW; ++c) {
        const int ct = ct0 + warp * CTW + c;
        if (ct >= a.Ct) continue;
        const float bv = a.bias ? a.bias[ct] : 0.f;
#pragma unroll
        for (int p = 0; p < P; ++p) {
            const int g = l0 + p * 32 + lane, oy = g / pitch, ox = g - oy * pitch;
            if (ox >= a.Wo || oy >= a.Ho) continue;
            const size_t o = (((size_t)n * a.Ct + ct) * a.Ho + oy) * a.Wo + ox;
            QCNN_CHECK(o < (size_t)a.N * a.Ct * a.Ho * a.Wo, QCNN_CHECK_GLOBAL);
            if (a.splits > 1) {
                a.partial[(size_t)split * a.N * a.Ct * a.Ho * a.Wo + o] = acc[c][p];
            } else {
                float v = acc[c][p] + bv;
                if (a.relu) v = fmaxf(v, 0.f);
                a.y[o] = v;
            }
        }
    }
}

// ---------------------------------------------------------- variant table --
struct PhaseVariant {
    int P, CTW, CSP4, CSPE, NW;
    void (*fn)(PhaseArgs);
};
#define QCNN_PHASE(P, CTW, C4, CE, NW) {P, CTW, C4, CE, NW, conv_phase_kernel<P, CTW, C4, CE, NW>}
static const PhaseVariant kPhase[] = {
    QCNN_PHASE(7, 6, 4, 3, 16),   // C'_s = 3, 96 channels (AlexNet conv1), 224 positions
    QCNN_PHASE(7, 6, 4, 4, 16),
    QCNN_PHASE(7, 8, 4, 4, 12),
    QCNN_PHASE(6, 8, 4, 4, 12),
    QCNN_PHASE(4, 8, 4, 4, 12),
    QCNN_PHASE(6, 8, 4, 4, 16),   // 128 channels
    QCNN_PHASE(4, 16, 4, 4, 16),  // 256 channels
    QCNN_PHASE(6, 8, 8, 8, 12),
    QCNN_PHASE(6, 8, 8, 8, 16),
    QCNN_PHASE(4, 16, 8, 8, 16),
};
#undef QCNN_PHASE
constexpr int kNumPhase = sizeof(kPhase) / sizeof(kPhase[0]);

static int phase_ks(int need) {  // smallest KS >= need with KS % 32 == 1
    int ks = need;
    while (ks % 32 != 1) ++ks;
    return ks;
}

static int floor_div_i(int a, int b) { return a >= 0 ? a / b : -((-a + b - 1) / b); }

ConvPhasePlan plan_conv_phase(const ConvShape &s, int force_cl) {
    ConvPhasePlan best;
    if (s.Csp > kMaxCsp || s.bf16) return best;
    const int csp4 = s.Csp <= 4 ? 4 : 8;
    const int kk = s.kh * s.kw;
    const int dymin = floor_div_i(-s.pad, s.stride), dymax = floor_div_i(s.kh - 1 - s.pad, s.stride);
    const int dxmin = floor_div_i(-s.pad, s.stride), dxmax = floor_div_i(s.kw - 1 - s.pad, s.stride);
    const int pitch = s.Wo + dxmax - dxmin;
    const int reach = (dymax - dymin) * pitch + (dxmax - dxmin);
    const int npos = (s.Ho - 1) * pitch + s.Wo;
    const int sms = num_sms();
    int dev = 0, smem_optin = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
            cudaSuccess ||
        smem_optin <= 0) {
        cudaGetLastError();
        smem_optin = 227 * 1024;
    }
    const int U = s.M * s.stride * s.stride;
    for (int v = 0; v < kNumPhase; ++v) {
        const PhaseVariant &pv = kPhase[v];
        if (pv.CSP4 != csp4 || s.Csp > pv.CSPE) continue;
        const int ST = pv.P * 32;
        const int HP = std::min(ST, npos) + reach;
        const int KS = phase_ks(ST + reach);
        const int ct_cta = pv.NW * pv.CTW;
        const int xs_floats = cdiv(HP, 4) * 4 * csp4;
        const size_t smem = phase_smem_layout(s.K, KS, xs_floats, csp4, kk, ct_cta).total;
        if (smem > (size_t)smem_optin) continue;
        const int pos_tiles = cdiv(npos, ST);
        const int ct_tiles = cdiv(s.Ct, ct_cta);
        const double ctas = (double)s.N * pos_tiles * ct_tiles;
        // per CTA and unit, in shared-memory wavefronts: the gather of the
        // unit's kk / s^2 offsets (average) and the table build, which is
        // not overlapped (about two wavefronts of time per 32 entries)
        const double per_u = (double)pv.P * ct_cta * kk / (s.stride * s.stride) +
                             (double)HP * s.K * 2.0 / 32.0;
        // splits of a tile may form a cluster that adds its partial tiles in
        // distributed shared memory (as in the fused planner)
        const bool red_fits = (size_t)ct_cta * ST * sizeof(float) <= smem;
        int splits = 1, cl = 1;
        double score = 0;
        for (int sp = 1; sp <= std::min(U, 64); sp *= 2) {
            const int ups = cdiv(U, sp), sp_eff = cdiv(U, ups);
            for (int c = 1; c <= std::min(sp_eff, 16); c *= 2) {
                if (sp_eff % c != 0 || (c > 1 && (!red_fits || force_cl == 1))) continue;
                if (force_cl > 1 && c != force_cl && sp_eff > 1) continue;
                double slots = sms;
                if (c > 1) {
                    const int cap = cluster_capacity(reinterpret_cast<const void *>(pv.fn),
                                                     pv.NW * 32, c, smem);
                    if (cap < 1) continue;
                    slots = std::min(slots, (double)cap * c);
                }
                const int groups = sp_eff / c;
                const double waves = std::ceil(ctas * sp_eff / slots);
                const double part =
                    groups > 1 ? 2.0 * groups * s.N * s.Ct * s.Ho * s.Wo * 4.0 : 0.0;
                const double red = c > 1 ? (double)ct_cta * ST / 8.0 + 1500.0 : 0.0;
                const double sc = waves * per_u * ups + part / 3000.0 +
                                  (groups > 1 ? 6000.0 : 0.0) + red;
                if ((sp == 1 && c == 1) || sc < score) {
                    score = sc;
                    splits = sp_eff;
                    cl = c;
                }
            }
            if (ctas * sp >= 2.0 * sms) break;
        }
        // a variant made for this C'_s exactly is preferred at equal cost
        if (pv.CSPE == s.Csp && pv.CSPE < pv.CSP4) score *= 0.97;
        if (!best.ok || score < best.score) {
            best.ok = true;
            best.variant = v;
            best.pitch = pitch;
            best.dymin = dymin;
            best.dxmin = dxmin;
            best.HP = HP;
            best.ST = ST;
            best.KS = KS;
            best.ct_cta = ct_cta;
            best.pos_tiles = pos_tiles;
            best.ct_tiles = ct_tiles;
            best.splits = splits;
            best.cl = cl;
            best.units_per_split = cdiv(U, splits);
            best.partial_bytes = splits / cl > 1 ? (size_t)(splits / cl) * s.N * s.Ct * s.Ho *
                                                       s.Wo * sizeof(float)
                                                 : 0;
            best.smem = smem;
            best.score = score;
        }
    }
    return best;
}

qcnn_status launch_conv_phase(const ConvShape &s, const ConvPhasePlan &p, const float *x,
                              const float *D, const uint8_t *packed, const float *bias, float *y,
                              int relu, float *partial_ws, cudaStream_t st, bool early,
                              bool leave_partials) {
    const PhaseVariant &pv = kPhase[p.variant];
    PhaseArgs a;
    a.x = x;
    a.D = D;
    a.codes = packed;
    a.bias = bias;
    a.y = y;
    a.partial = partial_ws;
    a.N = s.N;
    a.Cs = s.Cs;
    a.H = s.H;
    a.W = s.W;
    a.Ct = s.Ct;
    a.kh = s.kh;
    a.kw = s.kw;
    a.s = s.stride;
    a.pad = s.pad;
    a.Csp = s.Csp;
    a.K = s.K;
    a.M = s.M;
    a.Ho = s.Ho;
    a.Wo = s.Wo;
    a.pitch = p.pitch;
    a.dymin = p.dymin;
    a.dxmin = p.dxmin;
    a.HP = p.HP;
    a.KS = p.KS;
    a.CtP = packed_ct(s.Ct);
    a.relu = relu;
    a.xs_floats = cdiv(p.HP, 4) * 4 * pv.CSP4;
    a.splits = p.splits;
    a.units_per_split = p.units_per_split;
    a.cl = p.cl;
    a.early = early ? 1 : 0;
    cudaError_t e = cudaFuncSetAttribute(pv.fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)p.smem);
    if (e != cudaSuccess) return cuda_status(e);
    if (p.cl > 8) {
        e = cudaFuncSetAttribute(pv.fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return cuda_status(e);
    }
    const dim3 grid(p.pos_tiles, p.ct_tiles, s.N * p.splits);
    const dim3 cluster = p.cl > 1 ? dim3(1, 1, p.cl) : dim3(0, 0, 0);
    qcnn_status rc = launch_k(pv.fn, grid, dim3(pv.NW * 32), p.smem, st, cluster, a);
    if (rc != QCNN_OK || p.splits / p.cl == 1 || leave_partials) return rc;
    return launch_split_reduce(partial_ws, p.splits / p.cl, (size_t)s.N * s.Ct * s.Ho * s.Wo, s.Ct,
                               s.Ho * s.Wo, bias, relu, y, st);
}

}  // namespace qcnn
