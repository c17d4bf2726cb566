// conv.cu -- PQ convolutional layer response (Sec. 3.2, Eq. 7):
//   y[n][ct][oy][ox] = bias[ct] + sum_{ky,kx} sum_m LUT_n[m][p_s][k_m(ct, p_k)]
//   LUT_n[m][p_s][k] = <x_n^(m)(p_s), D^(m)_k>,  p_s = (oy*s - pad + ky, ox*s - pad + kx)
//
// Two kernels compute it:
//  * conv_fused (stride 1): outputs live on a padded grid of row pitch
//    max(W + pad, Wo), output (oy, ox) at linear position l = oy*pitch + ox;
//    the halo grid has the same pitch, input (iy, ix) at (iy + pad)*pitch +
//    ix + pad, so output l reads halo position l + ky*pitch + kx at kernel
//    offset (ky, kx).  A read past the end of a row runs on, in linear
//    order, into the next row's `pad` leading zero columns: the right
//    padding of one row and the left padding of the next share one gap.
//    One CTA owns an image, a run of ST consecutive output positions (a
//    tile; it need not start or end on a row) and CT_CTA output channels.
//    For each sub-space m it builds, in shared memory, the table of the
//    ST + reach halo positions its outputs read -- layout lut[k][h], h
//    relative to the tile's first position -- and then gathers from it.
//    Lanes of a warp take consecutive positions, so for one (c_t, p_k) the
//    whole warp shares one code k and reads 32 consecutive words of row k:
//    bank-conflict free, and the kernel offset is a plain shift of the read
//    address.  Lanes on padding columns (or past the last output) compute
//    values that are discarded.
//    bfloat16 tables (BF): every 32-bit word holds the entries of two
//    neighbouring positions, (h, h+1), so one load serves two look-ups.  A
//    kernel offset can be odd, so the table is kept twice: copy 0 holds the
//    pairs that start at even h (word h/2), copy 1 those that start at odd h
//    (word (h-1)/2).  A lane takes two neighbouring positions and reads copy
//    (offset & 1); the two copies of 2-byte entries fill the space of one
//    fp32 table.
//  * conv_unfused (any stride): tables are first written to the workspace
//    in a stride-phase-split layout lut[nb][m][k][ay][ax][py][px] with
//    (iy, ix) = (py*s + ay, px*s + ax), so that consecutive output columns
//    read consecutive words for every kernel offset; a gather kernel then
//    reads them through L1/L2.  Images are processed in chunks sized to
//    stay L2 resident.
#include "conv_fused.cuh"

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <vector>

namespace qcnn {

// ===================================================================== pack
int packed_ct(int Ct) { return cdiv(Ct, 256) * 256; }
size_t packed_codes_bytes(int Ct, int kk, int M) {
    return (size_t)M * kk * (size_t)packed_ct(Ct);
}

// packed[m][pk][ct] = min(codes[ct][pk][m], K - 1); zero for ct >= Ct.
__global__ void pack_codes_kernel(const uint8_t *__restrict__ codes, int Ct, int kk,
                                  int M, int K, int CtP, uint8_t *__restrict__ packed) {
    grid_dep_sync();
    const size_t total = (size_t)M * kk * CtP;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (size_t)gridDim.x * blockDim.x) {
        const int ct = (int)(i % CtP);
        const size_t r = i / CtP;
        const int pk = (int)(r % kk);
        const int m = (int)(r / kk);
        unsigned v = 0;
        if (ct < Ct) {
            v = codes[((size_t)ct * kk + pk) * M + m];
            QCNN_CHECK(v < (unsigned)K, QCNN_CHECK_CODE);
            v = v < (unsigned)K ? v : (unsigned)(K - 1);
        }
        packed[i] = (uint8_t)v;
    }
}

qcnn_status launch_pack_codes(const uint8_t *codes, int Ct, int kk, int M, int K,
                              uint8_t *packed, cudaStream_t st) {
    const size_t total = packed_codes_bytes(Ct, kk, M);
    const int blocks = (int)std::min<size_t>((total + 255) / 256, (size_t)num_sms() * 8);
    return launch_pdl(pack_codes_kernel, dim3(blocks), dim3(256), 0, st, codes, Ct, kk, M, K,
                      packed_ct(Ct), packed);
}

// Stream-K fix-up: the tile cut at the end of CTA b's range gets
// y = (sub-spaces before the cut) + (after) + bias, then ReLU.  Grid
// (boundaries, piece / 1024): each thread adds four consecutive piece
// entries (one channel, four positions) with 16-byte loads; boundaries that
// fall between tiles have nothing to do.  Entries on discarded positions were
// never written and are read but not stored.
// Stream-K fix-up.  CTA c owns units [u0(c), u1(c)), u = tile * M + m; a
// tile whose units fall to several CTAs left pieces [CT_CTA][ST] in
// part[c][1] (the CTA that began the tile and ended inside it: its head) and
// part[c][0] (every later CTA: a middle or its tail).  Block row b handles
// the tile cut at the boundary after CTA b when that CTA began the tile, and
// adds its pieces in CTA order (a fixed order), then bias and ReLU.
__device__ __forceinline__ long long sk_u0(int c, int base, int extra) {
    return (long long)c * base + min(c, extra);
}
// the CTA whose range holds unit u
__device__ __forceinline__ int sk_cta_of(long long u, int base, int extra) {
    const long long big = (long long)extra * (base + 1);  // units of the first extra CTAs
    return u < big ? (int)(u / (base + 1)) : extra + (int)((u - big) / base);
}
__global__ void conv_sk_fixup_kernel(const float *part, int base, int extra, int M,
                                     int pos_tiles, int ct_tiles, int ST, int ct_cta, int Ct,
                                     int pitch, int Ho, int Wo, const float *__restrict__ bias,
                                     int relu, float *__restrict__ y) {
    grid_dep_sync();
    const int b = blockIdx.x;
    const long long ub = sk_u0(b + 1, base, extra);  // first unit after CTA b
    if (ub % M == 0) return;                          // no tile cut here
    const long long t = ub / M;
    if (t * M < sk_u0(b, base, extra)) return;  // CTA b did not begin tile t
    const int c_last = sk_cta_of(t * M + M - 1, base, extra);
    const size_t piece = (size_t)ct_cta * ST;  // a multiple of 4: ST % 32 == 0
    const size_t o4 = ((size_t)blockIdx.y * blockDim.x + threadIdx.x) * 4;
    if (o4 >= piece) return;
    const int n = (int)(t / ((long long)ct_tiles * pos_tiles));
    const int rest = (int)(t - (long long)n * ct_tiles * pos_tiles);
    const int ct0 = (rest / pos_tiles) * ct_cta, l0 = (rest % pos_tiles) * ST;
    float4 a = *reinterpret_cast<const float4 *>(part + ((size_t)b * 2 + 1) * piece + o4);
    for (int c = b + 1; c <= c_last; ++c) {
        const float4 v = *reinterpret_cast<const float4 *>(part + (size_t)c * 2 * piece + o4);
        a.x += v.x;
        a.y += v.y;
        a.z += v.z;
        a.w += v.w;
    }
    const float v4[4] = {a.x, a.y, a.z, a.w};
    const int cl = (int)(o4 / ST), ct = ct0 + cl;
    if (ct >= Ct) return;
    const float bv = bias ? bias[ct] : 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int g = l0 + (int)(o4 - (size_t)cl * ST) + i;
        const int oy = g / pitch, col = g - oy * pitch;
        if (oy >= Ho || col >= Wo) continue;
        float v = v4[i] + bv;
        if (relu) v = fmaxf(v, 0.f);
        y[(((size_t)n * Ct + ct) * Ho + oy) * Wo + col] = v;
    }
}

// y = bias + sum over splits of the partial sums, in split order; then ReLU.
__global__ void conv_split_reduce_kernel(const float *partial, int splits,
                                         size_t total, int Ct, int HoWo,
                                         const float *__restrict__ bias, int relu,
                                         float *__restrict__ y) {
    grid_dep_sync();
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (size_t)gridDim.x * blockDim.x) {
        float v = 0.f;
        // (unrolled: the loads of up to 16 splits in flight at once, added in order)
#pragma unroll 16
        for (int s = 0; s < splits; ++s) v += partial[(size_t)s * total + i];
        if (bias) v += bias[(i / HoWo) % Ct];
        if (relu) v = fmaxf(v, 0.f);
        y[i] = v;
    }
}

// ---------------------------------------------------------- variant table --
// Assembled once from the instantiating units, in a fixed order.
static const std::vector<FusedVariant> &fused_table() {
    static const std::vector<FusedVariant> table = [] {
        std::vector<FusedVariant> t;
        for (auto part : {fused_variants_plain, fused_variants_bf16, fused_variants_sk,
                          fused_variants_tc, fused_variants_tc_sk, fused_variants_narrow}) {
            int n = 0;
            const FusedVariant *v = part(&n);
            t.insert(t.end(), v, v + n);
        }
        return t;
    }();
    return table;
}


static int ks_for(int need) {  // smallest KS >= need with KS % 32 == 1
    int ks = need;
    while (ks % 32 != 1) ++ks;
    return ks;
}

int conv_fused_variant_count() { return (int)fused_table().size(); }

void conv_fused_variant_info(int v, int info[10]) {
    const FusedVariant &f = fused_table()[v];
    const int vals[10] = {f.P, f.CTW, f.WP, f.CSP4, f.NW, f.MINB, f.PIPE, f.BF, f.SK, f.TC};
    for (int i = 0; i < 10; ++i) info[i] = vals[i];
}

ConvFusedPlan plan_conv_fused(const ConvShape &s, int force, int force_cl) {
    ConvFusedPlan best;
    if (s.stride != 1 || s.Csp > kMaxCsp) return best;
    const int csp4 = s.Csp <= 4 ? 4 : 8;
    // Row pitch of the halo grid: >= W + pad, so that every read past a
    // row's data lands on zeros (this row's tail or the next row's `pad`
    // leading columns), and >= Wo, so that a row of outputs fits in a row.
    const int pitch = std::max(s.W + s.pad, s.Wo);
    const int kk = s.kh * s.kw;
    const int sms = num_sms();
    int dev = 0;
    cudaGetDevice(&dev);
    int smem_optin = 0;
    if (cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
            cudaSuccess ||
        smem_optin <= 0) {
        cudaGetLastError();
        smem_optin = 227 * 1024;
    }
    int smem_sm = 0;
    if (cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) !=
            cudaSuccess ||
        smem_sm <= 0) {
        cudaGetLastError();
        smem_sm = 228 * 1024;
    }
#ifdef QCNN_TUNING  // tuning builds only: force a variant from the environment
    const char *force_env = getenv("QCNN_FUSED_VARIANT");
    if (force < 0 && force_env) force = atoi(force_env);
#endif
    for (int v = 0; v < (int)fused_table().size(); ++v) {
        if (force >= 0 && v != force) continue;
        const FusedVariant &fv = fused_table()[v];
        // (the tensor-core build keeps sub-vectors 8 wide in any case)
        if ((fv.CSP4 != csp4 && !fv.TC) || fv.BF != s.bf16) continue;
        const int slots = fv.WP * fv.P;
        const int E = fv.BF ? 2 : 1;  // positions per lane and slot
        const int ST = slots * 32 * E;  // output positions per tile
        const int npos = (s.Ho - 1) * pitch + s.Wo;  // through the last output
        const int pos_tiles = cdiv(npos, ST);
        const int reach = (s.kh - 1) * pitch + (s.kw - 1);  // largest kernel offset
        // halo positions read by the lanes of a tile; a map shorter than one
        // tile needs only those of its own positions (lanes past them read
        // rows that are never written, and their values are discarded)
        const int HP = std::min(ST, npos) + reach;
        // fp32: KS floats per row, >= every position read; bf16: two copies
        // of RW words per row, RW > every pair word read or written
        int KS;
        if (fv.BF) {
            const int RW = ks_for(slots * 32 + (reach >> 1) + 1);
            if ((HP - 1) / 2 >= RW) continue;
            KS = 2 * RW;
        } else {
            KS = ks_for(ST + reach);
        }
        const int ct_cta = (fv.NW / fv.WP) * fv.CTW;
        // tensor-core build: whole 128-row MMA tiles of halo positions, K
        // (a multiple of 32, at most 256) accumulator columns per tile, all
        // tiles within the 512 columns of tensor memory of the one CTA per SM
        const int n_mt = cdiv(HP, 128);
        // (measured: with C'_s <= 4 the split pass, MMA latency and fences cost
        // more than the 4 FMAs per entry they replace -- AlexNet conv2-5 7-12%
        // slower -- so the tensor cores build only wider sub-vectors)
        if (fv.TC && (s.Csp <= 4 || s.K % 32 != 0 || s.K > 256 || n_mt * s.K > 512)) continue;
        const int vw = fv.CSP4;  // sub-vector width of the variant's staging
        const int xs_floats = fv.TC ? n_mt * 128 * vw : cdiv(HP, 4) * 4 * vw;
        const size_t smem = fused_smem_layout(s.K, KS, xs_floats, vw, kk, ct_cta,
                                              fv.PIPE ? 2 : 1, fv.TC ? n_mt * 128 : 0)
                                .total;
        if (smem > (size_t)smem_optin) continue;
        // One tensor-core CTA per SM: each allocates all 512 columns of
        // tensor memory, and an allocation waits until the columns are free.
        // Two CTAs of one cluster on one SM would wait for each other (the
        // first frees its columns only after the cluster's barrier), so
        // the shared memory asked for keeps a second CTA off the SM.
        size_t smem_launch = smem;
        if (fv.TC) smem_launch = std::max(smem, ((size_t)smem_sm / 2 + 1024 + 15) / 16 * 16);
        if (smem_launch > (size_t)smem_optin) continue;
        const int cps = std::max(1, std::min(fv.MINB, (int)(smem_sm / (smem_launch + 1024))));
        if (fv.TC && cps != 1) continue;
        const int ct_tiles = cdiv(s.Ct, ct_cta);
        const double ctas = (double)s.N * pos_tiles * ct_tiles;
        // work per CTA and sub-space in shared-memory wavefronts (~cycles):
        // gather (incl. lanes on discarded positions and channels past Ct)
        // over the variant's measured efficiency, plus the exposed part of the
        // table build (about 4 wavefronts of time per 32 entries:
        // latency-bound FMA chains)
        const double gather_m = (double)slots * ct_cta * kk / fv.eff;
        const double build_m = (double)HP * s.K * 4.0 / 32.0;
        const double per_m = gather_m + build_m * fv.build;
        // a CTA with mps sub-spaces: the first table build is never hidden,
        // the later ones at the variant's exposure (two-buffer tiles: a short
        // run of sub-spaces hides little -- measured at batch 1, AlexNet conv3
        // and conv5: 27.3 us with the 128-position two-buffer tile against
        // 25.2 us with the 192-position one-buffer tile)
        auto cta_work = [&](int mps) {
            return gather_m * mps + build_m * (1.0 + fv.build * (mps - 1));
        };
        // Small batches: split the sub-spaces of each tile over `splits` CTAs
        // (partial sums through the workspace, then a reduction) when the
        // grid would leave SMs idle.
        // The 12-warp tiles lose to 16-warp ones when a CTA gets only a few
        // sub-spaces (measured: AlexNet conv3 at batch 1, 64 splits, 47 us
        // against 33 us), so they are split at most 8 ways.
        // The splits of a tile can form a thread-block cluster (cl CTAs, a
        // power of two dividing the split count, at most 16) whose partial
        // tiles are added in distributed shared memory: then only
        // splits / cl partial sums per output go through the workspace, and
        // none (no reduction launch) when cl == splits.  The cluster's tile
        // of sums reuses the table's shared memory.
        const int max_sp = fv.NW == 12 ? 8 : 64;
        const bool red_fits = (size_t)ct_cta * ST * sizeof(float) <= smem;
        int splits = 1, cl = 1;
        double score = 0;
        for (int sp = 1; sp <= std::min(s.M, max_sp); sp *= 2) {
            const int mps = cdiv(s.M, sp);
            const int sp_eff = cdiv(s.M, mps);
            for (int c = 1; c <= std::min(sp_eff, 16); c *= 2) {
                if (sp_eff % c != 0 || (c > 1 && (!red_fits || force_cl == 1))) continue;
                if (force_cl > 1 && c != force_cl && sp_eff > 1) continue;
                double slots = (double)sms * cps;
                if (c > 1) {
                    const int cap = cluster_capacity(reinterpret_cast<const void *>(fv.fn),
                                                     fv.NW * 32, c, smem_launch);
                    if (cap < 1) continue;
                    slots = std::min(slots, (double)cap * c);
                }
                const int groups = sp_eff / c;
                const double waves = std::ceil(ctas * sp_eff / slots);
                const double part =
                    groups > 1 ? 2.0 * groups * s.N * s.Ct * s.Ho * s.Wo * 4.0 : 0.0;
                const double red = c > 1 ? ((double)ct_cta * ST / 8.0 + 1500.0) * cps : 0.0;
                const double sc = waves * cta_work(mps) * cps + part / 3000.0 +
                                  (groups > 1 ? 3000.0 : 0.0) + red;
                if ((sp == 1 && c == 1) || sc < score) {
                    score = sc;
                    splits = sp_eff;
                    cl = c;
                }
            }
            if (ctas * sp >= 2.0 * sms * cps) break;
        }
        // Large batches: a stream-K schedule gives every one of the G CTA
        // slots the same number of (tile, sub-space) units, instead of whole
        // tiles in ceil(ctas / G) waves; a tile cut between two CTAs costs a
        // partial-sum round trip and a fix-up launch.
        const int G = sms * cps;
        int sk = 0;
        double sk_units = 0;
        bool allow_sk = true;
#ifdef QCNN_TUNING
        allow_sk = getenv("QCNN_NO_SK") == nullptr;
#endif
        // Measured on the AlexNet and VGG shapes: a stream-K unit costs 5-10%
        // more than a plain one (tile hand-overs, cut tiles), and 20% more
        // with the build-heavy bf16 tables; it pays only when the last wave
        // of the plain grid is well short of full.
        const double wave_fill = ctas / (std::ceil(ctas / G) * G);
        if (fv.SK) {
            // At least half as many tiles as CTA slots: every CTA then takes
            // >= M / 2 units, so a tile spreads over at most three CTAs.
            // (Fewer tiles -- small batches -- are split by sub-space ranges
            // instead.)  The planner's own choice also wants a short last
            // wave on the plain grid.
            if (2 * ctas < G || ctas * s.M < G) continue;  // (and every CTA >= 1 unit)
            if (force < 0 && (!allow_sk || wave_fill >= 0.9)) continue;
            sk_units = std::ceil(ctas * s.M / G);
            const double part = 2.0 * 2.0 * (G - 1) * ct_cta * ST * 4.0;
            score = sk_units * per_m * cps * 1.05 + part / 3000.0 + 6000.0;
            sk = 1;
            splits = 1;
            cl = 1;
        }
        if (!best.ok || score < best.score) {
            best.splits = splits;
            best.cl = cl;
            best.m_per_split = cdiv(s.M, splits);
            best.partial_bytes = splits / cl > 1 ? (size_t)(splits / cl) * s.N * s.Ct * s.Ho *
                                                       s.Wo * sizeof(float)
                                                 : 0;
            best.sk = sk;
            if (sk) {
                const long long units = (long long)s.N * pos_tiles * ct_tiles * s.M;
                best.sk_ctas = G;
                best.sk_base = (int)(units / G);
                best.sk_extra = (int)(units % G);
                best.partial_bytes = (size_t)G * 2 * ct_cta * ST * sizeof(float);
            }
            best.ok = true;
            best.variant = v;
            best.P = fv.P;
            best.CTW = fv.CTW;
            best.WP = fv.WP;
            best.ST = ST;
            best.pitch = pitch;
            best.KS = KS;
            best.HP = HP;
            best.ct_cta = ct_cta;
            best.pos_tiles = pos_tiles;
            best.ct_tiles = ct_tiles;
            best.smem = smem_launch;
            best.xs_floats = xs_floats;
            best.score = score;
        }
    }
#ifdef QCNN_TUNING
    if (best.ok && getenv("QCNN_PLAN_VERBOSE"))
        fprintf(stderr,
                "fused plan: v=%d P=%d CTW=%d WP=%d NW=%d pipe=%d ST=%d tiles=%d KS=%d ct_cta=%d smem=%zu "
                "splits=%d sk=%d sk_ctas=%d base=%d extra=%d\n",
                best.variant, best.P, best.CTW, best.WP, fused_table()[best.variant].NW,
                fused_table()[best.variant].PIPE, best.ST, best.pos_tiles, best.KS, best.ct_cta, best.smem, best.splits,
                best.sk, best.sk_ctas, best.sk_base, best.sk_extra);
#endif
    return best;
}

qcnn_status launch_conv_fused(const ConvShape &s, const ConvFusedPlan &p, const float *x,
                              const float *D, const uint8_t *packed, const float *bias,
                              float *y, int relu, float *partial_ws, cudaStream_t st,
                              bool early, bool leave_partials) {
    const FusedVariant &fv = fused_table()[p.variant];
    ConvFusedArgs a;
    a.x = x;
    a.D = D;
    a.codes = packed;
    a.bias = bias;
    a.y = y;
    a.N = s.N;
    a.Cs = s.Cs;
    a.H = s.H;
    a.W = s.W;
    a.Ct = s.Ct;
    a.kh = s.kh;
    a.kw = s.kw;
    a.pad = s.pad;
    a.Csp = s.Csp;
    a.K = s.K;
    a.M = s.M;
    a.Ho = s.Ho;
    a.Wo = s.Wo;
    a.pitch = p.pitch;
    a.ST = p.ST;
    a.KS = p.KS;
    a.HP = p.HP;
    a.CtP = packed_ct(s.Ct);
    a.relu = relu;
    a.xs_floats = p.xs_floats;
    a.splits = p.splits;
    a.m_per_split = p.m_per_split;
    a.cl = p.cl;
    a.partial = partial_ws;
    a.sk = p.sk;
    a.sk_base = p.sk_base;
    a.sk_extra = p.sk_extra;
    a.pos_tiles = p.pos_tiles;
    a.ct_tiles = p.ct_tiles;
    a.early = early ? 1 : 0;
    cudaError_t e = cudaFuncSetAttribute(fv.fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)p.smem);
    if (e == cudaSuccess && p.cl > 8)
        e = cudaFuncSetAttribute(fv.fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return cuda_status(e);
    const dim3 grid = p.sk ? dim3(p.sk_ctas, 1, 1) : dim3(p.pos_tiles, p.ct_tiles, s.N * p.splits);
    const dim3 cluster = p.cl > 1 ? dim3(1, 1, p.cl) : dim3(0, 0, 0);
    qcnn_status rc = launch_k(fv.fn, grid, dim3(fv.NW * 32), p.smem, st, cluster, a);
    if (rc != QCNN_OK) return rc;
    if (p.sk) {
        if (p.sk_ctas < 2) return QCNN_OK;
        const dim3 fgrid(p.sk_ctas - 1, (unsigned)cdiv(p.ct_cta * p.ST / 4, 256));
        return launch_pdl(conv_sk_fixup_kernel, fgrid, dim3(256), 0, st,
                          static_cast<const float *>(partial_ws), p.sk_base, p.sk_extra, s.M,
                          p.pos_tiles, p.ct_tiles, p.ST, p.ct_cta, s.Ct, p.pitch, s.Ho, s.Wo,
                          bias, relu, y);
    }
    if (p.splits / p.cl == 1 || leave_partials) return rc;
    return launch_split_reduce(partial_ws, p.splits / p.cl, (size_t)s.N * s.Ct * s.Ho * s.Wo,
                               s.Ct, s.Ho * s.Wo, bias, relu, y, st);
}

qcnn_status launch_split_reduce(const float *partial, int splits, size_t total, int Ct, int HoWo,
                                const float *bias, int relu, float *y, cudaStream_t st) {
    const int blocks = (int)std::min<size_t>((total + 255) / 256, (size_t)num_sms() * 8);
    return launch_pdl(conv_split_reduce_kernel, dim3(blocks), dim3(256), 0, st, partial, splits,
                      total, Ct, HoWo, bias, relu, y);
}

// ================================================================== unfused
// Tables of a chunk of NB images in the stride-phase-split layout
//   lut[nb][m][k][ay][ax][py][px],  iy = py*s + ay,  ix = px*s + ax.
struct UnfusedLutArgs {
    const float *x;  // usually the output of the kernel before: coherent loads
    const float *__restrict__ D;
    float *__restrict__ lut;
    int n0, NB, Cs, H, W, s, Csp, K, M, HQ, WQ;
};

__global__ void __launch_bounds__(256) conv_unfused_lut_kernel(const UnfusedLutArgs a) {
    extern __shared__ __align__(16) float dsm[];  // D[m] : [K][Csp]
    grid_dep_sync();
    const int m = blockIdx.y, nb = blockIdx.z;
    const int n = a.n0 + nb;
    for (int e = threadIdx.x; e < a.K * a.Csp + kMaxCsp; e += blockDim.x)
        dsm[e] = e < a.K * a.Csp ? a.D[(size_t)m * a.K * a.Csp + e] : 0.f;
    __syncthreads();
    const int PQ = a.s * a.s * a.HQ * a.WQ;
    const int q = blockIdx.x * blockDim.x + threadIdx.x;
    if (q >= PQ) return;
    const int px = q % a.WQ;
    int r = q / a.WQ;
    const int py = r % a.HQ;
    r /= a.HQ;
    const int ax = r % a.s, ay = r / a.s;
    const int iy = py * a.s + ay, ix = px * a.s + ax;
    float xv[kMaxCsp];
    const bool in = iy < a.H && ix < a.W;
    const float *xp = a.x + (((size_t)n * a.Cs + (size_t)m * a.Csp) * a.H + (in ? iy : 0)) * a.W +
                      (in ? ix : 0);
#pragma unroll
    for (int j = 0; j < kMaxCsp; ++j) {
        // the address stays inside x even for the lanes j >= Csp that are discarded
        const float v = xp[(size_t)min(j, a.Csp - 1) * a.H * a.W];
        xv[j] = (in && j < a.Csp) ? v : 0.f;
    }
    float *out = a.lut + ((size_t)nb * a.M + m) * a.K * (size_t)PQ + q;
    for (int k = 0; k < a.K; ++k) {
        const float *dk = dsm + k * a.Csp;  // dsm is padded by kMaxCsp floats
        float v = 0.f;
#pragma unroll
        for (int j = 0; j < kMaxCsp; ++j)
            if (j < a.Csp) v = fmaf(xv[j], dk[j], v);
        out[(size_t)k * PQ] = v;
    }
}

struct UnfusedGatherArgs {
    const float *lut;                   // written by the kernel before
    const uint8_t *codes;               // packed [M][kk][CtP] (maybe by the kernel before)
    const float *__restrict__ bias;
    float *__restrict__ y;
    int n0, Ct, CtP, H, W, kh, kw, s, pad, K, M, Ho, Wo, HQ, WQ, relu;
    int col_tiles;
};

constexpr int kUnfCTW = 16;  // channels per warp
constexpr int kUnfSL = 2;    // 32-column slots per warp

// grid: x = row tile (8 rows, one per warp) * col tile, y = channel tile, z = image in chunk
__global__ void __launch_bounds__(256) conv_unfused_gather_kernel(const UnfusedGatherArgs a) {
    grid_dep_sync();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int rt = blockIdx.x / a.col_tiles, ctile = blockIdx.x % a.col_tiles;
    const int oy = rt * 8 + warp;
    const int ct0 = blockIdx.y * kUnfCTW;
    const int nb = blockIdx.z;
    if (oy >= a.Ho) return;
    const int PQ = a.s * a.s * a.HQ * a.WQ;
    float acc[kUnfCTW][kUnfSL];
#pragma unroll
    for (int c = 0; c < kUnfCTW; ++c)
#pragma unroll
        for (int sl = 0; sl < kUnfSL; ++sl) acc[c][sl] = 0.f;
    int ox[kUnfSL];
#pragma unroll
    for (int sl = 0; sl < kUnfSL; ++sl) ox[sl] = (ctile * kUnfSL + sl) * 32 + lane;
    const int kk = a.kh * a.kw;
    for (int m = 0; m < a.M; ++m) {
        const float *lm = a.lut + ((size_t)nb * a.M + m) * a.K * (size_t)PQ;
        for (int ky = 0; ky < a.kh; ++ky) {
            const int iy = oy * a.s - a.pad + ky;
            if (iy < 0 || iy >= a.H) continue;
            const int ay = iy % a.s, py = iy / a.s;
            for (int kx = 0; kx < a.kw; ++kx) {
                const int t = kx - a.pad;
                const int ax = ((t % a.s) + a.s) % a.s;
                const int dx = (t - ax) / a.s;  // exact
                bool ok[kUnfSL];
                int off[kUnfSL];
#pragma unroll
                for (int sl = 0; sl < kUnfSL; ++sl) {
                    const int ix = ox[sl] * a.s + t;
                    ok[sl] = ox[sl] < a.Wo && ix >= 0 && ix < a.W;
                    off[sl] = ((ay * a.s + ax) * a.HQ + py) * a.WQ + ox[sl] + dx;
                }
                const uint8_t *cp = a.codes + ((size_t)m * kk + ky * a.kw + kx) * a.CtP + ct0;
                const uint4 cw = *reinterpret_cast<const uint4 *>(cp);
                const unsigned kmax4 = (unsigned)(a.K - 1) * 0x01010101u;
                QCNN_CHECK((__vcmpgtu4(cw.x, kmax4) | __vcmpgtu4(cw.y, kmax4) |
                            __vcmpgtu4(cw.z, kmax4) | __vcmpgtu4(cw.w, kmax4)) == 0u,
                           QCNN_CHECK_CODE);
                const unsigned w[4] = {__vminu4(cw.x, kmax4), __vminu4(cw.y, kmax4),
                                       __vminu4(cw.z, kmax4), __vminu4(cw.w, kmax4)};
#pragma unroll
                for (int c = 0; c < kUnfCTW; ++c) {
                    const unsigned code = byte_of(w[c >> 2], c & 3);
                    const float *row = lm + (size_t)code * PQ;
#pragma unroll
                    for (int sl = 0; sl < kUnfSL; ++sl) {
                        QCNN_CHECK(!ok[sl] || (size_t)code * PQ + off[sl] < (size_t)a.K * PQ,
                                   QCNN_CHECK_TABLE);
                        if (ok[sl]) acc[c][sl] += row[off[sl]];
                    }
                }
            }
        }
    }
    const int n = a.n0 + nb;
#pragma unroll
    for (int c = 0; c < kUnfCTW; ++c) {
        const int ct = ct0 + c;
        if (ct >= a.Ct) continue;
        const float bv = a.bias ? a.bias[ct] : 0.f;
#pragma unroll
        for (int sl = 0; sl < kUnfSL; ++sl) {
            if (ox[sl] >= a.Wo) continue;
            float v = acc[c][sl] + bv;
            if (a.relu) v = fmaxf(v, 0.f);
            a.y[(((size_t)n * a.Ct + ct) * a.Ho + oy) * a.Wo + ox[sl]] = v;
        }
    }
}

constexpr size_t kUnfusedLutBudget = (size_t)64 << 20;  // keep a chunk L2 resident

ConvUnfusedPlan plan_conv_unfused(const ConvShape &s) {
    ConvUnfusedPlan p;
    p.HQ = cdiv(s.H, s.stride);
    p.WQ = cdiv(s.W, s.stride);
    const size_t per_image =
        (size_t)s.M * s.K * s.stride * s.stride * p.HQ * p.WQ * sizeof(float);
    p.NB = (int)std::max<size_t>(1, std::min<size_t>(s.N, kUnfusedLutBudget / per_image));
    p.lut_bytes = per_image * p.NB;
    return p;
}

qcnn_status launch_conv_unfused(const ConvShape &s, const ConvUnfusedPlan &p, const float *x,
                                const float *D, const uint8_t *packed, const float *bias,
                                float *y, int relu, float *lut_ws, cudaStream_t st) {
    const int PQ = s.stride * s.stride * p.HQ * p.WQ;
    const int col_tiles = cdiv(s.Wo, 32 * kUnfSL);
    for (int n0 = 0; n0 < s.N; n0 += p.NB) {
        const int nb = std::min(p.NB, s.N - n0);
        UnfusedLutArgs la{x, D, lut_ws, n0, nb, s.Cs, s.H, s.W, s.stride, s.Csp, s.K, s.M,
                          p.HQ, p.WQ};
        dim3 g1(cdiv(PQ, 256), s.M, nb);
        qcnn_status rc = launch_pdl(conv_unfused_lut_kernel, g1, dim3(256),
                                    ((size_t)s.K * s.Csp + kMaxCsp) * sizeof(float), st, la);
        if (rc != QCNN_OK) return rc;
        UnfusedGatherArgs ga{lut_ws, packed, bias, y, n0, s.Ct, packed_ct(s.Ct), s.H, s.W,
                             s.kh, s.kw, s.stride, s.pad, s.K, s.M, s.Ho, s.Wo, p.HQ, p.WQ,
                             relu, col_tiles};
        dim3 g2(cdiv(s.Ho, 8) * col_tiles, cdiv(s.Ct, kUnfCTW), nb);
        rc = launch_pdl(conv_unfused_gather_kernel, g2, dim3(256), 0, st, ga);
        if (rc != QCNN_OK) return rc;
    }
    return QCNN_OK;
}

}  // namespace qcnn
