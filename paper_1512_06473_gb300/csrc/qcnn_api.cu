// qcnn_api.cu -- the extern "C" entry points of include/qcnn.h: argument
// checks (all done on the host before anything is enqueued), workspace
// carving, algorithm choice and the layer-stack driver.
#include "qcnn_internal.cuh"

#include <algorithm>
#include <atomic>
#include <climits>
#include <mutex>
#include <string>
#include <unordered_map>
#include <vector>

namespace qcnn {

static std::atomic<uint64_t> g_launches{0};
static std::atomic<int> g_last_cuda_error{0};

void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

qcnn_status cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return QCNN_OK;
    g_last_cuda_error.store((int)e);
    return QCNN_ERR_CUDA;
}

qcnn_status after_launch() {
    count_launch();
    return cuda_status(cudaGetLastError());
}

// State of programmatic launches on this host thread: 0 outside a call
// scope (plain launches), 1 in a scope before its first launch (plain), 2 in
// a scope after it (programmatic).
thread_local int t_pdl = 0;

PdlScope::PdlScope() : saved(t_pdl) { t_pdl = 1; }
PdlScope::~PdlScope() { t_pdl = saved; }

void pdl_break() {
    if (t_pdl == 2) t_pdl = 1;
}

bool pdl_next_launch() {
    if (t_pdl == 0) return false;
    const bool programmatic = t_pdl == 2;
    t_pdl = 2;
    return programmatic;
}

// Readers of the translation units' device-check records (debug builds
// register one per unit at load time; release builds none).
std::mutex &check_mutex() {
    static std::mutex m;
    return m;
}
std::vector<CheckReader> &check_readers() {
    static std::vector<CheckReader> v;
    return v;
}

void register_check_reader(CheckReader r) {
    std::lock_guard<std::mutex> g(check_mutex());
    check_readers().push_back(r);
}

qcnn_status collect_device_checks(unsigned *flags) {
    std::lock_guard<std::mutex> g(check_mutex());
    qcnn_status rc = QCNN_OK;
    for (CheckReader r : check_readers()) {
        const qcnn_status s = r(flags);
        if (rc == QCNN_OK) rc = s;
    }
    return rc;
}

qcnn_status sync_and_check(cudaStream_t st) {
    qcnn_status rc = cuda_status(cudaStreamSynchronize(st));
    if (rc != QCNN_OK) return rc;
    unsigned flags = 0;
    if ((rc = collect_device_checks(&flags)) != QCNN_OK) return rc;
    return flags ? QCNN_ERR_DEVICE_CHECK : QCNN_OK;
}

int cluster_capacity(const void *kernel, int threads, int C, size_t smem) {
    static std::mutex mu;
    // keyed by (device, kernel, threads, C, smem); planning asks for hundreds
    static std::unordered_map<std::string, int> cache;
    int dev = 0, ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev < 1 || cudaGetDevice(&dev) != cudaSuccess) {
        // No GPU (planning on a build host, e.g. for plan queries): the
        // cluster occupancy measured on a GB300 (152 SMs) for 1..8 CTAs per
        // SM; clusters do not span GPCs, so fewer SMs hold the large ones.
        cudaGetLastError();
        const int by_threads = std::max(1, 2048 / std::max(threads, 1));
        const int per_sm = std::max(1, std::min(by_threads, (int)(228 * 1024 / (smem + 1024))));
        const int sms_in_clusters = C <= 2 ? 152 : C == 4 ? 146 : C == 8 ? 128 : 112;
        return per_sm * sms_in_clusters / C;
    }
    std::string key(reinterpret_cast<const char *>(&kernel), sizeof kernel);
    const long long rest[4] = {dev, threads, C, (long long)smem};
    key.append(reinterpret_cast<const char *>(rest), sizeof rest);
    {
        std::lock_guard<std::mutex> g(mu);
        const auto it = cache.find(key);
        if (it != cache.end()) return it->second;
    }
    int n = 0;
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) ==
            cudaSuccess &&
        cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) ==
            cudaSuccess) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(C, 1, 1);
        cfg.blockDim = dim3(threads);
        cfg.dynamicSmemBytes = smem;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = C;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess) n = 0;
    }
    cudaGetLastError();
    std::lock_guard<std::mutex> g(mu);
    cache.emplace(std::move(key), n);
    return n;
}

int num_sms() {
    static std::atomic<int> cached[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
        cudaGetLastError();
        return 152;
    }
    int v = cached[dev].load();
    if (v > 0) return v;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) {
        cudaGetLastError();
        v = 152;
    }
    cached[dev].store(v);
    return v;
}

}  // namespace qcnn

using namespace qcnn;

namespace {

inline cudaStream_t as_stream(void *s) { return reinterpret_cast<cudaStream_t>(s); }

bool fits_int(long long v) { return v > 0 && v < (long long)INT_MAX; }

// Device arrays are read with accesses of their element size (4-byte
// cp.async for fp32) and PACKED code arrays with 16-byte copies, so a
// misaligned pointer is refused on the host rather than faulting a kernel.
// NULL passes (NULL-ness is checked where it matters).
bool aligned(const void *p, uintptr_t a) { return reinterpret_cast<uintptr_t>(p) % a == 0; }
bool f32_ok(const void *p) { return aligned(p, 4); }

// The device pointers of every layer of a stack, for qcnn_net_forward*.
bool layer_pointers_ok(const qcnn_layer *layers, int n) {
    for (int i = 0; i < n; ++i) {
        const qcnn_layer &L = layers[i];
        if (L.kind == QCNN_LAYER_MAXPOOL) continue;
        if (!f32_ok(L.D) || !f32_ok(L.bias)) return false;
        if (L.codes_layout == QCNN_CODES_PACKED && !aligned(L.codes, 16)) return false;
    }
    return true;
}

bool pq_ok(int Cs, int Csp, int K) {
    return Cs > 0 && Csp >= 1 && Csp <= kMaxCsp && K >= 1 && K <= kMaxK && Cs % Csp == 0;
}

bool lut_type_ok(int t) { return t == QCNN_LUT_FP32 || t == QCNN_LUT_BF16; }

bool conv_shape(int N, int Cs, int H, int W, int Ct, int kh, int kw, int stride, int pad,
                int Csp, int K, int lut_type, ConvShape *s) {
    if (!lut_type_ok(lut_type)) return false;
    if (N <= 0 || H <= 0 || W <= 0 || Ct <= 0 || kh <= 0 || kw <= 0 || stride <= 0 || pad < 0)
        return false;
    if (!pq_ok(Cs, Csp, K)) return false;
    if (H + 2 * pad < kh || W + 2 * pad < kw) return false;
    const int Ho = (H + 2 * pad - kh) / stride + 1, Wo = (W + 2 * pad - kw) / stride + 1;
    if (Ho <= 0 || Wo <= 0) return false;
    if (!fits_int((long long)N * Cs * H * W) || !fits_int((long long)N * Ct * Ho * Wo) ||
        !fits_int((long long)Ct * kh * kw * (Cs / Csp)))
        return false;
    *s = ConvShape{N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K, Cs / Csp, Ho, Wo,
                   lut_type == QCNN_LUT_BF16};
    return true;
}

bool fc_shape(int N, int Cs, int Ct, int Csp, int K, int lut_type, FcShape *s) {
    if (N <= 0 || Ct <= 0 || !pq_ok(Cs, Csp, K) || !lut_type_ok(lut_type)) return false;
    if (!fits_int((long long)N * Cs) || !fits_int((long long)N * Ct) ||
        !fits_int((long long)(Cs / Csp) * Ct))
        return false;
    *s = FcShape{N, Cs, Ct, Csp, K, Cs / Csp, lut_type == QCNN_LUT_BF16, 0};
    return true;
}

// ------------------------------------------------------------ conv plan ---
struct ConvCall {
    ConvShape s;
    int algo;  // resolved: FUSED, PHASE, CHUNKED or UNFUSED
    ConvFusedPlan fp;
    ConvPhasePlan pp;
    ConvChunkPlan cp;
    ConvUnfusedPlan up;
    size_t packed_off, lut_off, total;
};

qcnn_status plan_conv_call(const ConvShape &s, int codes_layout, int algo, ConvCall *c) {
    if (codes_layout != QCNN_CODES_CANONICAL && codes_layout != QCNN_CODES_PACKED)
        return QCNN_ERR_INVALID_ARG;
    const int force_cl = (algo & QCNN_ALGO_NO_CLUSTER) ? 1 : 0;
    algo &= ~QCNN_ALGO_NO_CLUSTER;
    const bool forced = algo >= QCNN_ALGO_FUSED_VARIANT;
    if (forced) {
        if (algo - QCNN_ALGO_FUSED_VARIANT >= conv_fused_variant_count())
            return QCNN_ERR_INVALID_ARG;
    } else if (algo != QCNN_ALGO_AUTO && algo != QCNN_ALGO_FUSED && algo != QCNN_ALGO_UNFUSED &&
               algo != QCNN_ALGO_CHUNKED && algo != QCNN_ALGO_PHASE) {
        return QCNN_ERR_INVALID_ARG;
    }
    c->s = s;
    c->algo = QCNN_ALGO_UNFUSED;
    if (forced) {
        c->fp = plan_conv_fused(s, algo - QCNN_ALGO_FUSED_VARIANT, force_cl);
        if (!c->fp.ok) return QCNN_ERR_UNSUPPORTED;
        c->algo = QCNN_ALGO_FUSED;
    } else if (algo == QCNN_ALGO_AUTO || algo == QCNN_ALGO_FUSED) {
        c->fp = plan_conv_fused(s, -1, force_cl);
        if (c->fp.ok) c->algo = QCNN_ALGO_FUSED;
        else if (algo == QCNN_ALGO_FUSED) return QCNN_ERR_UNSUPPORTED;
    }
    if (c->algo == QCNN_ALGO_UNFUSED && (algo == QCNN_ALGO_AUTO || algo == QCNN_ALGO_PHASE)) {
        c->pp = plan_conv_phase(s, force_cl);
        if (c->pp.ok) c->algo = QCNN_ALGO_PHASE;
        else if (algo == QCNN_ALGO_PHASE) return QCNN_ERR_UNSUPPORTED;
    }
    if (c->algo == QCNN_ALGO_UNFUSED && (algo == QCNN_ALGO_AUTO || algo == QCNN_ALGO_CHUNKED)) {
        c->cp = plan_conv_chunked(s);
        if (c->cp.ok) c->algo = QCNN_ALGO_CHUNKED;
        else if (algo == QCNN_ALGO_CHUNKED) return QCNN_ERR_UNSUPPORTED;
    }
    // the unfused path has fp32 tables only
    if (c->algo == QCNN_ALGO_UNFUSED && s.bf16) return QCNN_ERR_UNSUPPORTED;
    size_t off = 0;
    c->packed_off = off;
    // the chunked path reads either code layout directly
    if (codes_layout == QCNN_CODES_CANONICAL && c->algo != QCNN_ALGO_CHUNKED)
        off += align_up(packed_codes_bytes(s.Ct, s.kh * s.kw, s.M), kWsAlign);
    c->lut_off = off;
    if (c->algo == QCNN_ALGO_UNFUSED) {
        c->up = plan_conv_unfused(s);
        off += align_up(c->up.lut_bytes, kWsAlign);
    } else if (c->algo == QCNN_ALGO_CHUNKED) {
        off += c->cp.entries_bytes + c->cp.starts_bytes;
    } else if (c->algo == QCNN_ALGO_PHASE) {
        off += align_up(c->pp.partial_bytes, kWsAlign);
    } else {
        off += align_up(c->fp.partial_bytes, kWsAlign);
    }
    c->total = off;
    return QCNN_OK;
}

// Plans of single conv calls, cached like the net plans: planning a layer
// tries every tile variant, split count and cluster size (with cached
// occupancy queries), tens of microseconds of host time, which at batch 1 is
// as long as the layer.  Keyed by device, shape, code layout and algorithm;
// at most kConvPlanCache entries, oldest replaced first.
constexpr size_t kConvPlanCache = 32;
qcnn_status plan_conv_call_cached(const ConvShape &s, int codes_layout, int algo, ConvCall *c) {
    static std::mutex mu;
    static std::vector<std::pair<std::vector<int>, ConvCall>> cache;
    static size_t next = 0;
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        dev = -1;
    }
    const std::vector<int> key = {dev,  s.N,  s.Cs,   s.H,          s.W,  s.Ct,   s.kh,
                                  s.kw, s.stride, s.pad, s.Csp,     s.K,  s.bf16, codes_layout,
                                  algo};
    {
        std::lock_guard<std::mutex> g(mu);
        for (const auto &e : cache)
            if (e.first == key) {
                *c = e.second;
                return QCNN_OK;
            }
    }
    const qcnn_status rc = plan_conv_call(s, codes_layout, algo, c);
    if (rc != QCNN_OK) return rc;
    std::lock_guard<std::mutex> g(mu);
    if (cache.size() < kConvPlanCache) {
        cache.emplace_back(key, *c);
    } else {
        cache[next] = {key, *c};
        next = (next + 1) % kConvPlanCache;
    }
    return QCNN_OK;
}

// Partial sums per output a conv call leaves for a reduction (fused and
// stride-phase plans whose split sub-spaces are not all in one cluster), in
// its workspace at lut_off; 1 when the call writes y itself.
int conv_groups(const ConvCall &c) {
    if (c.algo == QCNN_ALGO_FUSED && !c.fp.sk) return c.fp.splits / c.fp.cl;
    if (c.algo == QCNN_ALGO_PHASE) return c.pp.splits / c.pp.cl;
    return 1;
}

// leave_partials: a call with conv_groups(c) > 1 leaves its partial sums in
// the workspace instead of reducing them into y (the net's conv -> max-pool)
qcnn_status run_conv(const ConvCall &c, const float *x, const float *D, const uint8_t *codes,
                     int codes_layout, const float *bias, float *y, int relu, void *ws,
                     cudaStream_t st, bool leave_partials = false) {
    if (c.algo == QCNN_ALGO_CHUNKED)
        return launch_conv_chunked(c.s, c.cp, x, D, codes, codes_layout == QCNN_CODES_PACKED, bias,
                                   y, relu, static_cast<uint8_t *>(ws) + c.lut_off, st);
    const uint8_t *packed = codes;
    // codes packed by this call are written by a kernel of the call: the
    // conv kernel then reads them only after its wait on that kernel
    const bool early = codes_layout == QCNN_CODES_PACKED;
    if (codes_layout == QCNN_CODES_CANONICAL) {
        uint8_t *p = static_cast<uint8_t *>(ws) + c.packed_off;
        qcnn_status rc =
            launch_pack_codes(codes, c.s.Ct, c.s.kh * c.s.kw, c.s.M, c.s.K, p, st);
        if (rc != QCNN_OK) return rc;
        packed = p;
    }
    float *lut = reinterpret_cast<float *>(static_cast<uint8_t *>(ws) + c.lut_off);
    if (c.algo == QCNN_ALGO_FUSED)
        return launch_conv_fused(c.s, c.fp, x, D, packed, bias, y, relu, lut, st, early,
                                 leave_partials);
    if (c.algo == QCNN_ALGO_PHASE)
        return launch_conv_phase(c.s, c.pp, x, D, packed, bias, y, relu, lut, st, early,
                                 leave_partials);
    return launch_conv_unfused(c.s, c.up, x, D, packed, bias, y, relu, lut, st);
}

bool ws_ok(const void *ws, size_t have, size_t need) {
    if (need == 0) return true;
    return ws != nullptr && have >= need && (reinterpret_cast<uintptr_t>(ws) % kWsAlign) == 0;
}

// -------------------------------------------------------------- net plan ---
// FC layers hand their partial sums to the next FC layer up to this batch
// (above it the next layer's staging would re-read many partials per input)
constexpr int kChainMaxBatch = 8;

struct NetStep {
    int kind;
    int N;              // batch this step is planned for
    ConvCall conv;
    FcShape fc;
    FcPlan fcp;
    int C, H, W;        // input of this layer (per image)
    int oC, oH, oW;     // output
    size_t scratch;     // bytes of layer scratch
    // small batches, FC followed by FC: this layer leaves its partial sums
    // (chain region part_region, 1 or 2) instead of reducing them, and the
    // next layer adds them while staging its input (x_from_prev).  A conv
    // layer followed by a max-pool leaves them in the scratch region, and
    // the pool adds them while staging its planes.
    int leave_partials = 0, part_region = 0, x_from_prev = 0;
};

struct NetPlan {
    int N;
    std::vector<NetStep> steps;
    // host I/O: the input is copied in `chunks` slices of N / chunks images,
    // and the first layer runs on each slice as soon as it has arrived
    // (step0c, planned for the slice), overlapping the remaining copies
    int chunks = 1;
    NetStep step0c;
    size_t act_floats;  // floats of one ping-pong activation buffer
    size_t scratch;     // max layer scratch
    size_t act_off[2], scratch_off, xin_off, yout_off, total;
    size_t chain_bytes = 0, chain_off[2] = {0, 0};  // partial sums handed between FC layers
};

qcnn_status plan_step(const qcnn_layer &L, int N, int c, int h, int w, NetStep *out) {
    NetStep st{};
    st.kind = L.kind;
    st.N = N;
    st.C = c;
    st.H = h;
    st.W = w;
    if (L.kind == QCNN_LAYER_CONV) {
        if (!L.D || !L.codes) return QCNN_ERR_INVALID_ARG;
        ConvShape s;
        if (!conv_shape(N, c, h, w, L.Ct, L.kh, L.kw, L.stride, L.pad, L.Csp, L.K, L.lut_type,
                        &s))
            return QCNN_ERR_INVALID_ARG;
        qcnn_status rc = plan_conv_call(s, L.codes_layout, L.algo, &st.conv);
        if (rc != QCNN_OK) return rc;
        st.scratch = st.conv.total;
        st.oC = L.Ct;
        st.oH = s.Ho;
        st.oW = s.Wo;
    } else if (L.kind == QCNN_LAYER_FC) {
        if (!L.D || !L.codes) return QCNN_ERR_INVALID_ARG;
        const long long cs = (long long)c * h * w;
        if (cs >= INT_MAX) return QCNN_ERR_INVALID_ARG;
        if (!fc_shape(N, (int)cs, L.Ct, L.Csp, L.K, L.lut_type, &st.fc))
            return QCNN_ERR_INVALID_ARG;
        if (L.codes_layout == QCNN_CODES_PACKED) st.fc.code_bits = code_bits(L.K);
        else if (L.codes_layout != QCNN_CODES_CANONICAL) return QCNN_ERR_INVALID_ARG;
        st.fcp = plan_fc(st.fc);
        st.scratch = align_up(st.fcp.partial_bytes, kWsAlign);
        st.oC = L.Ct;
        st.oH = 1;
        st.oW = 1;
    } else if (L.kind == QCNN_LAYER_MAXPOOL) {
        if (L.kh <= 0 || L.stride <= 0 || L.kh > h || L.kh > w) return QCNN_ERR_INVALID_ARG;
        st.oC = c;
        st.oH = (h - L.kh) / L.stride + 1;
        st.oW = (w - L.kh) / L.stride + 1;
    } else {
        return QCNN_ERR_INVALID_ARG;
    }
    *out = st;
    return QCNN_OK;
}

qcnn_status plan_net(const qcnn_layer *layers, int n_layers, int N, int C, int H, int W,
                     int host_io, NetPlan *np) {
    if (!layers || n_layers <= 0 || N <= 0 || C <= 0 || H <= 0 || W <= 0)
        return QCNN_ERR_INVALID_ARG;
    if (!fits_int((long long)N * C * H * W)) return QCNN_ERR_INVALID_ARG;
    np->N = N;
    np->steps.clear();
    np->act_floats = 0;
    np->scratch = 0;
    int c = C, h = H, w = W;
    for (int i = 0; i < n_layers; ++i) {
        NetStep st;
        qcnn_status rc = plan_step(layers[i], N, c, h, w, &st);
        if (rc != QCNN_OK) return rc;
        const long long out = (long long)N * st.oC * st.oH * st.oW;
        if (!fits_int(out)) return QCNN_ERR_INVALID_ARG;
        if (i + 1 < n_layers) np->act_floats = std::max(np->act_floats, (size_t)out);
        np->scratch = std::max(np->scratch, st.scratch);
        c = st.oC;
        h = st.oH;
        w = st.oW;
        np->steps.push_back(st);
    }
    // FC -> FC at small batches: the first layer's partial sums go straight to
    // the second layer's staging (no reduction kernel between them); the
    // regions alternate so that a layer never overwrites the partials it reads
    np->chain_bytes = 0;
    for (int i = 0, r = 0; i + 1 < n_layers; ++i) {
        NetStep &a = np->steps[i], &b = np->steps[i + 1];
        if (a.kind == QCNN_LAYER_FC && b.kind == QCNN_LAYER_FC && N <= kChainMaxBatch &&
            a.fcp.splits / a.fcp.cl > 1) {
            a.leave_partials = 1;
            a.part_region = 1 + (r++ & 1);
            b.x_from_prev = 1;
            np->chain_bytes = std::max(np->chain_bytes, a.fcp.partial_bytes);
        }
    }
    np->chunks = 1;
    if (host_io) {
        const int ch = (N % 4 == 0 && N / 4 >= 8) ? 4 : (N % 2 == 0 && N / 2 >= 8) ? 2 : 1;
        if (ch > 1 && plan_step(layers[0], N / ch, C, H, W, &np->step0c) == QCNN_OK) {
            np->chunks = ch;
            np->scratch = std::max(np->scratch, np->step0c.scratch);
        }
    }
    // conv -> max-pool with split partial sums (small batches): the pool adds
    // them (groups in order, then bias and ReLU: the reduction's arithmetic,
    // so the output is bit-identical) instead of a reduction launch between
    // the two.  Not for a first layer run on input slices (host I/O).
    for (int i = 0; i + 1 < n_layers; ++i) {
        NetStep &a = np->steps[i], &b = np->steps[i + 1];
        if (a.kind == QCNN_LAYER_CONV && b.kind == QCNN_LAYER_MAXPOOL &&
            conv_groups(a.conv) > 1 && (size_t)a.oH * a.oW <= kPoolPlaneMax &&
            !(i == 0 && np->chunks > 1)) {
            a.leave_partials = 1;
            b.x_from_prev = 1;
        }
    }
    size_t off = 0;
    for (int b = 0; b < 2; ++b) {
        np->act_off[b] = off;
        off += align_up(np->act_floats * sizeof(float), kWsAlign);
    }
    np->scratch_off = off;
    off += align_up(np->scratch, kWsAlign);
    for (int r = 0; r < 2; ++r) {
        np->chain_off[r] = off;
        off += align_up(np->chain_bytes, kWsAlign);
    }
    np->xin_off = np->yout_off = off;
    if (host_io) {
        np->xin_off = off;
        off += align_up((size_t)N * C * H * W * sizeof(float), kWsAlign);
        const NetStep &last = np->steps.back();
        np->yout_off = off;
        off += align_up((size_t)N * last.oC * last.oH * last.oW * sizeof(float), kWsAlign);
    }
    np->total = off;
    return QCNN_OK;
}

// Net plans are cached per (device, batch, input shape, layer shapes and
// options): planning a stack costs tens of microseconds on the host, which is
// a tenth of a batch-1 forward.  Layer pointers only enter the key as
// NULL / non-NULL (the plan depends on shapes alone).  At most kPlanCache
// entries, oldest replaced first; the mutex guards the table.
constexpr size_t kPlanCache = 16;
struct PlanKey {
    std::vector<int> v;
    bool operator==(const PlanKey &o) const { return v == o.v; }
};
struct PlanCache {
    std::mutex mu;
    std::vector<std::pair<PlanKey, NetPlan>> entries;
    size_t next = 0;
};
PlanCache &plan_cache() {
    static PlanCache c;
    return c;
}

qcnn_status plan_net_cached(const qcnn_layer *layers, int n_layers, int N, int C, int H, int W,
                            int host_io, NetPlan *np) {
    if (!layers || n_layers <= 0 || n_layers > 4096)
        return plan_net(layers, n_layers, N, C, H, W, host_io, np);
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        dev = -1;
    }
    PlanKey key;
    key.v.reserve(7 + 14 * (size_t)n_layers);
    key.v.insert(key.v.end(), {dev, n_layers, N, C, H, W, host_io});
    for (int i = 0; i < n_layers; ++i) {
        const qcnn_layer &L = layers[i];
        key.v.insert(key.v.end(), {L.kind, L.Ct, L.kh, L.kw, L.stride, L.pad, L.Csp, L.K, L.relu,
                                   L.algo, L.codes_layout, L.lut_type, L.D != nullptr,
                                   L.codes != nullptr});
    }
    PlanCache &pc = plan_cache();
    {
        std::lock_guard<std::mutex> g(pc.mu);
        for (const auto &e : pc.entries)
            if (e.first == key) {
                *np = e.second;
                return QCNN_OK;
            }
    }
    const qcnn_status rc = plan_net(layers, n_layers, N, C, H, W, host_io, np);
    if (rc != QCNN_OK) return rc;
    std::lock_guard<std::mutex> g(pc.mu);
    if (pc.entries.size() < kPlanCache) {
        pc.entries.emplace_back(std::move(key), *np);
    } else {
        pc.entries[pc.next] = {std::move(key), *np};
        pc.next = (pc.next + 1) % kPlanCache;
    }
    return QCNN_OK;
}

qcnn_status run_step(const qcnn_layer &L, const NetStep &s, const float *in, float *out,
                     void *scratch, cudaStream_t st, const PartialInput *xin = nullptr) {
    if (s.kind == QCNN_LAYER_CONV)
        return run_conv(s.conv, in, L.D, L.codes, L.codes_layout, L.bias, out, L.relu, scratch,
                        st, s.leave_partials != 0);
    if (s.kind == QCNN_LAYER_FC)
        return launch_fc(s.fc, s.fcp, in, L.D, L.codes, L.bias, out, L.relu,
                         reinterpret_cast<float *>(scratch), st, xin, s.leave_partials != 0);
    if (xin) return launch_maxpool_partial(*xin, s.N, s.C, s.H, s.W, L.kh, L.stride, out, st);
    return launch_maxpool(in, s.N, s.C, s.H, s.W, L.kh, L.stride, out, st);
}

// Layers [first, n) of the stack; `in` is the input of layer `first`.
qcnn_status run_net(const qcnn_layer *layers, const NetPlan &np, const float *in, float *y,
                    void *ws, cudaStream_t st, int first = 0) {
    uint8_t *base = static_cast<uint8_t *>(ws);
    const int n = (int)np.steps.size();
    for (int i = first; i < n; ++i) {
        const NetStep &s = np.steps[i];
        float *out = (i + 1 == n) ? y : reinterpret_cast<float *>(base + np.act_off[i & 1]);
        uint8_t *scratch =
            s.part_region ? base + np.chain_off[s.part_region - 1] : base + np.scratch_off;
        PartialInput xin{};
        if (s.x_from_prev) {  // (the previous step left its partial sums)
            const NetStep &p = np.steps[i - 1];
            if (p.kind == QCNN_LAYER_FC)
                xin = {reinterpret_cast<const float *>(base + np.chain_off[p.part_region - 1]),
                       p.fcp.splits / p.fcp.cl, layers[i - 1].bias, layers[i - 1].relu};
            else  // a conv layer: in the scratch region, where its call put them
                xin = {reinterpret_cast<const float *>(base + np.scratch_off + p.conv.lut_off),
                       conv_groups(p.conv), layers[i - 1].bias, layers[i - 1].relu};
        }
        qcnn_status rc = run_step(layers[i], s, in, out, scratch, st, s.x_from_prev ? &xin : nullptr);
        if (rc != QCNN_OK) return rc;
        in = out;
    }
    return QCNN_OK;
}

// Per device: the stream that copies host input slices and the events that
// order them, created on the first qcnn_net_forward_host call on that device
// and kept for the life of the process.  The mutex serializes host-I/O calls
// on one device (each ends with a stream synchronization anyway).
constexpr int kHostChunksMax = 4;
struct HostIo {
    std::mutex mu;
    bool ok = false;
    cudaStream_t copy = nullptr;
    cudaEvent_t start = nullptr, ready[kHostChunksMax] = {};
};

HostIo *host_io(int dev) {
    static HostIo slots[64];
    if (dev < 0 || dev >= 64) return nullptr;
    return &slots[dev];
}

bool host_io_init(HostIo &h) {  // called with h.mu held
    if (h.ok) return true;
    if (cudaStreamCreateWithFlags(&h.copy, cudaStreamNonBlocking) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    bool ok = cudaEventCreateWithFlags(&h.start, cudaEventDisableTiming) == cudaSuccess;
    for (int c = 0; ok && c < kHostChunksMax; ++c)
        ok = cudaEventCreateWithFlags(&h.ready[c], cudaEventDisableTiming) == cudaSuccess;
    if (!ok) {  // undo, so that a later call starts from scratch
        cudaGetLastError();
        for (cudaEvent_t &e : h.ready)
            if (e) cudaEventDestroy(e), e = nullptr;
        if (h.start) cudaEventDestroy(h.start), h.start = nullptr;
        cudaStreamDestroy(h.copy);
        h.copy = nullptr;
        return false;
    }
    h.ok = true;
    return true;
}

}  // namespace

namespace qcnn {

qcnn_status fc_forward_limited(const float *x, int N, int Cs, int Ct, const float *D, int Csp,
                               int K, const uint8_t *codes, const float *bias, float *y,
                               int relu, size_t max_partial_bytes,
                               qcnn_status (*get_scratch)(void **), cudaStream_t st) {
    FcShape s;
    if (!x || !D || !codes || !y || !fc_shape(N, Cs, Ct, Csp, K, QCNN_LUT_FP32, &s))
        return QCNN_ERR_INVALID_ARG;
    if (!f32_ok(x) || !f32_ok(D) || !f32_ok(y) || !f32_ok(bias)) return QCNN_ERR_INVALID_ARG;
    const FcPlan p = plan_fc(s, max_partial_bytes);
    void *scratch = nullptr;
    if (p.partial_bytes > 0) {
        if (p.partial_bytes > max_partial_bytes) return QCNN_ERR_WORKSPACE;
        const qcnn_status rc = get_scratch(&scratch);
        if (rc != QCNN_OK) return rc;
    }
    PdlScope pdl;
    return launch_fc(s, p, x, D, codes, bias, y, relu, static_cast<float *>(scratch), st);
}

}  // namespace qcnn

extern "C" {

const char *qcnn_status_string(qcnn_status s) {
    switch (s) {
        case QCNN_OK: return "ok";
        case QCNN_ERR_INVALID_ARG: return "invalid argument";
        case QCNN_ERR_UNSUPPORTED: return "unsupported by this build";
        case QCNN_ERR_WORKSPACE: return "workspace too small or misaligned";
        case QCNN_ERR_CUDA: return "CUDA error";
        case QCNN_ERR_DATA: return "input data unusable (rank-deficient calibration set)";
        case QCNN_ERR_DEVICE_CHECK:
            return "a kernel found a code >= K or an index outside its arrays (debug build)";
    }
    return "unknown status";
}

int qcnn_debug_checks(void) {
#ifdef QCNN_DEBUG_CHECKS
    return 1;
#else
    return 0;
#endif
}

qcnn_status qcnn_device_check(void *stream, unsigned *flags) {
    if (flags) *flags = 0;
    qcnn_status rc = cuda_status(cudaStreamSynchronize(as_stream(stream)));
    if (rc != QCNN_OK) return rc;
    unsigned f = 0;
    if ((rc = collect_device_checks(&f)) != QCNN_OK) return rc;
    if (flags) *flags = f;
    return f ? QCNN_ERR_DEVICE_CHECK : QCNN_OK;
}

int qcnn_last_cuda_error(void) { return g_last_cuda_error.load(); }

uint64_t qcnn_launch_count(void) { return g_launches.load(); }

qcnn_status qcnn_lut_build(const float *x, int N, int Cs, int H, int W, const float *D, int Csp,
                           int K, void *lut, int lut_type, void *stream) {
    if (!x || !D || !lut || N <= 0 || H <= 0 || W <= 0 || !pq_ok(Cs, Csp, K) ||
        !lut_type_ok(lut_type))
        return QCNN_ERR_INVALID_ARG;
    if (!f32_ok(x) || !f32_ok(D) || !aligned(lut, lut_type == QCNN_LUT_BF16 ? 2 : 4))
        return QCNN_ERR_INVALID_ARG;
    const long long P = (long long)H * W;
    if (!fits_int((long long)N * Cs * P) || !fits_int((long long)N * (Cs / Csp) * P * K))
        return QCNN_ERR_INVALID_ARG;
    PdlScope pdl;
    return launch_lut_build(x, N, Cs, (int)P, D, Csp, K, lut, lut_type == QCNN_LUT_BF16,
                            as_stream(stream));
}

qcnn_status qcnn_fc_workspace_size(int N, int Cs, int Ct, int Csp, int K, int lut_type,
                                   size_t *bytes) {
    FcShape s;
    if (!bytes || !fc_shape(N, Cs, Ct, Csp, K, lut_type, &s)) return QCNN_ERR_INVALID_ARG;
    *bytes = align_up(plan_fc(s).partial_bytes, kWsAlign);
    return QCNN_OK;
}

qcnn_status qcnn_fc_forward(const float *x, int N, int Cs, int Ct, const float *D, int Csp,
                            int K, const uint8_t *codes, const float *bias, float *y, int relu,
                            int lut_type, void *workspace, size_t workspace_bytes,
                            void *stream) {
    FcShape s;
    if (!x || !D || !codes || !y || !fc_shape(N, Cs, Ct, Csp, K, lut_type, &s))
        return QCNN_ERR_INVALID_ARG;
    if (!f32_ok(x) || !f32_ok(D) || !f32_ok(y) || !f32_ok(bias)) return QCNN_ERR_INVALID_ARG;
    const FcPlan p = plan_fc(s);
    if (!ws_ok(workspace, workspace_bytes, p.partial_bytes)) return QCNN_ERR_WORKSPACE;
    PdlScope pdl;
    return launch_fc(s, p, x, D, codes, bias, y, relu, static_cast<float *>(workspace),
                     as_stream(stream));
}

qcnn_status qcnn_fc_forward_packed(const float *x, int N, int Cs, int Ct, const float *D,
                                   int Csp, int K, const uint8_t *packed, const float *bias,
                                   float *y, int relu, int lut_type, void *workspace,
                                   size_t workspace_bytes, void *stream) {
    FcShape s;
    if (!x || !D || !packed || !y || !fc_shape(N, Cs, Ct, Csp, K, lut_type, &s))
        return QCNN_ERR_INVALID_ARG;
    if (!aligned(packed, 16) || !f32_ok(x) || !f32_ok(D) || !f32_ok(y) || !f32_ok(bias))
        return QCNN_ERR_INVALID_ARG;
    s.code_bits = code_bits(K);
    const FcPlan p = plan_fc(s);
    if (!ws_ok(workspace, workspace_bytes, p.partial_bytes)) return QCNN_ERR_WORKSPACE;
    PdlScope pdl;
    return launch_fc(s, p, x, D, packed, bias, y, relu, static_cast<float *>(workspace),
                     as_stream(stream));
}

size_t qcnn_conv_packed_codes_bytes(int Ct, int kh, int kw, int M) {
    if (Ct <= 0 || kh <= 0 || kw <= 0 || M <= 0) return 0;
    return packed_codes_bytes(Ct, kh * kw, M);
}

qcnn_status qcnn_conv_pack_codes(const uint8_t *codes, int Ct, int kh, int kw, int M, int K,
                                 uint8_t *packed, void *stream) {
    if (!codes || !packed || Ct <= 0 || kh <= 0 || kw <= 0 || M <= 0 || K < 1 || K > kMaxK)
        return QCNN_ERR_INVALID_ARG;
    if (!fits_int((long long)packed_ct(Ct) * kh * kw * M)) return QCNN_ERR_INVALID_ARG;
    return launch_pack_codes(codes, Ct, kh * kw, M, K, packed, as_stream(stream));
}

int qcnn_conv_fused_variant_count(void) { return conv_fused_variant_count(); }

qcnn_status qcnn_conv_fused_variant_info(int v, int info[10]) {
    if (!info || v < 0 || v >= conv_fused_variant_count()) return QCNN_ERR_INVALID_ARG;
    conv_fused_variant_info(v, info);
    return QCNN_OK;
}

qcnn_status qcnn_conv_workspace_size(int N, int Cs, int H, int W, int Ct, int kh, int kw,
                                     int stride, int pad, int Csp, int K, int codes_layout,
                                     int algo, int lut_type, size_t *bytes) {
    ConvShape s;
    if (!bytes || !conv_shape(N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K, lut_type, &s))
        return QCNN_ERR_INVALID_ARG;
    ConvCall c;
    qcnn_status rc = plan_conv_call_cached(s, codes_layout, algo, &c);
    if (rc != QCNN_OK) return rc;
    *bytes = c.total;
    return QCNN_OK;
}

qcnn_status qcnn_conv_plan_info(int N, int Cs, int H, int W, int Ct, int kh, int kw, int stride,
                                int pad, int Csp, int K, int codes_layout, int algo,
                                int lut_type, int info[8]) {
    ConvShape s;
    if (!info || !conv_shape(N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K, lut_type, &s))
        return QCNN_ERR_INVALID_ARG;
    ConvCall c;
    const qcnn_status rc = plan_conv_call_cached(s, codes_layout, algo, &c);
    if (rc != QCNN_OK) return rc;
    for (int i = 0; i < 8; ++i) info[i] = 0;
    info[0] = c.algo;
    info[7] = 1;
    if (c.algo == QCNN_ALGO_FUSED) {
        const ConvFusedPlan &p = c.fp;
        info[1] = p.variant;
        info[2] = p.ST;
        info[3] = p.ct_cta;
        info[4] = p.splits;
        info[5] = p.sk;
        info[6] = p.sk ? p.sk_ctas : p.pos_tiles * p.ct_tiles * s.N * p.splits;
        info[7] = p.cl;
    } else if (c.algo == QCNN_ALGO_PHASE) {
        const ConvPhasePlan &p = c.pp;
        info[1] = p.variant;
        info[2] = p.ST;
        info[3] = p.ct_cta;
        info[4] = p.splits;
        info[6] = p.pos_tiles * p.ct_tiles * s.N * p.splits;
        info[7] = p.cl;
    } else if (c.algo == QCNN_ALGO_CHUNKED) {
        const ConvChunkPlan &p = c.cp;
        info[1] = p.variant;
        info[3] = p.ct_cta;
        info[4] = 1;
        info[6] = p.row_tiles * p.ct_tiles * s.N;
    } else {
        info[1] = -1;
        info[4] = 1;
    }
    return QCNN_OK;
}

qcnn_status qcnn_fc_plan_info(int N, int Cs, int Ct, int Csp, int K, int lut_type, int info[6]) {
    FcShape s;
    if (!info || !fc_shape(N, Cs, Ct, Csp, K, lut_type, &s)) return QCNN_ERR_INVALID_ARG;
    const FcPlan p = plan_fc(s);
    info[0] = p.NT;
    info[1] = p.CT_CTA;
    info[2] = p.splits;
    info[3] = p.MCH;
    info[4] = p.ct_tiles * p.n_tiles * p.splits;
    info[5] = p.cl;
    return QCNN_OK;
}

qcnn_status qcnn_conv_forward(const float *x, int N, int Cs, int H, int W, int Ct, int kh,
                              int kw, int stride, int pad, const float *D, int Csp, int K,
                              const uint8_t *codes, int codes_layout, const float *bias,
                              float *y, int relu, int algo, int lut_type, void *workspace,
                              size_t workspace_bytes, void *stream) {
    ConvShape s;
    if (!x || !D || !codes || !y ||
        !conv_shape(N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K, lut_type, &s))
        return QCNN_ERR_INVALID_ARG;
    if (!f32_ok(x) || !f32_ok(D) || !f32_ok(y) || !f32_ok(bias) ||
        (codes_layout == QCNN_CODES_PACKED && !aligned(codes, 16)))
        return QCNN_ERR_INVALID_ARG;
    ConvCall c;
    qcnn_status rc = plan_conv_call_cached(s, codes_layout, algo, &c);
    if (rc != QCNN_OK) return rc;
    if (!ws_ok(workspace, workspace_bytes, c.total)) return QCNN_ERR_WORKSPACE;
    PdlScope pdl;
    return run_conv(c, x, D, codes, codes_layout, bias, y, relu, workspace, as_stream(stream));
}

qcnn_status qcnn_maxpool(const float *x, int N, int C, int H, int W, int k, int s, float *y,
                         void *stream) {
    if (!x || !y || N <= 0 || C <= 0 || H <= 0 || W <= 0 || k <= 0 || s <= 0 || k > H || k > W)
        return QCNN_ERR_INVALID_ARG;
    if (!f32_ok(x) || !f32_ok(y)) return QCNN_ERR_INVALID_ARG;
    if (!fits_int((long long)N * C * H * W)) return QCNN_ERR_INVALID_ARG;
    return launch_maxpool(x, N, C, H, W, k, s, y, as_stream(stream));
}

qcnn_status qcnn_net_output_shape(const qcnn_layer *layers, int n_layers, int C, int H, int W,
                                  int *out_C, int *out_H, int *out_W) {
    if (!out_C || !out_H || !out_W) return QCNN_ERR_INVALID_ARG;
    NetPlan np;
    qcnn_status rc = plan_net_cached(layers, n_layers, 1, C, H, W, 0, &np);
    if (rc != QCNN_OK) return rc;
    *out_C = np.steps.back().oC;
    *out_H = np.steps.back().oH;
    *out_W = np.steps.back().oW;
    return QCNN_OK;
}

qcnn_status qcnn_net_workspace_size(const qcnn_layer *layers, int n_layers, int N, int C, int H,
                                    int W, int host_io, size_t *bytes) {
    if (!bytes) return QCNN_ERR_INVALID_ARG;
    NetPlan np;
    qcnn_status rc = plan_net_cached(layers, n_layers, N, C, H, W, host_io, &np);
    if (rc != QCNN_OK) return rc;
    *bytes = np.total;
    return QCNN_OK;
}

qcnn_status qcnn_net_plan_info(const qcnn_layer *layers, int n_layers, int N, int C, int H,
                               int W, int host_io, int *info) {
    if (!info) return QCNN_ERR_INVALID_ARG;
    NetPlan np;
    qcnn_status rc = plan_net_cached(layers, n_layers, N, C, H, W, host_io, &np);
    if (rc != QCNN_OK) return rc;
    for (int i = 0; i < n_layers; ++i) {
        info[2 * i] = np.steps[i].leave_partials;
        info[2 * i + 1] = np.steps[i].x_from_prev;
    }
    return QCNN_OK;
}

qcnn_status qcnn_net_forward(const qcnn_layer *layers, int n_layers, const float *x, int N,
                             int C, int H, int W, float *y, void *workspace,
                             size_t workspace_bytes, void *stream) {
    if (!x || !y || !f32_ok(x) || !f32_ok(y)) return QCNN_ERR_INVALID_ARG;
    NetPlan np;
    qcnn_status rc = plan_net_cached(layers, n_layers, N, C, H, W, 0, &np);
    if (rc != QCNN_OK) return rc;
    if (!layer_pointers_ok(layers, n_layers)) return QCNN_ERR_INVALID_ARG;
    if (!ws_ok(workspace, workspace_bytes, np.total)) return QCNN_ERR_WORKSPACE;
    PdlScope pdl;
    return run_net(layers, np, x, y, workspace, as_stream(stream));
}

qcnn_status qcnn_net_forward_host(const qcnn_layer *layers, int n_layers, const float *x_host,
                                  int N, int C, int H, int W, float *y_host, void *workspace,
                                  size_t workspace_bytes, void *stream) {
    if (!x_host || !y_host) return QCNN_ERR_INVALID_ARG;
    NetPlan np;
    qcnn_status rc = plan_net_cached(layers, n_layers, N, C, H, W, 1, &np);
    if (rc != QCNN_OK) return rc;
    if (!layer_pointers_ok(layers, n_layers)) return QCNN_ERR_INVALID_ARG;
    if (!ws_ok(workspace, workspace_bytes, np.total)) return QCNN_ERR_WORKSPACE;
    cudaStream_t st = as_stream(stream);
    PdlScope pdl;
    uint8_t *base = static_cast<uint8_t *>(workspace);
    float *xd = reinterpret_cast<float *>(base + np.xin_off);
    float *yd = reinterpret_cast<float *>(base + np.yout_off);
    const NetStep &last = np.steps.back();
    const size_t xb = (size_t)N * C * H * W * sizeof(float);
    const size_t yb = (size_t)N * last.oC * last.oH * last.oW * sizeof(float);
    int dev = 0;
    HostIo *hio = cudaGetDevice(&dev) == cudaSuccess ? host_io(dev) : nullptr;
    cudaGetLastError();
    std::unique_lock<std::mutex> lock;
    if (np.chunks > 1 && hio) {
        lock = std::unique_lock<std::mutex>(hio->mu);
        if (!host_io_init(*hio)) {
            lock.unlock();
            hio = nullptr;
        }
    }
    if (np.chunks > 1 && hio) {
        // slice c of the input is copied on the copy stream (after the work
        // already queued on `stream`), and the first layer runs on it as soon
        // as it has arrived, while the later slices are still copying
        const int nc = np.chunks;
        const size_t xs = xb / nc;
        const NetStep &s0 = np.step0c;
        const size_t ys = (size_t)s0.N * s0.oC * s0.oH * s0.oW;
        float *y0 = np.steps.size() == 1 ? yd : reinterpret_cast<float *>(base + np.act_off[0]);
        rc = cuda_status(cudaEventRecord(hio->start, st));
        if (rc == QCNN_OK) rc = cuda_status(cudaStreamWaitEvent(hio->copy, hio->start, 0));
        for (int c = 0; c < nc && rc == QCNN_OK; ++c) {
            rc = cuda_status(cudaMemcpyAsync(reinterpret_cast<uint8_t *>(xd) + c * xs,
                                             reinterpret_cast<const uint8_t *>(x_host) + c * xs,
                                             xs, cudaMemcpyHostToDevice, hio->copy));
            if (rc == QCNN_OK) rc = cuda_status(cudaEventRecord(hio->ready[c], hio->copy));
        }
        for (int c = 0; c < nc && rc == QCNN_OK; ++c) {
            rc = cuda_status(cudaStreamWaitEvent(st, hio->ready[c], 0));
            pdl_break();  // the first kernel on slice c waits for its copy in full
            if (rc == QCNN_OK)
                rc = run_step(layers[0], s0, xd + (size_t)c * (xs / sizeof(float)), y0 + c * ys,
                              base + np.scratch_off, st);
        }
        if (rc == QCNN_OK && np.steps.size() > 1) rc = run_net(layers, np, y0, yd, workspace, st, 1);
    } else {
        rc = cuda_status(cudaMemcpyAsync(xd, x_host, xb, cudaMemcpyHostToDevice, st));
        if (rc == QCNN_OK) rc = run_net(layers, np, xd, yd, workspace, st);
    }
    if (rc == QCNN_OK) rc = cuda_status(cudaMemcpyAsync(y_host, yd, yb, cudaMemcpyDeviceToHost, st));
    const qcnn_status sync = sync_and_check(st);
    return rc != QCNN_OK ? rc : sync;
}

}  // extern "C"
