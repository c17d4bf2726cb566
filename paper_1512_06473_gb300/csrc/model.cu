// model.cu -- a Q-CNN model in one blob: every layer's sub-codebooks, codes
// stored in ceil(log2 K) bits (the storage model of Table 1, Sec. 3.4) and
// biases; plus its loader, which uploads a blob into one caller-provided
// device buffer and lays the codes out for the kernels.
//
// Blob layout (little-endian, every array 16-byte aligned in the payload):
//   header   (32 B)  magic "QCNNMDL1", u32 version = 1, u32 n_layers,
//                    u32 C, H, W (input of one image), u32 reserved
//   records  (80 B each) u32 kind, Ct, kh, kw, stride, pad, Csp, K, relu,
//                    bits, has_bias, Cs; u64 off_D, off_codes, off_bias,
//                    u64 reserved  (offsets from the payload start)
//   payload  D [M][K][Csp] fp32; codes as one bit stream in the canonical
//            order (FC [M][Ct]; conv [Ct][kh*kw][M]); bias [Ct] fp32
// A max-pool record uses kh (= kw) and stride and has no arrays.
#include "qcnn_internal.cuh"

#include <algorithm>
#include <climits>
#include <cstring>
#include <vector>

namespace qcnn {
namespace {

constexpr char kMagic[8] = {'Q', 'C', 'N', 'N', 'M', 'D', 'L', '1'};
constexpr uint32_t kVersion = 1;
constexpr size_t kHeaderBytes = 32, kRecordBytes = 80;

struct Rec {
    uint32_t kind, Ct, kh, kw, stride, pad, Csp, K, relu, bits, has_bias, Cs;
    uint64_t off_D, off_codes, off_bias, reserved;
};
static_assert(sizeof(Rec) == kRecordBytes, "record layout");

size_t a16(size_t v) { return (v + 15) / 16 * 16; }

template <typename T>
void put(uint8_t *p, const T &v) {
    std::memcpy(p, &v, sizeof(T));
}

// Shapes of every layer, checked like the network planner does.
struct LayerGeo {
    int Cs, H, W, oC, oH, oW, M, kk;
    size_t nD, ncodes, stream_bytes;
};

bool layer_geo(const Rec &r, int C, int H, int W, LayerGeo *g) {
    g->Cs = C;
    g->H = H;
    g->W = W;
    if (r.kind == QCNN_LAYER_MAXPOOL) {
        if (r.kh < 1 || r.stride < 1 || (int)r.kh > H || (int)r.kh > W) return false;
        g->oC = C;
        g->oH = (H - (int)r.kh) / (int)r.stride + 1;
        g->oW = (W - (int)r.kh) / (int)r.stride + 1;
        g->M = g->kk = 0;
        g->nD = g->ncodes = g->stream_bytes = 0;
        return true;
    }
    if (r.Csp < 1 || r.Csp > (uint32_t)kMaxCsp || r.K < 1 || r.K > (uint32_t)kMaxK || r.Ct < 1 ||
        r.Ct > (uint32_t)INT_MAX)
        return false;
    long long cs = C;
    int kk = 1;
    if (r.kind == QCNN_LAYER_FC) {
        cs = (long long)C * H * W;
        g->oC = (int)r.Ct;
        g->oH = g->oW = 1;
    } else if (r.kind == QCNN_LAYER_CONV) {
        if (r.kh < 1 || r.kw < 1 || r.stride < 1 || r.pad > 1024u) return false;
        const int hp = H + 2 * (int)r.pad, wp = W + 2 * (int)r.pad;
        if (hp < (int)r.kh || wp < (int)r.kw) return false;
        g->oC = (int)r.Ct;
        g->oH = (hp - (int)r.kh) / (int)r.stride + 1;
        g->oW = (wp - (int)r.kw) / (int)r.stride + 1;
        kk = (int)(r.kh * r.kw);
    } else {
        return false;
    }
    if (cs >= INT_MAX || cs % r.Csp != 0) return false;
    if (r.Cs != 0 && (long long)r.Cs != cs) return false;
    g->Cs = (int)cs;
    g->M = (int)(cs / r.Csp);
    g->kk = kk;
    g->nD = (size_t)g->M * r.K * r.Csp;
    g->ncodes = (size_t)g->M * r.Ct * kk;
    g->stream_bytes = (g->ncodes * code_bits((int)r.K) + 7) / 8;
    return true;
}

void pack_host(const uint8_t *codes, size_t n, int b, int K, uint8_t *out) {
    std::memset(out, 0, (n * b + 7) / 8);
    for (size_t i = 0; i < n; ++i) {
        const unsigned c = std::min<unsigned>(codes[i], (unsigned)K - 1);
        for (int t = 0; t < b; ++t)
            if ((c >> t) & 1u) out[(i * b + t) >> 3] |= (uint8_t)(1u << ((i * b + t) & 7));
    }
}

// Parse and validate; fills the records and the geometry of every layer.
qcnn_status parse(const void *blob, size_t bytes, std::vector<Rec> *recs,
                  std::vector<LayerGeo> *geo, int *C, int *H, int *W, size_t *payload) {
    if (!blob || bytes < kHeaderBytes) return QCNN_ERR_INVALID_ARG;
    const uint8_t *p = static_cast<const uint8_t *>(blob);
    if (std::memcmp(p, kMagic, 8) != 0) return QCNN_ERR_INVALID_ARG;
    uint32_t ver, n, c, h, w;
    std::memcpy(&ver, p + 8, 4);
    std::memcpy(&n, p + 12, 4);
    std::memcpy(&c, p + 16, 4);
    std::memcpy(&h, p + 20, 4);
    std::memcpy(&w, p + 24, 4);
    if (ver != kVersion || n < 1 || n > 4096 || c < 1 || h < 1 || w < 1 ||
        (long long)c * h * w >= INT_MAX)
        return QCNN_ERR_INVALID_ARG;
    const size_t pay = kHeaderBytes + (size_t)n * kRecordBytes;
    if (bytes < pay) return QCNN_ERR_INVALID_ARG;
    recs->resize(n);
    geo->resize(n);
    int cc = (int)c, hh = (int)h, ww = (int)w;
    for (uint32_t i = 0; i < n; ++i) {
        Rec &r = (*recs)[i];
        std::memcpy(&r, p + kHeaderBytes + i * kRecordBytes, kRecordBytes);
        LayerGeo &g = (*geo)[i];
        if (!layer_geo(r, cc, hh, ww, &g)) return QCNN_ERR_INVALID_ARG;
        if (r.kind != QCNN_LAYER_MAXPOOL) {
            if (r.bits != (uint32_t)code_bits((int)r.K)) return QCNN_ERR_INVALID_ARG;
            auto fits = [&](uint64_t off, size_t len) {
                return off % 16 == 0 && off <= bytes - pay && len <= bytes - pay - off;
            };
            if (!fits(r.off_D, g.nD * 4) || !fits(r.off_codes, g.stream_bytes) ||
                (r.has_bias && !fits(r.off_bias, (size_t)r.Ct * 4)))
                return QCNN_ERR_INVALID_ARG;
        }
        cc = g.oC;
        hh = g.oH;
        ww = g.oW;
    }
    *C = (int)c;
    *H = (int)h;
    *W = (int)w;
    *payload = pay;
    return QCNN_OK;
}

// Device buffer carve-up for an upload: per layer D, bias, kernel-layout
// codes; then one staging area for a bit stream and one for canonical codes.
struct DevLayout {
    std::vector<size_t> D, bias, codes;
    size_t stream_stage, canon_stage, total;
};

DevLayout dev_layout(const std::vector<Rec> &recs, const std::vector<LayerGeo> &geo) {
    DevLayout L;
    size_t off = 0, max_stream = 0, max_canon = 0;
    for (size_t i = 0; i < recs.size(); ++i) {
        const Rec &r = recs[i];
        const LayerGeo &g = geo[i];
        L.D.push_back(off);
        L.bias.push_back(0);
        L.codes.push_back(0);
        if (r.kind == QCNN_LAYER_MAXPOOL) continue;
        off += align_up(g.nD * 4, kWsAlign);
        L.bias[i] = off;
        if (r.has_bias) off += align_up((size_t)r.Ct * 4, kWsAlign);
        L.codes[i] = off;
        const size_t kb = r.kind == QCNN_LAYER_FC
                              ? (size_t)g.M * fc_packed_pitch((int)r.Ct, (int)r.K)
                              : packed_codes_bytes((int)r.Ct, g.kk, g.M);
        off += align_up(kb, kWsAlign);
        max_stream = std::max(max_stream, g.stream_bytes);
        max_canon = std::max(max_canon, g.ncodes);
    }
    L.stream_stage = off;
    off += align_up(max_stream, kWsAlign);
    L.canon_stage = off;
    off += align_up(max_canon, kWsAlign);
    L.total = off;
    return L;
}

}  // namespace
}  // namespace qcnn

using namespace qcnn;

extern "C" {

qcnn_status qcnn_model_serialize(const qcnn_layer *layers, int n_layers, int C, int H, int W,
                                 void *out, size_t out_bytes, size_t *bytes_needed) {
    if (!layers || n_layers < 1 || n_layers > 4096 || C < 1 || H < 1 || W < 1 || !bytes_needed)
        return QCNN_ERR_INVALID_ARG;
    std::vector<Rec> recs(n_layers);
    std::vector<LayerGeo> geo(n_layers);
    size_t pay = 0;  // payload bytes
    int c = C, h = H, w = W;
    for (int i = 0; i < n_layers; ++i) {
        const qcnn_layer &L = layers[i];
        Rec r{};
        r.kind = (uint32_t)L.kind;
        r.Ct = (uint32_t)std::max(L.Ct, 0);
        r.kh = (uint32_t)std::max(L.kh, 0);
        r.kw = (uint32_t)std::max(L.kind == QCNN_LAYER_MAXPOOL ? L.kh : L.kw, 0);
        r.stride = (uint32_t)std::max(L.stride, 0);
        r.pad = (uint32_t)std::max(L.pad, 0);
        r.Csp = (uint32_t)std::max(L.Csp, 0);
        r.K = (uint32_t)std::max(L.K, 0);
        r.relu = L.relu ? 1u : 0u;
        if (!layer_geo(r, c, h, w, &geo[i])) return QCNN_ERR_INVALID_ARG;
        if (L.kind != QCNN_LAYER_MAXPOOL) {
            if (!L.D || !L.codes || L.codes_layout != QCNN_CODES_CANONICAL)
                return QCNN_ERR_INVALID_ARG;
            r.Cs = (uint32_t)geo[i].Cs;
            r.bits = (uint32_t)code_bits((int)r.K);
            r.has_bias = L.bias ? 1u : 0u;
            r.off_D = pay;
            pay = a16(pay + geo[i].nD * 4);
            r.off_codes = pay;
            pay = a16(pay + geo[i].stream_bytes);
            r.off_bias = pay;
            if (L.bias) pay = a16(pay + (size_t)r.Ct * 4);
        }
        recs[i] = r;
        c = geo[i].oC;
        h = geo[i].oH;
        w = geo[i].oW;
    }
    const size_t head = kHeaderBytes + (size_t)n_layers * kRecordBytes;
    *bytes_needed = head + pay;
    if (!out) return QCNN_OK;
    if (out_bytes < head + pay) return QCNN_ERR_WORKSPACE;
    uint8_t *o = static_cast<uint8_t *>(out);
    std::memset(o, 0, head + pay);
    std::memcpy(o, kMagic, 8);
    put(o + 8, kVersion);
    put(o + 12, (uint32_t)n_layers);
    put(o + 16, (uint32_t)C);
    put(o + 20, (uint32_t)H);
    put(o + 24, (uint32_t)W);
    uint8_t *pl = o + head;
    for (int i = 0; i < n_layers; ++i) {
        std::memcpy(o + kHeaderBytes + (size_t)i * kRecordBytes, &recs[i], kRecordBytes);
        const qcnn_layer &L = layers[i];
        if (L.kind == QCNN_LAYER_MAXPOOL) continue;
        std::memcpy(pl + recs[i].off_D, L.D, geo[i].nD * 4);
        pack_host(L.codes, geo[i].ncodes, (int)recs[i].bits, (int)recs[i].K, pl + recs[i].off_codes);
        if (L.bias) std::memcpy(pl + recs[i].off_bias, L.bias, (size_t)recs[i].Ct * 4);
    }
    return QCNN_OK;
}

qcnn_status qcnn_model_info(const void *blob, size_t bytes, int *n_layers, int *C, int *H,
                            int *W, size_t *device_bytes) {
    if (!n_layers || !C || !H || !W || !device_bytes) return QCNN_ERR_INVALID_ARG;
    std::vector<Rec> recs;
    std::vector<LayerGeo> geo;
    size_t pay = 0;
    qcnn_status rc = parse(blob, bytes, &recs, &geo, C, H, W, &pay);
    if (rc != QCNN_OK) return rc;
    *n_layers = (int)recs.size();
    *device_bytes = dev_layout(recs, geo).total;
    return QCNN_OK;
}

qcnn_status qcnn_model_upload(const void *blob, size_t bytes, void *device_buffer,
                              size_t device_bytes, qcnn_layer *layers, void *stream) {
    if (!layers) return QCNN_ERR_INVALID_ARG;
    std::vector<Rec> recs;
    std::vector<LayerGeo> geo;
    int C, H, W;
    size_t pay = 0;
    qcnn_status rc = parse(blob, bytes, &recs, &geo, &C, &H, &W, &pay);
    if (rc != QCNN_OK) return rc;
    const DevLayout L = dev_layout(recs, geo);
    if (!device_buffer || device_bytes < L.total ||
        reinterpret_cast<uintptr_t>(device_buffer) % kWsAlign != 0)
        return QCNN_ERR_WORKSPACE;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    uint8_t *dev = static_cast<uint8_t *>(device_buffer);
    const uint8_t *pl = static_cast<const uint8_t *>(blob) + pay;
    uint8_t *stage = dev + L.stream_stage, *canon = dev + L.canon_stage;
    for (size_t i = 0; i < recs.size(); ++i) {
        const Rec &r = recs[i];
        const LayerGeo &g = geo[i];
        qcnn_layer &out = layers[i];
        std::memset(&out, 0, sizeof(out));
        out.kind = (int)r.kind;
        out.Ct = (int)r.Ct;
        out.kh = (int)r.kh;
        out.kw = (int)r.kw;
        out.stride = (int)r.stride;
        out.pad = (int)r.pad;
        out.Csp = (int)r.Csp;
        out.K = (int)r.K;
        out.relu = (int)r.relu;
        out.algo = QCNN_ALGO_AUTO;
        out.lut_type = QCNN_LUT_FP32;
        if (r.kind == QCNN_LAYER_MAXPOOL) continue;
        float *D = reinterpret_cast<float *>(dev + L.D[i]);
        uint8_t *codes = dev + L.codes[i];
        if ((rc = cuda_status(cudaMemcpyAsync(D, pl + r.off_D, g.nD * 4, cudaMemcpyHostToDevice,
                                              st))) != QCNN_OK)
            return rc;
        if (r.has_bias) {
            float *bias = reinterpret_cast<float *>(dev + L.bias[i]);
            if ((rc = cuda_status(cudaMemcpyAsync(bias, pl + r.off_bias, (size_t)r.Ct * 4,
                                                  cudaMemcpyHostToDevice, st))) != QCNN_OK)
                return rc;
            out.bias = bias;
        }
        if ((rc = cuda_status(cudaMemcpyAsync(stage, pl + r.off_codes, g.stream_bytes,
                                              cudaMemcpyHostToDevice, st))) != QCNN_OK)
            return rc;
        if ((rc = launch_unpack_bits(stage, (long long)g.ncodes, (int)r.bits, canon, st)) != QCNN_OK)
            return rc;
        if (r.kind == QCNN_LAYER_FC)
            rc = launch_pack_bits(canon, r.Ct, g.M, r.Ct,
                                  (long long)fc_packed_pitch((int)r.Ct, (int)r.K), (int)r.bits,
                                  (int)r.K, codes, st);
        else
            rc = launch_pack_codes(canon, (int)r.Ct, g.kk, g.M, (int)r.K, codes, st);
        if (rc != QCNN_OK) return rc;
        out.D = D;
        out.codes = codes;
        out.codes_layout = QCNN_CODES_PACKED;
    }
    // the staging areas are reused layer after layer and the blob is read by
    // the copies: finish before returning
    return sync_and_check(st);
}

}  // extern "C"
