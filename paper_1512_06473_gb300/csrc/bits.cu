// bits.cu -- sub-codeword indices stored in b = ceil(log2 K) bits each, the
// storage model of Table 1 (Sec. 3.4).
//
// Stream layout: code i occupies stream bits [i*b, (i+1)*b), its bit t at
// stream bit i*b + t; stream bit s is bit (s mod 8) of byte s / 8.
// FC row layout (what the FC kernels read): row m of the [M][Ct] codes packed
// on its own and zero-padded to a pitch that is a multiple of 16 bytes, so
// a CTA's slice of a row is a whole number of 16-byte copies.
#include "qcnn_internal.cuh"

#include <algorithm>

namespace qcnn {

int code_bits(int K) {
    int b = 1;
    while ((1 << b) < K) ++b;
    return b;
}

size_t fc_packed_pitch(int Ct, int K) {
    return align_up(((size_t)Ct * code_bits(K) + 7) / 8, 16);
}

// One thread per output byte: gathers the bits of the codes it overlaps.
__global__ void pack_bits_kernel(const uint8_t *__restrict__ codes, long long n, int b,
                                 long long row_len, long long rows, long long in_pitch,
                                 long long out_pitch, int kmax, uint8_t *__restrict__ out) {
    const long long row_bytes = (row_len * b + 7) / 8;
    const long long total = rows * out_pitch;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const long long r = i / out_pitch, byte = i % out_pitch;
        unsigned v = 0;
        if (byte < row_bytes) {
            const uint8_t *c = codes + r * in_pitch;
            for (int t = 0; t < 8; ++t) {
                const long long s = byte * 8 + t;
                const long long ci = s / b;
                if (ci < row_len) {
                    QCNN_CHECK((unsigned)c[ci] <= (unsigned)kmax, QCNN_CHECK_CODE);
                    const unsigned code = min((unsigned)c[ci], (unsigned)kmax);
                    v |= ((code >> (s - ci * b)) & 1u) << t;
                }
            }
        }
        out[i] = (uint8_t)v;
    }
    (void)n;
}

// One thread per code.
__global__ void unpack_bits_kernel(const uint8_t *__restrict__ in, long long n, int b,
                                   uint8_t *__restrict__ codes) {
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x) {
        const long long s = i * b;
        const long long B = s >> 3;
        const int sh = (int)(s & 7);
        unsigned w = in[B];
        if (sh + b > 8) w |= (unsigned)in[B + 1] << 8;
        codes[i] = (uint8_t)((w >> sh) & ((1u << b) - 1u));
    }
}

static int grid_for(long long n) {
    return (int)std::max<long long>(1, std::min<long long>((n + 255) / 256, (long long)num_sms() * 16));
}

qcnn_status launch_pack_bits(const uint8_t *codes, long long row_len, long long rows,
                             long long in_pitch, long long out_pitch, int b, int K, uint8_t *out,
                             cudaStream_t st) {
    pack_bits_kernel<<<grid_for(rows * out_pitch), 256, 0, st>>>(codes, row_len * rows, b,
                                                                 row_len, rows, in_pitch,
                                                                 out_pitch, K - 1, out);
    return after_launch();
}

qcnn_status launch_unpack_bits(const uint8_t *in, long long n, int b, uint8_t *codes,
                               cudaStream_t st) {
    unpack_bits_kernel<<<grid_for(n), 256, 0, st>>>(in, n, b, codes);
    return after_launch();
}

}  // namespace qcnn

using namespace qcnn;

extern "C" {

int qcnn_code_bits(int K) { return (K >= 1 && K <= kMaxK) ? code_bits(K) : 0; }

qcnn_status qcnn_pack_bits(const uint8_t *codes, long long n, int bits, uint8_t *stream,
                           void *cuda_stream) {
    if (!codes || !stream || n <= 0 || bits < 1 || bits > 8) return QCNN_ERR_INVALID_ARG;
    const long long bytes = (n * bits + 7) / 8;
    return launch_pack_bits(codes, n, 1, n, bytes, bits, 1 << bits, stream,
                            reinterpret_cast<cudaStream_t>(cuda_stream));
}

qcnn_status qcnn_unpack_bits(const uint8_t *stream, long long n, int bits, uint8_t *codes,
                             void *cuda_stream) {
    if (!codes || !stream || n <= 0 || bits < 1 || bits > 8) return QCNN_ERR_INVALID_ARG;
    return launch_unpack_bits(stream, n, bits, codes, reinterpret_cast<cudaStream_t>(cuda_stream));
}

size_t qcnn_fc_packed_codes_bytes(int M, int Ct, int K) {
    if (M <= 0 || Ct <= 0 || K < 1 || K > kMaxK) return 0;
    return (size_t)M * fc_packed_pitch(Ct, K);
}

qcnn_status qcnn_fc_pack_codes(const uint8_t *codes, int M, int Ct, int K, uint8_t *packed,
                               void *stream) {
    if (!codes || !packed || M <= 0 || Ct <= 0 || K < 1 || K > kMaxK) return QCNN_ERR_INVALID_ARG;
    return launch_pack_bits(codes, Ct, M, Ct, (long long)fc_packed_pitch(Ct, K), code_bits(K), K,
                            packed, reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"
