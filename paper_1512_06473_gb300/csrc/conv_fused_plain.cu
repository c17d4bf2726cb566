// conv_fused_plain.cu -- instantiates the fp32-table tiles (C'_s width 4 and 8) of the fused
// conv kernel (conv_fused.cuh); one unit per group so that they compile in
// parallel.
#include "conv_fused.cuh"

namespace qcnn {

static const FusedVariant kPart[] = {
    QCNN_FUSED_SET(4), QCNN_FUSED_SET(8)};

const FusedVariant *fused_variants_plain(int *n) {
    *n = (int)(sizeof(kPart) / sizeof(kPart[0]));
    return kPart;
}

// 64-channel tiles (4 channels per warp): layers with Ct <= 64, where the
// 128-channel tiles gather half their look-ups for channels past Ct
static const FusedVariant kNarrow[] = {
    QCNN_FUSED(7, 4, 1, 4, 16, 1, false, 0.9, 1.0), QCNN_FUSED(7, 4, 1, 8, 16, 1, false, 0.9, 1.0)};

const FusedVariant *fused_variants_narrow(int *n) {
    *n = (int)(sizeof(kNarrow) / sizeof(kNarrow[0]));
    return kNarrow;
}

}  // namespace qcnn
