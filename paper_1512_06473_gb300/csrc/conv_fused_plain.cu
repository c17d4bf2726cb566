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

}  // namespace qcnn
