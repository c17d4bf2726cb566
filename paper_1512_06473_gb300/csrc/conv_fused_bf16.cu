// conv_fused_bf16.cu -- instantiates the bfloat16-table tiles of the fused
// conv kernel (conv_fused.cuh); one unit per group so that they compile in
// parallel.
#include "conv_fused.cuh"

namespace qcnn {

static const FusedVariant kPart[] = {
    QCNN_FUSED_BF_SET(4), QCNN_FUSED_BF_SET(8)};

const FusedVariant *fused_variants_bf16(int *n) {
    *n = (int)(sizeof(kPart) / sizeof(kPart[0]));
    return kPart;
}

}  // namespace qcnn
