// conv_fused_sk.cu -- instantiates the stream-K tiles of the fused
// conv kernel (conv_fused.cuh); one unit per group so that they compile in
// parallel.
#include "conv_fused.cuh"

namespace qcnn {

static const FusedVariant kPart[] = {
    QCNN_FUSED_SK_SET(4), QCNN_FUSED_SK_SET(8)};

const FusedVariant *fused_variants_sk(int *n) {
    *n = (int)(sizeof(kPart) / sizeof(kPart[0]));
    return kPart;
}

}  // namespace qcnn
