// conv_fused_tc.cu -- instantiates the tiles with the table build on the tensor cores of the fused
// conv kernel (conv_fused.cuh); one unit per group so that they compile in
// parallel.
// kernels of this unit record wait time-outs in every build
#define QCNN_UNIT_RECORDS
#include "conv_fused.cuh"

namespace qcnn {

static const FusedVariant kPart[] = {
    QCNN_FUSED_TC(6, 8, 1, 16, 1.0, 0.6), QCNN_FUSED_TC(7, 8, 1, 16, 1.0, 0.6),
    QCNN_FUSED_TC(4, 16, 1, 16, 1.0, 0.6), QCNN_FUSED_TC(5, 16, 1, 16, 1.0, 0.6),
    QCNN_FUSED_TC(4, 8, 1, 16, 1.0, 0.6), QCNN_FUSED_TC(5, 8, 1, 16, 1.0, 0.6),
    QCNN_FUSED_TC(6, 16, 1, 12, 1.0, 0.6)};

const FusedVariant *fused_variants_tc(int *n) {
    *n = (int)(sizeof(kPart) / sizeof(kPart[0]));
    return kPart;
}

}  // namespace qcnn
