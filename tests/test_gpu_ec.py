"""Error-corrected FC quantization (Eq. 8 - 12) through the C ABI against the
float64 oracle (oracle/ec.py).

Both sides work in double and take the Eq. 12 argmin in double; only the
order of the sums over calibration vectors differs (chunks on the GPU), so
the codes must be identical and the codewords agree to 1e-9 of their size."""
import numpy as np
import pytest
import torch

import oracle
import oracle.ec as ec
import paper_1512_06473_gb300 as q
import synth
from test_gpu_parity import cuda, host
from test_gpu_quantize import init_from, subvectors_fc

pytestmark = pytest.mark.gpu


def calib(seed, N, Cs, Ct, Csp, K):
    """Calibration pairs for a dense layer W: S post-ReLU activations, T = S W^T
    (the original layer's response), and the plain k-means start (Eq. 4)."""
    S = synth.relu_normal((N, Cs), seed, 1)
    W = synth.normal((Ct, Cs), (2.0 / Cs) ** 0.5, seed, 2)
    T = (S.astype(np.float64) @ W.astype(np.float64).T).astype(np.float32)
    init = init_from(subvectors_fc(W, Csp), K, seed + 1)
    D0, c0 = q.pq_quantize_fc(cuda(W), Csp, K, cuda(init), 5)
    return S, T, host(D0), host(c0)


@pytest.mark.parametrize("N,Cs,Ct,Csp,K,outer,inner", [
    (256, 64, 100, 4, 16, 2, 2),
    (64, 24, 50, 3, 8, 1, 3),
    (300, 96, 257, 8, 32, 2, 1),
    (512, 1024, 300, 4, 32, 1, 2),
    (40, 16, 33, 1, 4, 2, 2),
])
def test_ec_matches_oracle(N, Cs, Ct, Csp, K, outer, inner):
    S, T, D0, c0 = calib(110 + N, N, Cs, Ct, Csp, K)
    D, codes = q.ec_quantize_fc(cuda(S), cuda(T), cuda(D0), cuda(c0), outer, inner)
    D, codes = host(D), host(codes)
    Do, co = ec.ec_quantize_fc(S, T, D0, c0, outer, inner)
    assert np.array_equal(codes, co)
    assert np.max(np.abs(D - Do.astype(np.float32))) <= 1e-6 * max(1.0, np.max(np.abs(Do)))
    e0 = ec.objective(S, T, D0, c0)
    e1 = ec.objective(S, T, D, codes)
    assert e1 <= e0 * (1 + 1e-6)


def test_ec_lowers_response_error_fc8_shape():
    """fc8-shaped layer (4096 -> 1000, C's = 4, K = 32, 512 calibration
    vectors): the error-corrected quantizer's response error on held-out
    inputs is below plain k-means' (the point of Sec. 3.3)."""
    N, Cs, Ct, Csp, K = 512, 4096, 1000, 4, 32
    S, T, D0, c0 = calib(120, N, Cs, Ct, Csp, K)
    D, codes = q.ec_quantize_fc(cuda(S), cuda(T), cuda(D0), cuda(c0), 1, 2)
    D, codes = host(D), host(codes)
    assert ec.objective(S, T, D, codes) < 0.9 * ec.objective(S, T, D0, c0)


def test_ec_rank_deficient_calibration_is_reported():
    N, Cs, Ct, Csp, K = 2, 16, 10, 4, 4     # 2 vectors cannot span 4 dimensions
    S, T, D0, c0 = calib(130, N, Cs, Ct, Csp, K)
    with pytest.raises(q.QcnnError) as e:
        q.ec_quantize_fc(cuda(S), cuda(T), cuda(D0), cuda(c0), 1, 1)
    assert e.value.status == 5  # QCNN_ERR_DATA
