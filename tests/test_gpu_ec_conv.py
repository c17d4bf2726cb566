"""Error-corrected conv quantization (Appendix B) through the C ABI against
the float64 oracle (oracle/ec_conv.py).

Both sides work in double and take the Eq. B.8 argmin in double; only the
order of the sums over (image, position) differs, so the codes must be
identical and the codewords agree to float32 rounding."""
import numpy as np
import pytest
import torch

import oracle.ec_conv as ecc
import paper_1512_06473_gb300 as q
import synth
from test_gpu_parity import cuda, host
from test_gpu_quantize import init_from, subvectors_conv

pytestmark = pytest.mark.gpu


def calib(seed, N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K):
    """Calibration maps S (post-ReLU), T = the dense layer's response (no
    bias), and the plain k-means start (Eq. 6)."""
    S = synth.relu_normal((N, Cs, H, W), seed, 1)
    Wd = synth.normal((Ct, Cs, kh, kw), (2.0 / (Cs * kh * kw)) ** 0.5, seed, 2)
    T = torch.nn.functional.conv2d(torch.from_numpy(S).double(), torch.from_numpy(Wd).double(),
                                   stride=stride, padding=pad).float().numpy()
    init = init_from(subvectors_conv(Wd, Csp), K, seed + 1)
    D0, c0 = q.pq_quantize_conv(cuda(Wd), Csp, K, cuda(init), 4)
    return S, T, host(D0), host(c0)


@pytest.mark.parametrize("N,Cs,H,W,Ct,kh,kw,s,p,Csp,K,outer,inner", [
    (2, 8, 9, 9, 12, 3, 3, 1, 1, 4, 16, 1, 1),
    (3, 6, 7, 8, 10, 3, 3, 2, 1, 3, 8, 2, 1),     # stride 2, Csp = 3
    (2, 8, 6, 6, 9, 2, 3, 1, 0, 8, 5, 1, 2),      # non-square kernel, one sub-space
    (4, 32, 13, 13, 64, 3, 3, 1, 1, 4, 32, 1, 1),  # AlexNet conv3 map, smaller widths
    (2, 4, 5, 5, 7, 1, 1, 1, 0, 2, 1, 2, 2),      # 1x1 kernel, K = 1
])
def test_ec_conv_matches_oracle(N, Cs, H, W, Ct, kh, kw, s, p, Csp, K, outer, inner):
    S, T, D0, c0 = calib(200 + N * H + Ct, N, Cs, H, W, Ct, kh, kw, s, p, Csp, K)
    D, codes = q.ec_quantize_conv(cuda(S), cuda(T), cuda(D0), cuda(c0), kh, kw, s, p, outer, inner)
    D, codes = host(D), host(codes)
    Do, co = ecc.ec_quantize_conv(S, T, D0, c0, kh, kw, s, p, outer, inner)
    assert np.array_equal(codes, co)
    assert np.max(np.abs(D - Do.astype(np.float32))) <= 1e-6 * max(1.0, np.max(np.abs(Do)))
    e0 = ecc.objective(S, T, D0, c0, kh, kw, s, p)
    assert ecc.objective(S, T, D, codes, kh, kw, s, p) <= e0 * (1 + 1e-6)


def test_ec_conv_lowers_response_error():
    """The point of Sec. 3.3: error correction fits the layer's response
    better than the plain k-means quantization it starts from."""
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = 8, 32, 13, 13, 64, 3, 3, 1, 1, 4, 16
    S, T, D0, c0 = calib(230, N, Cs, H, W, Ct, kh, kw, s, p, Csp, K)
    D, codes = q.ec_quantize_conv(cuda(S), cuda(T), cuda(D0), cuda(c0), kh, kw, s, p, 1, 2)
    e0 = ecc.objective(S, T, D0, c0, kh, kw, s, p)
    assert ecc.objective(S, T, host(D), host(codes), kh, kw, s, p) < 0.9 * e0


def test_ec_conv_rank_deficient_is_reported():
    """One image of a 1x1 map: a single calibration vector cannot determine
    a 4-dimensional codeword."""
    S, T, D0, c0 = calib(240, 1, 8, 1, 1, 5, 1, 1, 1, 0, 4, 3)
    with pytest.raises(q.QcnnError) as e:
        q.ec_quantize_conv(cuda(S), cuda(T), cuda(D0), cuda(c0), 1, 1, 1, 0, 1, 1)
    assert e.value.status == 5  # QCNN_ERR_DATA
