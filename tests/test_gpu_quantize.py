"""The k-means quantizer (Eq. 4 / Eq. 6) through the C ABI against the oracle.

Both sides take the assignment decision in binary32 with the same operation
order and sum the centroids in double in point order, so centroids, codes and
assignments must be bit-identical, at every size."""
import numpy as np
import pytest
import torch

import oracle
import paper_1512_06473_gb300 as q
import synth
from test_gpu_parity import cuda, host

pytestmark = pytest.mark.gpu


def subvectors_fc(W, Csp):
    """[Ct, Cs] -> points [M, Ct, Csp] (sub-vector m of each weight vector)."""
    Ct, Cs = W.shape
    return W.reshape(Ct, Cs // Csp, Csp).transpose(1, 0, 2).copy()


def subvectors_conv(W, Csp):
    """[Ct, Cs, kh, kw] -> points [M, Ct*kh*kw, Csp], point p = ct*kh*kw + pk."""
    Ct, Cs, kh, kw = W.shape
    M = Cs // Csp
    return W.reshape(Ct, M, Csp, kh * kw).transpose(1, 0, 3, 2).reshape(M, Ct * kh * kw, Csp).copy()


def init_from(points, K, seed):
    M, P, _ = points.shape
    return np.stack([points[m][synth.sample_indices(P, K, seed, m)] for m in range(M)])


@pytest.mark.parametrize("M,P,Csp,K,iters", [
    (5, 700, 4, 16, 5),
    (3, 1000, 3, 128, 3),
    (2, 513, 8, 256, 2),
    (4, 300, 1, 7, 4),
    (2, 100, 2, 1, 3),       # K = 1: the mean of everything
    (2, 40, 4, 64, 2),       # K > P: repeated initial points, empty clusters
    (1, 1, 4, 3, 1),         # a single point
    (6, 2000, 4, 32, 0),     # iters = 0: assignment to the initial centroids
])
def test_kmeans_bit_exact(M, P, Csp, K, iters):
    pts = synth.normal((M, P, Csp), 1.0, 90, M, P, Csp, K)
    init = init_from(pts, K, 91)
    D, a = q.kmeans(cuda(pts), cuda(init), iters)
    D, a = host(D), host(a)
    for m in range(M):
        cen, am = oracle.kmeans(pts[m], init[m], iters)
        assert np.array_equal(D[m], cen), m
        assert np.array_equal(a[m], am), m


@pytest.mark.parametrize("Ct,Cs,kh,kw,Csp,K,iters", [
    (64, 48, 3, 3, 4, 32, 4),
    (40, 30, 5, 5, 3, 16, 3),
    (16, 16, 1, 1, 8, 8, 2),
    (384, 256, 3, 3, 4, 128, 3),    # AlexNet conv3, full size
])
def test_pq_quantize_conv_bit_exact(Ct, Cs, kh, kw, Csp, K, iters):
    W = synth.normal((Ct, Cs, kh, kw), 0.05, 92, Ct, Cs, kh)
    init = init_from(subvectors_conv(W, Csp), K, 93)
    D, codes = q.pq_quantize_conv(cuda(W), Csp, K, cuda(init), iters)
    Do, co = oracle.pq_quantize_conv(W, Csp, K, init, iters)
    assert np.array_equal(host(D), Do)
    assert np.array_equal(host(codes), co)


@pytest.mark.parametrize("Ct,Cs,Csp,K,iters", [
    (100, 64, 4, 16, 5),
    (1000, 4096, 4, 32, 2),         # AlexNet fc8, full size
    (33, 12, 3, 256, 3),
])
def test_pq_quantize_fc_bit_exact(Ct, Cs, Csp, K, iters):
    W = synth.normal((Ct, Cs), 0.02, 94, Ct, Cs)
    init = init_from(subvectors_fc(W, Csp), K, 95)
    D, codes = q.pq_quantize_fc(cuda(W), Csp, K, cuda(init), iters)
    Do, co = oracle.pq_quantize_fc(W, Csp, K, init, iters)
    assert np.array_equal(host(D), Do)
    assert np.array_equal(host(codes), co)


def test_quantize_is_deterministic():
    W = synth.normal((256, 96, 5, 5), 0.05, 96)
    init = init_from(subvectors_conv(W, 4), 128, 97)
    a = [tuple(host(t) for t in q.pq_quantize_conv(cuda(W), 4, 128, cuda(init), 3)) for _ in range(2)]
    assert np.array_equal(a[0][0], a[1][0]) and np.array_equal(a[0][1], a[1][1])


def test_exact_recovery_at_full_size_and_forward():
    """AlexNet conv2 weights (256 x 96 x 5 x 5) built from K = 128 prototypes
    per sub-space: started from the prototypes, the GPU quantizer returns
    them and the codes, so the quantized layer's response equals the dense
    conv of W (Eq. 3 with equality) -- checked on the GPU forward against
    torch's float64 conv2d."""
    Ct, Cs, kh, kw, Csp, K = 256, 96, 5, 5, 4, 128
    M = Cs // Csp
    D0 = synth.normal((M, K, Csp), 0.05, 98)
    c0 = synth.uniform_codes((Ct, kh * kw, M), K, 99)
    sel = D0[np.arange(M)[None, None, :], c0.astype(np.int64)]          # [Ct, kk, M, Csp]
    W = sel.reshape(Ct, kh, kw, M * Csp).transpose(0, 3, 1, 2).copy()   # Eq. 6 meaning of codes
    D, codes = q.pq_quantize_conv(cuda(W), Csp, K, cuda(D0), 2)
    used = np.zeros((M, K), bool)
    used[np.arange(M)[None, None, :], c0.astype(np.int64)] = True
    assert np.array_equal(host(codes), c0)
    assert np.array_equal(host(D)[used], D0[used])
    x = synth.relu_normal((2, Cs, 27, 27), 100)
    got = host(q.conv_forward(cuda(x), D, codes, kh, kw, 1, 2))
    ref = torch.nn.functional.conv2d(torch.from_numpy(x).double(), torch.from_numpy(W).double(),
                                     padding=2).numpy()
    assert np.max(np.abs(got - ref)) <= 1e-5 * np.max(np.abs(ref))


def test_quantize_rejects_bad_arguments():
    W = cuda(synth.normal((8, 12), 1.0, 1))
    init = cuda(synth.normal((3, 4, 4), 1.0, 2))
    with pytest.raises(q.QcnnError):
        q.pq_quantize_fc(W, 5, 4, cuda(synth.normal((2, 4, 5), 1.0, 3)), 1)  # Cs % Csp
    with pytest.raises(ValueError):
        q.pq_quantize_fc(W, 4, 5, init, 1)  # init shape
