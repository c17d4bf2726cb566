"""Bit-packed codes and the model blob on the GPU: packing bit-exact against
the oracle's packer, FC layers reading packed rows bit-identical to byte
codes, and a network loaded from a blob bit-identical to one built from
arrays (and within 1e-5 of the float64 oracle)."""
import numpy as np
import pytest
import torch

import oracle
import paper_1512_06473_gb300 as q
import synth
from oracle import bits
from test_gpu_parity import build_net, cuda, host, oracle_layers, rel

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("b,n", [(1, 1), (1, 1001), (2, 37), (3, 1000), (4, 4096), (5, 9999),
                                 (6, 17), (7, 11616), (8, 300)])
def test_pack_unpack_bits(b, n):
    c = synth.uniform_codes((n,), 1 << b, 140, b, n)
    s = host(q.pack_bits(cuda(c), b))
    assert s.tobytes() == bits.pack(c, b)
    assert np.array_equal(host(q.unpack_bits(cuda(s), n, b)), c)


@pytest.mark.parametrize("M,Ct,K", [(4, 1000, 32), (3, 4096, 32), (5, 1030, 16), (2, 513, 256),
                                    (7, 100, 2), (1, 8, 5)])
def test_fc_pack_rows(M, Ct, K):
    c = synth.uniform_codes((M, Ct), K, 141, M, Ct)
    got = host(q.fc_pack_codes(cuda(c), K)).tobytes()
    b = bits.bits_for(K)
    pitch = -(-((Ct * b + 7) // 8) // 16) * 16
    assert got == bits.pack_rows(c, b, pitch)


@pytest.mark.parametrize("N,Cs,Ct,Csp,K", [
    (1, 9216, 4096, 4, 32),      # fc6 at batch 1: the code-bound case
    (128, 4096, 1000, 4, 32),    # fc8, ragged last output tile
    (3, 96, 1030, 3, 16),
    (33, 128, 520, 4, 256),      # 8-bit codes
    (2, 64, 100, 8, 2),          # 1-bit codes
    (70, 2304, 513, 4, 5),       # 3-bit codes, splits
    (100, 6144, 1030, 6, 64),    # 6-bit codes, 16 images per lane
])
@pytest.mark.parametrize("lut", ["fp32", "bf16"])
def test_fc_packed_codes_match_byte_codes(N, Cs, Ct, Csp, K, lut):
    M = Cs // Csp
    x = synth.normal((N, Cs), 1.0, 142, N, Cs)
    D = synth.normal((M, K, Csp), 0.5, 143, M, K)
    c = synth.uniform_codes((M, Ct), K, 144, Ct)
    b = synth.normal((Ct,), 0.1, 145, Ct)
    a = host(q.fc_forward(cuda(x), cuda(D), cuda(c), cuda(b), relu=True, lut=lut))
    p = q.fc_pack_codes(cuda(c), K)
    g = host(q.fc_forward(cuda(x), cuda(D), p, cuda(b), relu=True, lut=lut, Ct=Ct))
    assert np.array_equal(a, g)
    if lut == "fp32":
        assert rel(g, oracle.fc_forward(x, D, c, b, relu=True)) <= 1e-5


def test_loaded_alexnet_matches_built_net():
    w = synth.WORKLOADS["alexnet_qcnn"]
    params = w.params()
    layers = oracle_layers(w, params)
    net = q.load_model(q.serialize_model(layers, w.in_shape))
    built = build_net(w, params, packed=True)
    x = w.input(4, 3)
    got = host(net.forward(cuda(x)))
    assert np.array_equal(got, host(built.forward(cuda(x))))
    assert rel(got[:2], oracle.net_forward(x[:2], layers)) <= 1e-5
    net.set_lut("bf16")
    gb = host(net.forward(cuda(x)))
    assert not np.array_equal(gb, got) and rel(gb, got) < 1e-2


def test_loaded_vgg_stack_and_file(tmp_path):
    w = synth.WORKLOADS["vgg16_conv_stack"]
    params = w.params()
    layers = oracle_layers(w, params)
    path = tmp_path / "vgg.qcnn"
    path.write_bytes(q.serialize_model(layers, w.in_shape))
    net = q.load_model(str(path))
    x = w.input(1, 4)
    assert rel(host(net.forward(cuda(x))), oracle.net_forward(x, layers)) <= 1e-5
