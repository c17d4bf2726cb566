"""The debug build (libqcnn_debug.so, QCNN_DEBUG_CHECKS) through the C ABI.

Its kernels test what the release kernels only clamp: codes k_m >= K (Eq. 5
and Eq. 7 index K sub-codewords), table reads outside the table a kernel
built, device-memory accesses outside an array.  A kernel that finds one
records a flag and carries on with the clamped value; qcnn_device_check (and
the calls that synchronize anyway) report it as QCNN_ERR_DEVICE_CHECK.

Every algorithm is fed codes >= K (conv codes in both layouts, FC byte codes
and bit-packed FC codes); the flag must be raised and the result must equal
the one with clamped codes.  Valid inputs must raise nothing, give the
release build's result bit for bit, and leave the release build's
qcnn_device_check at 0."""
import numpy as np
import pytest
import torch

import paper_1512_06473_gb300 as q
import synth
from paper_1512_06473_gb300 import _lib
from test_gpu_parity import build_net, conv_case, cuda, host

pytestmark = pytest.mark.gpu


@pytest.fixture
def debug():
    q.set_debug(True)
    assert q.debug_checks()
    q.device_check()  # start from a clean record
    try:
        yield
    finally:
        q.device_check()
        q.set_debug(False)


def packed_conv_codes(codes, K, kh, kw):
    """The packed layout [M][kh*kw][Ct rounded up to 256] built on the host,
    codes kept as they are (qcnn_conv_pack_codes would clamp them)."""
    Ct, kk, M = codes.shape
    CtP = (Ct + 255) // 256 * 256
    p = np.zeros((M, kk, CtP), np.uint8)
    p[:, :, :Ct] = codes.transpose(2, 1, 0)
    t = torch.empty(p.size + 256, dtype=torch.uint8, device="cuda")
    off = (-t.data_ptr()) % 256
    t = t[off:off + p.size]
    t.copy_(torch.from_numpy(p.reshape(-1)))
    return t


CONV = [  # (algo, stride, pad)
    ("fused", 1, 1),
    ("phase", 2, 1),
    ("chunked", 2, 1),
    ("unfused", 1, 1),
]


@pytest.mark.parametrize("algo,stride,pad", CONV)
@pytest.mark.parametrize("layout", ["canonical", "packed"])
def test_conv_codes_out_of_range_are_flagged(debug, algo, stride, pad, layout):
    N, Cs, H, W, Ct, kh, kw, Csp, K = 2, 16, 11, 11, 40, 3, 3, 4, 100
    x, D, codes, b = conv_case(71, N, Cs, H, W, Ct, kh, kw, Csp, K)
    bad = codes.copy()
    bad[::3, ::2, :] = 200
    good = np.minimum(bad, K - 1).astype(np.uint8)

    def run(c):
        if layout == "packed":
            return host(q.conv_forward(cuda(x), cuda(D), packed_conv_codes(c, K, kh, kw), kh, kw,
                                       stride, pad, cuda(b), algo=algo, packed=True, Ct=Ct))
        return host(q.conv_forward(cuda(x), cuda(D), cuda(c), kh, kw, stride, pad, cuda(b),
                                   algo=algo))

    got = run(bad)
    flags = q.device_check()
    assert flags & _lib.CHECK_CODE, flags
    assert flags & ~_lib.CHECK_CODE == 0, flags
    ref = run(good)
    assert q.device_check() == 0
    assert np.array_equal(got, ref)


def test_fc_byte_codes_out_of_range_are_flagged(debug):
    N, Cs, Ct, Csp, K = 3, 64, 70, 4, 20
    M = Cs // Csp
    x = synth.normal((N, Cs), 1.0, 72)
    D = synth.normal((M, K, Csp), 1.0, 73)
    codes = synth.uniform_codes((M, Ct), 32, 74)  # values up to 31 >= K
    assert codes.max() >= K
    got = host(q.fc_forward(cuda(x), cuda(D), cuda(codes)))
    assert q.device_check() == _lib.CHECK_CODE
    ref = host(q.fc_forward(cuda(x), cuda(D), cuda(np.minimum(codes, K - 1).astype(np.uint8))))
    assert q.device_check() == 0
    assert np.array_equal(got, ref)


def test_fc_packed_codes_out_of_range_are_flagged(debug):
    """Rows of 5-bit codes (K = 20 needs 5 bits) holding values 20..31: the
    packer of the library clamps, so the rows are packed for K = 32 and read
    as K = 20."""
    N, Cs, Ct, Csp, K = 2, 64, 96, 4, 20
    M = Cs // Csp
    x = synth.normal((N, Cs), 1.0, 75)
    D = synth.normal((M, K, Csp), 1.0, 76)
    codes = synth.uniform_codes((M, Ct), 32, 77)
    rows = q.fc_pack_codes(cuda(codes), 32)
    assert q.device_check() == 0  # within K = 32: nothing to flag
    got = host(q.fc_forward(cuda(x), cuda(D), rows, Ct=Ct))
    assert q.device_check() == _lib.CHECK_CODE
    ref = host(q.fc_forward(cuda(x), cuda(D), cuda(np.minimum(codes, K - 1).astype(np.uint8))))
    assert np.array_equal(got, ref)


def test_synchronizing_call_reports_the_check(debug):
    """qcnn_net_forward_host synchronizes its stream, so it returns
    QCNN_ERR_DEVICE_CHECK itself when a layer read a code >= K."""
    w = synth.fc_layer()
    params = w.params()
    P = dict(params[0])
    P["codes"] = np.full_like(P["codes"], 250)
    net = build_net(w, [P], packed=True)
    N = 8
    xh = torch.from_numpy(w.input(N).reshape(N, -1, 1, 1)).pin_memory()
    yh = torch.empty((N, w.layers[0].Ct), dtype=torch.float32).pin_memory()
    ws = net.alloc_workspace(N, host_io=True)
    with pytest.raises(q.QcnnError) as e:
        net.forward_host(xh, yh, ws)
    assert e.value.status == _lib.ERR_DEVICE_CHECK
    assert q.device_check() == 0  # the call cleared the record


@pytest.mark.parametrize("name,N", [("alexnet_qcnn", 1), ("alexnet_qcnn", 16),
                                    ("vgg16_conv_stack", 1), ("alexnet_fc678", 8),
                                    ("conv3x3_64x56x56_b1", 1), ("fc_512x256_b8", 8)])
def test_valid_inputs_raise_nothing_and_match_release(name, N):
    """No false alarms on the benchmark's stacks (every planned kernel and
    tile), and the checks do not change a single bit of the result."""
    w = synth.WORKLOADS[name]
    params = w.params()
    x = w.input(N)
    xin = cuda(x if x.ndim == 4 else x.reshape(N, -1, 1, 1))
    rel_net = build_net(w, params, packed=True)
    ref = host(rel_net.forward(xin))
    assert q.device_check() == 0  # release build: always 0
    q.set_debug(True)
    try:
        q.device_check()
        dbg_net = build_net(w, params, packed=True)
        got = host(dbg_net.forward(xin))
        assert q.device_check() == 0
    finally:
        q.set_debug(False)
    assert np.array_equal(got, ref)


def test_release_build_reports_nothing():
    assert not q.debug_checks()
    N, Cs, Ct, Csp, K = 2, 32, 16, 4, 8
    M = Cs // Csp
    x = synth.normal((N, Cs), 1.0, 78)
    D = synth.normal((M, K, Csp), 1.0, 79)
    codes = np.full((M, Ct), 255, np.uint8)
    host(q.fc_forward(cuda(x), cuda(D), cuda(codes)))
    assert q.device_check() == 0
