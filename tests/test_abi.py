"""The C ABI of include/qcnn.h: the library builds, loads and exports every
declared function, and its host-side argument checks and workspace planning
work without a GPU (no kernel is launched by these tests)."""
import ctypes

import pytest

from paper_1512_06473_gb300 import _lib
import synth

lib = _lib.load()


def test_every_declared_symbol_is_exported():
    names = _lib.header_functions()
    assert len(names) >= 15
    missing = [n for n in names if not hasattr(lib, n)]
    assert missing == []
    # and the binding knows the signature of each
    assert sorted(_lib._SIGS) == names


def test_status_strings():
    for s in range(7):
        assert lib.qcnn_status_string(s) != b"unknown status"
    assert lib.qcnn_status_string(99) == b"unknown status"


def test_debug_library_exports_every_symbol():
    """libqcnn_debug.so (the device-checking build) has the same ABI; only
    qcnn_debug_checks tells the two apart."""
    from paper_1512_06473_gb300 import build as _build
    dbg = _lib.load(_build.build_debug())
    names = _lib.header_functions()
    assert [n for n in names if not hasattr(dbg, n)] == []
    assert dbg.qcnn_debug_checks() == 1
    assert lib.qcnn_debug_checks() == 0


N0 = None  # null device pointer


@pytest.mark.parametrize("args", [
    (8, 10, 4, 3, 16),     # Cs not a multiple of Csp
    (8, 12, 4, 3, 0),      # K = 0
    (8, 12, 4, 3, 257),    # K > 256
    (8, 18, 4, 9, 16),     # Csp > 8
    (0, 12, 4, 3, 16),     # N = 0
    (8, 12, 0, 3, 16),     # Ct = 0
])
def test_fc_rejects_bad_sizes(args):
    N, Cs, Ct, Csp, K = args
    nb = ctypes.c_size_t()
    assert lib.qcnn_fc_workspace_size(N, Cs, Ct, Csp, K, 0, ctypes.byref(nb)) \
        == _lib.ERR_INVALID_ARG
    assert lib.qcnn_fc_forward(8, N, Cs, Ct, 8, Csp, K, 8, None, 8, 0, 0, None, 0, None) \
        == _lib.ERR_INVALID_ARG


def test_fc_rejects_null_pointers():
    assert lib.qcnn_fc_forward(None, 2, 8, 4, 8, 4, 16, 8, None, 8, 0, 0, None, 0, None) \
        == _lib.ERR_INVALID_ARG
    assert lib.qcnn_fc_forward(8, 2, 8, 4, None, 4, 16, 8, None, 8, 0, 0, None, 0, None) \
        == _lib.ERR_INVALID_ARG
    assert lib.qcnn_fc_forward(8, 2, 8, 4, 8, 4, 16, None, None, 8, 0, 0, None, 0, None) \
        == _lib.ERR_INVALID_ARG
    assert lib.qcnn_fc_forward(8, 2, 8, 4, 8, 4, 16, 8, None, None, 0, 0, None, 0, None) \
        == _lib.ERR_INVALID_ARG


@pytest.mark.parametrize("args", [
    (1, 8, 5, 5, 4, 7, 7, 1, 0, 4, 16),   # kernel larger than the padded map
    (1, 8, 5, 5, 4, 3, 3, 0, 1, 4, 16),   # stride 0
    (1, 8, 5, 5, 4, 3, 3, 1, -1, 4, 16),  # negative pad
    (1, 9, 5, 5, 4, 3, 3, 1, 1, 4, 16),   # Cs % Csp
    (1, 8, 5, 5, 4, 3, 3, 1, 1, 4, 300),  # K
])
def test_conv_rejects_bad_sizes(args):
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = args
    nb = ctypes.c_size_t()
    assert lib.qcnn_conv_workspace_size(N, Cs, H, W, Ct, kh, kw, s, p, Csp, K, 0, 0, 0,
                                        ctypes.byref(nb)) == _lib.ERR_INVALID_ARG
    assert lib.qcnn_conv_forward(8, N, Cs, H, W, Ct, kh, kw, s, p, 8, Csp, K, 8, 0, None, 8, 0, 0,
                                 0, None, 0, None) == _lib.ERR_INVALID_ARG


def test_conv_bad_enums_and_fused_stride():
    nb = ctypes.c_size_t()
    assert lib.qcnn_conv_workspace_size(1, 8, 9, 9, 4, 3, 3, 1, 1, 4, 16, 7, 0, 0,
                                        ctypes.byref(nb)) == _lib.ERR_INVALID_ARG
    assert lib.qcnn_conv_workspace_size(1, 8, 9, 9, 4, 3, 3, 1, 1, 4, 16, 0, 9, 0,
                                        ctypes.byref(nb)) == _lib.ERR_INVALID_ARG
    # lut type outside the enum
    assert lib.qcnn_conv_workspace_size(1, 8, 9, 9, 4, 3, 3, 1, 1, 4, 16, 0, 0, 2,
                                        ctypes.byref(nb)) == _lib.ERR_INVALID_ARG
    assert lib.qcnn_fc_workspace_size(2, 8, 4, 4, 16, -1, ctypes.byref(nb)) \
        == _lib.ERR_INVALID_ARG
    # the fused kernel serves stride 1 only
    assert lib.qcnn_conv_workspace_size(1, 8, 9, 9, 4, 3, 3, 2, 1, 4, 16, 0, 1, 0,
                                        ctypes.byref(nb)) == _lib.ERR_UNSUPPORTED
    assert lib.qcnn_conv_workspace_size(1, 8, 9, 9, 4, 3, 3, 2, 1, 4, 16, 0, 0, 0,
                                        ctypes.byref(nb)) == _lib.OK
    # bf16 tables: fused and chunked serve them, the unfused path does not
    for algo in (0, 1, 3):
        assert lib.qcnn_conv_workspace_size(1, 8, 9, 9, 4, 3, 3, 1, 1, 4, 16, 0, algo, 1,
                                            ctypes.byref(nb)) == _lib.OK, algo
    assert lib.qcnn_conv_workspace_size(1, 8, 9, 9, 4, 3, 3, 2, 1, 4, 16, 0, 0, 1,
                                        ctypes.byref(nb)) == _lib.OK
    assert lib.qcnn_conv_workspace_size(1, 8, 9, 9, 4, 3, 3, 1, 1, 4, 16, 0, 2, 1,
                                        ctypes.byref(nb)) == _lib.ERR_UNSUPPORTED


def test_conv_workspace_too_small_is_reported_before_launch():
    nb = ctypes.c_size_t()
    assert lib.qcnn_conv_workspace_size(1, 8, 9, 9, 4, 3, 3, 1, 1, 4, 16, 0, 0, 0,
                                        ctypes.byref(nb)) == _lib.OK
    assert nb.value > 0  # canonical codes are re-laid out in the workspace
    assert lib.qcnn_conv_forward(8, 1, 8, 9, 9, 4, 3, 3, 1, 1, 8, 4, 16, 8, 0, None, 8, 0, 0,
                                 0, None, 0, None) == _lib.ERR_WORKSPACE
    # misaligned workspace
    assert lib.qcnn_conv_forward(8, 1, 8, 9, 9, 4, 3, 3, 1, 1, 8, 4, 16, 8, 0, None, 8, 0, 0,
                                 0, 4096 + 8, nb.value, None) == _lib.ERR_WORKSPACE


def _layers(workload, N=1):
    arr = (_lib.Layer * len(workload.layers))()
    for i, L in enumerate(workload.layers):
        d = arr[i]
        if isinstance(L, synth.Conv):
            d.kind, d.Ct, d.kh, d.kw, d.stride, d.pad = 0, L.Ct, L.kh, L.kw, L.stride, L.pad
            d.Csp, d.K, d.relu = L.Csp, L.K, int(L.relu)
            d.D, d.codes = 8, 8
        elif isinstance(L, synth.FC):
            d.kind, d.Ct, d.Csp, d.K, d.relu = 1, L.Ct, L.Csp, L.K, int(L.relu)
            d.D, d.codes = 8, 8
        else:
            d.kind, d.kh, d.kw, d.stride = 2, L.k, L.k, L.s
    return arr


@pytest.mark.parametrize("name", sorted(synth.WORKLOADS))
def test_net_shapes_and_workspace(name):
    w = synth.WORKLOADS[name]
    if len(w.in_shape) == 1:
        C, H, W = w.in_shape[0], 1, 1
    else:
        C, H, W = w.in_shape
    arr = _layers(w)
    oc, oh, ow = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    assert lib.qcnn_net_output_shape(arr, len(arr), C, H, W, ctypes.byref(oc), ctypes.byref(oh),
                                     ctypes.byref(ow)) == _lib.OK
    last = w.shapes()[-1][1]
    assert (oc.value, oh.value, ow.value) == tuple(last) + (1,) * (3 - len(last))
    for N in w.batches:
        a, b = ctypes.c_size_t(), ctypes.c_size_t()
        assert lib.qcnn_net_workspace_size(arr, len(arr), N, C, H, W, 0, ctypes.byref(a)) == 0
        assert lib.qcnn_net_workspace_size(arr, len(arr), N, C, H, W, 1, ctypes.byref(b)) == 0
        assert b.value >= a.value + N * C * H * W * 4


def test_alexnet_output_is_1000_logits():
    w = synth.alexnet()
    arr = _layers(w)
    oc, oh, ow = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    assert lib.qcnn_net_output_shape(arr, len(arr), 3, 227, 227, ctypes.byref(oc),
                                     ctypes.byref(oh), ctypes.byref(ow)) == 0
    assert (oc.value, oh.value, ow.value) == (1000, 1, 1)


def test_net_rejects_mismatched_layer():
    w = synth.alexnet()
    arr = _layers(w)
    arr[2].Csp = 5  # conv2 has 96 inputs: 96 % 5 != 0
    nb = ctypes.c_size_t()
    assert lib.qcnn_net_workspace_size(arr, len(arr), 1, 3, 227, 227, 0, ctypes.byref(nb)) \
        == _lib.ERR_INVALID_ARG
    assert lib.qcnn_net_workspace_size(None, 3, 1, 3, 227, 227, 0, ctypes.byref(nb)) \
        == _lib.ERR_INVALID_ARG


def test_net_plan_cache_keys_on_every_planning_input():
    """Net plans are cached; a change of batch, host I/O, a layer option or a
    NULL pointer must not be answered from the cache."""
    w = synth.alexnet()
    arr = _layers(w)
    sizes = {}
    for N in (1, 2, 128):
        for host_io in (0, 1):
            nb = ctypes.c_size_t()
            for _ in range(2):  # the second call is served from the cache
                assert lib.qcnn_net_workspace_size(arr, len(arr), N, 3, 227, 227, host_io,
                                                   ctypes.byref(nb)) == 0
                sizes.setdefault((N, host_io), nb.value)
                assert sizes[(N, host_io)] == nb.value
    assert len(set(sizes.values())) == len(sizes)
    a, b = ctypes.c_size_t(), ctypes.c_size_t()
    assert lib.qcnn_net_workspace_size(arr, len(arr), 1, 3, 227, 227, 0, ctypes.byref(a)) == 0
    arr[0].algo = 2  # conv1 through the unfused path: its tables live in the workspace
    assert lib.qcnn_net_workspace_size(arr, len(arr), 1, 3, 227, 227, 0, ctypes.byref(b)) == 0
    assert b.value > a.value
    arr[0].algo = 0
    arr[4].D = None
    assert lib.qcnn_net_workspace_size(arr, len(arr), 1, 3, 227, 227, 0, ctypes.byref(b)) \
        == _lib.ERR_INVALID_ARG


def test_quantizer_argument_checks():
    nb = ctypes.c_size_t()
    FC, CONV = _lib.LAYER_FC, _lib.LAYER_CONV
    assert lib.qcnn_pq_quantize_workspace_size(FC, 10, 12, 0, 0, 4, 16, ctypes.byref(nb)) == _lib.OK
    assert nb.value > 0
    assert lib.qcnn_pq_quantize_workspace_size(CONV, 10, 12, 3, 3, 4, 16, ctypes.byref(nb)) == _lib.OK
    for bad in [(FC, 10, 12, 0, 0, 5, 16), (FC, 10, 12, 0, 0, 4, 0), (FC, 10, 12, 0, 0, 4, 257),
                (CONV, 10, 12, 0, 3, 4, 16), (7, 10, 12, 1, 1, 4, 16), (FC, 0, 12, 1, 1, 4, 16),
                (FC, 10, 18, 1, 1, 9, 16)]:
        assert lib.qcnn_pq_quantize_workspace_size(*bad, ctypes.byref(nb)) == _lib.ERR_INVALID_ARG, bad
    assert lib.qcnn_kmeans_workspace_size(4, 100, 4, 16, ctypes.byref(nb)) == _lib.OK
    assert lib.qcnn_kmeans(None, 4, 100, 4, 16, 8, 2, 8, 8, 8, nb.value, None) == _lib.ERR_INVALID_ARG
    assert lib.qcnn_kmeans(8, 4, 100, 4, 16, 8, -1, 8, 8, 8, nb.value, None) == _lib.ERR_INVALID_ARG
    assert lib.qcnn_kmeans(8, 4, 100, 4, 16, 8, 2, 8, 8, None, 0, None) == _lib.ERR_WORKSPACE
    assert lib.qcnn_pq_quantize(FC, 8, 10, 12, 1, 1, 4, 16, 8, 2, 8, 8, 4096 + 8, 1 << 20,
                                None) == _lib.ERR_WORKSPACE  # misaligned workspace


def test_fused_variant_table():
    n = lib.qcnn_conv_fused_variant_count()
    assert n >= 10
    info = (ctypes.c_int * 10)()
    seen_sk = seen_pipe = seen_bf = seen_tc = False
    for v in range(n):
        assert lib.qcnn_conv_fused_variant_info(v, info) == 0
        P, CTW, WP, CSP4, NW, MINB, PIPE, BF, SK, TC = list(info)
        if TC:  # tensor-core build: fp32 tables, 8-wide sub-vectors, one buffer, 1 CTA per SM
            assert CSP4 == 8 and not (PIPE or BF) and MINB == 1
            seen_tc = True
        assert P >= 1 and (CTW in (4, 8) or CTW % 16 == 0)
        assert CSP4 in (4, 8) and NW in (8, 12, 16, 32) and MINB in (1, 2)
        assert (NW // WP) * CTW % 16 == 0
        seen_sk |= bool(SK)
        seen_pipe |= bool(PIPE)
        assert not (SK and PIPE)  # stream-K runs one table buffer
        seen_bf |= bool(BF)
    assert seen_sk and seen_pipe and seen_bf and seen_tc
    assert lib.qcnn_conv_fused_variant_info(n, info) == _lib.ERR_INVALID_ARG
    assert lib.qcnn_conv_fused_variant_info(-1, info) == _lib.ERR_INVALID_ARG
    assert lib.qcnn_conv_fused_variant_info(0, None) == _lib.ERR_INVALID_ARG


def test_forced_fused_variant_planning():
    """Every variant either plans the shape or reports it unsupported; an
    index past the table is an argument error; strided convs never fuse."""
    n = lib.qcnn_conv_fused_variant_count()
    nb = ctypes.c_size_t()
    shape = (64, 64, 13, 13, 384, 3, 3, 1, 1, 4, 128)
    ok = 0
    for v in range(n):
        rc = lib.qcnn_conv_workspace_size(*shape, 0, _lib.ALGO_FUSED_VARIANT + v, 0,
                                          ctypes.byref(nb))
        assert rc in (0, _lib.ERR_UNSUPPORTED)
        ok += rc == 0
    assert ok >= 5
    assert lib.qcnn_conv_workspace_size(*shape, 0, _lib.ALGO_FUSED_VARIANT + n, 0,
                                        ctypes.byref(nb)) == _lib.ERR_INVALID_ARG
    strided = (1, 8, 15, 15, 4, 3, 3, 2, 1, 4, 16)
    assert lib.qcnn_conv_workspace_size(*strided, 0, _lib.ALGO_FUSED_VARIANT, 0,
                                        ctypes.byref(nb)) == _lib.ERR_UNSUPPORTED


# The calls below pass made-up device addresses; each one must be refused by
# the host-side checks.  On a machine with a GPU a missing check would launch
# a kernel on them, so the test only runs where no device is visible.
_no_device = pytest.mark.skipif(__import__("torch").cuda.is_available(),
                                reason="passes made-up device addresses")


@_no_device
def test_misaligned_pointers_are_refused_before_launch():
    A16, A4, ODD = 4096, 4100, 4098  # 16-byte aligned, 4-byte aligned, 2-byte aligned
    INV = _lib.ERR_INVALID_ARG
    PACKED = 1
    # conv: fp32 arrays need 4-byte alignment, PACKED codes 16-byte alignment
    conv = lambda x, D, codes, y, bias, layout: lib.qcnn_conv_forward(
        x, 2, 8, 9, 9, 4, 3, 3, 1, 1, D, 4, 16, codes, layout, bias, y, 0, 0, 0, None, 0, None)
    assert conv(A16, A16, A4, A16, None, PACKED) == INV
    assert conv(ODD, A16, A16, A16, None, PACKED) == INV
    assert conv(A16, ODD, A16, A16, None, PACKED) == INV
    assert conv(A16, A16, A16, ODD, None, PACKED) == INV
    assert conv(A16, A16, A16, A16, ODD, PACKED) == INV
    # FC
    fc = lambda x, D, codes, y, bias: lib.qcnn_fc_forward(x, 2, 12, 4, D, 3, 16, codes, bias, y,
                                                           0, 0, None, 0, None)
    assert fc(ODD, A16, A16, A16, None) == INV
    assert fc(A16, A16, A16, A16, ODD) == INV
    assert lib.qcnn_fc_forward_packed(A16, 2, 12, 4, A16, 3, 16, A4, None, A16, 0, 0, None, 0,
                                      None) == INV
    # table build: fp32 entries 4-byte, bfloat16 entries 2-byte aligned
    assert lib.qcnn_lut_build(A16, 1, 12, 1, 1, A16, 3, 16, ODD, 0, None) == INV
    assert lib.qcnn_lut_build(A16, 1, 12, 1, 1, A16, 3, 16, A16 + 1, 1, None) == INV
    assert lib.qcnn_maxpool(ODD, 1, 4, 8, 8, 2, 2, A16, None) == INV
    # a stack: the layers' D / bias and PACKED codes, and the net's x / y
    w = synth.alexnet()
    arr = _layers(w)
    for L in arr:
        if L.kind != 2:
            L.D, L.codes, L.codes_layout = A16, A16, PACKED
    nb = ctypes.c_size_t()
    assert lib.qcnn_net_workspace_size(arr, len(arr), 1, 3, 227, 227, 0, ctypes.byref(nb)) == 0
    assert lib.qcnn_net_forward(arr, len(arr), ODD, 1, 3, 227, 227, A16, None, 0, None) == INV
    arr[2].codes = A4  # conv2's PACKED codes
    assert lib.qcnn_net_forward(arr, len(arr), A16, 1, 3, 227, 227, A16, None, 0, None) == INV
    arr[2].codes = A16
    arr[len(arr) - 1].bias = ODD  # fc8's bias
    host = (ctypes.c_float * 4)()
    assert lib.qcnn_net_forward_host(arr, len(arr), ctypes.addressof(host), 1, 3, 227, 227,
                                     ctypes.addressof(host), None, 0, None) == INV


# ---- the planners' choices (host only) ------------------------------------
# The plans the measured launch list of the AlexNet-shaped benchmark shows
# (batch 128) and the batch-1 split plans, pinned so that a planner change
# that moves a layer off its measured-best kernel fails here, without a GPU.
# Without a device the planners assume GB300's 152 SMs and 227 KB of shared
# memory per block; another GPU would plan differently.
def _gb300_or_no_device():
    torch = __import__("torch")
    return (not torch.cuda.is_available()
            or torch.cuda.get_device_properties(0).multi_processor_count == 152)


_planner = pytest.mark.skipif(not _gb300_or_no_device(), reason="plans are for 152 SMs")
ALEX_CONV = {"conv1": (3, 227, 227, 96, 11, 11, 4, 0, 3), "conv2": (96, 27, 27, 256, 5, 5, 1, 2, 4),
             "conv3": (256, 13, 13, 384, 3, 3, 1, 1, 4), "conv4": (384, 13, 13, 384, 3, 3, 1, 1, 4),
             "conv5": (384, 13, 13, 256, 3, 3, 1, 1, 4)}
ALEX_FC = {"fc6": (9216, 4096), "fc7": (4096, 4096), "fc8": (4096, 1000)}


@_planner
def test_alexnet_batch128_plans():
    import paper_1512_06473_gb300 as q
    V = q.fused_variants()
    p = q.conv_plan(128, *ALEX_CONV["conv1"], K=128)
    assert (p["algo"], p["positions"], p["channels"], p["splits"]) == ("phase", 224, 96, 1)
    assert p["ctas"] == 14 * 128  # 14 tiles of 224 positions of the pitch-57 phase grid
    want = {"conv2": (5, 16, 16), "conv3": (6, 16, 12), "conv4": (6, 16, 12), "conv5": (6, 8, 16)}
    for name, (P, CTW, NW) in want.items():
        p = q.conv_plan(128, *ALEX_CONV[name], K=128)
        v = V[p["variant"]]
        assert p["algo"] == "fused" and p["stream_k"] == 1 and p["ctas"] == 152, name
        assert (v["P"], v["CTW"], v["NW"], v["SK"], v["BF"]) == (P, CTW, NW, 1, 0), name
        assert p["channels"] == CTW * NW and p["positions"] == 32 * P
    for name, (Cs, Ct) in ALEX_FC.items():
        f = q.fc_plan(128, Cs, Ct)
        assert (f["images"], f["outputs"]) == (16, 1024), name
        assert f["splits"] > 1 and f["ctas"] == f["splits"] * 8 * -(-Ct // 1024)


@_planner
def test_batch1_plans_split_the_subspaces():
    import paper_1512_06473_gb300 as q
    for name, shape in ALEX_CONV.items():
        p = q.conv_plan(1, *shape, K=128)
        assert p["algo"] == ("phase" if name == "conv1" else "fused"), name
        assert p["splits"] > 1 and p["stream_k"] == 0 and p["ctas"] >= 64, (name, p)
    for name, (Cs, Ct) in ALEX_FC.items():
        f = q.fc_plan(1, Cs, Ct)
        # one image per CTA, the sub-spaces over >= 64 CTAs; with several
        # output tiles (fc6, fc7) clusters of 8 add their partial sums in
        # distributed shared memory first
        assert f["images"] == 1 and f["splits"] >= 64, (name, f)
        assert f["cluster"] == (8 if Ct > 1024 else 1), (name, f)


@_planner
@pytest.mark.parametrize("lut", ["fp32", "bf16"])
def test_plans_are_consistent_on_every_workload(lut):
    """Every layer of every workload at batches 1-256: a fused conv plan's CTAs
    are its images x splits x position tiles x channel tiles (under stream-K
    at most one per (tile, sub-space) unit), clusters divide the splits, tiles
    are whole warps of positions and 16-channel code pieces; an FC plan's
    CTAs are its splits x image tiles x output tiles."""
    import paper_1512_06473_gb300 as q
    for name, w in synth.WORKLOADS.items():
        for N in (1, 2, 3, 4, 8, 16, 32, 64, 128, 256):
            for i, (L, (sin, sout)) in enumerate(zip(w.layers, w.shapes())):
                where = (name, N, i)
                if isinstance(L, synth.Conv):
                    p = q.conv_plan(N, L.Cs, sin[1], sin[2], L.Ct, L.kh, L.kw, L.stride, L.pad,
                                    L.Csp, L.K, lut=lut)
                    assert p["splits"] >= 1 and p["splits"] % p["cluster"] == 0, where
                    assert p["cluster"] in (1, 2, 4, 8, 16), where
                    if p["algo"] != "fused":
                        continue
                    Ho, Wo = sout[1], sout[2]
                    pitch = max(sin[2] + L.pad, Wo)
                    pos_tiles = -(-((Ho - 1) * pitch + Wo) // p["positions"])
                    ct_tiles = -(-L.Ct // p["channels"])
                    assert p["positions"] % 32 == 0 and p["channels"] % 16 == 0, where
                    if p["stream_k"]:
                        assert p["splits"] == 1 and p["cluster"] == 1, where
                        assert p["ctas"] <= N * pos_tiles * ct_tiles * L.M, where
                    else:
                        assert p["ctas"] == N * p["splits"] * pos_tiles * ct_tiles, where
                elif isinstance(L, synth.FC):
                    f = q.fc_plan(N, L.Cs, L.Ct, L.Csp, L.K, lut=lut)
                    assert f["splits"] % f["cluster"] == 0, where
                    assert f["ctas"] == f["splits"] * -(-N // f["images"]) * \
                        -(-L.Ct // f["outputs"]), where


@_planner
def test_net_partial_sum_handoffs():
    """qcnn_net_plan_info: a conv layer whose plan leaves split partial sums
    hands them to a max-pool after it, an FC layer to an FC layer after it at
    batch <= 8; every other layer reduces in its own launch.  In AlexNet at
    batch 1 that is conv2 -> pool2, conv5 -> pool5 and fc6 -> fc7 -> fc8; at
    batch 128 (stream-K conv plans, FC above batch 8) nothing."""
    import paper_1512_06473_gb300 as q
    w = synth.alexnet()
    arr = _layers(w)
    shapes = w.shapes()

    def info(N, host_io=0):
        out = (ctypes.c_int * (2 * len(arr)))()
        assert lib.qcnn_net_plan_info(arr, len(arr), N, 3, 227, 227, host_io, out) == _lib.OK
        return [(out[2 * i], out[2 * i + 1]) for i in range(len(arr))]

    for N, host_io in ((1, 0), (1, 1), (2, 0), (8, 0), (128, 0), (128, 1)):
        f = info(N, host_io)
        assert f[0][1] == 0 and f[-1][0] == 0
        for i, L in enumerate(w.layers[:-1]):
            assert f[i][0] == f[i + 1][1], (N, i)  # seen from both sides
            nxt = w.layers[i + 1]
            if isinstance(L, synth.Conv):
                sin = shapes[i][0]
                p = q.conv_plan(N, L.Cs, sin[1], sin[2], L.Ct, L.kh, L.kw, L.stride, L.pad,
                                L.Csp, L.K)
                groups = 1 if p["stream_k"] else p["splits"] // p["cluster"]
                want = isinstance(nxt, synth.Pool) and groups > 1
            elif isinstance(L, synth.FC):
                fp = q.fc_plan(N, L.Cs, L.Ct, L.Csp, L.K)
                want = isinstance(nxt, synth.FC) and N <= 8 and fp["splits"] // fp["cluster"] > 1
            else:
                want = False
            assert bool(f[i][0]) == want, (N, host_io, i)
    assert [i for i, (leaves, _) in enumerate(info(1)) if leaves] == [2, 6, 8, 9]
    assert not any(a or b for a, b in info(128))
    assert lib.qcnn_net_plan_info(arr, len(arr), 1, 3, 227, 227, 0, None) == _lib.ERR_INVALID_ARG


@_planner
def test_fc_16_image_tiles_take_two_chunks():
    """16-image FC tiles give every CTA at least two chunks of 16 sub-spaces
    (one chunk per CTA measured slower at batches 64-128)."""
    import paper_1512_06473_gb300 as q
    seen = 0
    for N in (64, 128, 256):
        for Cs, Ct in ALEX_FC.values():
            f = q.fc_plan(N, Cs, Ct)
            if f["images"] == 16:
                seen += 1
                n_chunks = -(-(Cs // 4) // f["chunk"])
                assert f["splits"] <= n_chunks // 2, (N, Cs, Ct, f)
    assert seen >= 6


@_planner
def test_stream_k_needs_half_as_many_tiles_as_slots():
    """A stream-K tile is taken with at least half as many tiles as CTA
    slots (tiles then spread over at most three CTAs); with fewer it is
    refused (the split sub-space plans serve small batches)."""
    import paper_1512_06473_gb300 as q
    V = q.fused_variants()
    v = [i for i, f in enumerate(V) if f["SK"] and not f["BF"] and not f["TC"]
         and (f["P"], f["CTW"], f["NW"], f["CSP4"]) == (6, 8, 16, 4)][0]
    # 13x13 maps: one 192-position tile per image, 2 tiles of 128 channels
    p = q.conv_plan(40, 8, 13, 13, 256, 3, 3, 1, 1, 4, 32, algo=v)   # 80 tiles
    assert p["stream_k"] == 1 and p["ctas"] == 152, p
    with pytest.raises(q.QcnnError) as e:
        q.conv_plan(30, 8, 13, 13, 256, 3, 3, 1, 1, 4, 32, algo=v)   # 60 tiles
    assert e.value.status == _lib.ERR_UNSUPPORTED


@_planner
def test_fc_clusters_only_with_many_splits():
    """The FC planner groups split CTAs into clusters only from 64 splits
    up (fewer splits measured slower with clusters), and then into clusters
    that divide the split count."""
    import paper_1512_06473_gb300 as q
    for N in (1, 2, 8, 16, 64, 128, 256):
        for Cs, Ct in list(ALEX_FC.values()) + [(512, 256)]:
            f = q.fc_plan(N, Cs, Ct, K=16 if Cs == 512 else 32)
            assert f["splits"] % f["cluster"] == 0, (N, Cs, Ct, f)
            if f["splits"] < 64:
                assert f["cluster"] == 1, (N, Cs, Ct, f)
            assert f["cluster"] in (1, 2, 4, 8), (N, Cs, Ct, f)


def test_plan_info_arguments():
    info7, info5 = (ctypes.c_int * 8)(), (ctypes.c_int * 6)()
    args = (2, 8, 9, 9, 4, 3, 3, 1, 1, 4, 16, 1)
    assert lib.qcnn_conv_plan_info(*args, 0, 0, None) == _lib.ERR_INVALID_ARG
    assert lib.qcnn_conv_plan_info(*args, 0, 0, info7) == _lib.OK
    assert info7[0] == 1 and info7[4] >= 1  # fused, stride 1
    # the fused kernel is stride-1 only; the unfused path has no bfloat16 tables
    assert lib.qcnn_conv_plan_info(2, 8, 9, 9, 4, 3, 3, 2, 1, 4, 16, 1, 1, 0, info7) \
        == _lib.ERR_UNSUPPORTED
    assert lib.qcnn_conv_plan_info(*args, 2, 1, info7) == _lib.ERR_UNSUPPORTED
    assert lib.qcnn_conv_plan_info(*args, 2, 0, info7) == _lib.OK
    assert (info7[0], info7[1], info7[6]) == (2, -1, 0)
    assert lib.qcnn_fc_plan_info(2, 12, 4, 3, 16, 0, None) == _lib.ERR_INVALID_ARG
    assert lib.qcnn_fc_plan_info(2, 10, 4, 3, 16, 0, info5) == _lib.ERR_INVALID_ARG
    assert lib.qcnn_fc_plan_info(2, 12, 4, 3, 16, 0, info5) == _lib.OK
    assert info5[4] == info5[2] * -(-2 // info5[0]) * -(-4 // info5[1])


@_planner
def test_net_plan_info_binding():
    """Net.plan_info marshals qcnn_net_plan_info (planning only: host tensors
    stand in for the device weights)."""
    import torch
    import paper_1512_06473_gb300 as q
    w = synth.alexnet()
    layers = []
    for L in w.layers:
        if isinstance(L, synth.Conv):
            layers.append(q.ConvLayer(torch.zeros(L.M, L.K, L.Csp),
                                      torch.zeros(L.Ct, L.kh * L.kw, L.M, dtype=torch.uint8), None,
                                      L.Ct, L.kh, L.kw, L.stride, L.pad, L.relu))
        elif isinstance(L, synth.FC):
            layers.append(q.FCLayer(torch.zeros(L.M, L.K, L.Csp),
                                    torch.zeros(L.M, L.Ct, dtype=torch.uint8), None, L.relu))
        else:
            layers.append(q.PoolLayer(L.k, L.s))
    net = q.Net(layers, tuple(w.in_shape))
    b1 = net.plan_info(1)
    assert [i for i, d in enumerate(b1) if d["leaves_partials"]] == [2, 6, 8, 9]
    assert [i for i, d in enumerate(b1) if d["takes_partials"]] == [3, 7, 9, 10]
    assert not any(d["leaves_partials"] or d["takes_partials"]
                   for d in net.plan_info(128, host_io=True))
