"""CUDA path (through the C ABI) against the float64 oracle, element by element.

Tolerance: max|gpu - oracle| / max|oracle| <= 1e-5 for every fp32 result
(the bar the method's fp32 path is held to); integer-valued inputs must give
bit-identical results, since then every partial sum is exact in fp32."""
import concurrent.futures as cf
import os

import numpy as np
import pytest
import torch

import oracle
import paper_1512_06473_gb300 as q
import synth

pytestmark = pytest.mark.gpu
TOL = 1e-5


def rel(got, ref):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    return float(np.max(np.abs(got - ref)) / max(np.max(np.abs(ref)), 1e-30))


def cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def conv_case(seed, N, Cs, H, W, Ct, kh, kw, Csp, K, integer=False):
    M = Cs // Csp
    if integer:
        x = synth.small_integers((N, Cs, H, W), -8, 8, seed, 0)
        D = synth.small_integers((M, K, Csp), -8, 8, seed, 1)
        b = synth.small_integers((Ct,), -8, 8, seed, 3)
    else:
        x = synth.normal((N, Cs, H, W), 1.0, seed, 0)
        D = synth.normal((M, K, Csp), 0.5, seed, 1)
        b = synth.normal((Ct,), 0.1, seed, 3)
    codes = synth.uniform_codes((Ct, kh * kw, M), K, seed, 2)
    return x, D, codes, b


# (N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K)
CONV_SWEEP = [
    (1, 4, 5, 5, 3, 3, 3, 1, 1, 4, 5),
    (2, 8, 13, 13, 40, 3, 3, 1, 1, 4, 128),     # several bands, ragged channel tile
    (1, 16, 27, 27, 70, 5, 5, 1, 2, 4, 128),    # AlexNet conv2-like, ragged Ct
    (1, 12, 20, 33, 17, 3, 3, 1, 1, 3, 64),     # Csp = 3, wide map
    (2, 16, 9, 11, 9, 3, 3, 1, 0, 8, 256),      # K = 256, no padding
    (1, 8, 7, 7, 5, 1, 1, 1, 0, 2, 16),         # 1x1 kernel
    (1, 8, 6, 9, 33, 3, 5, 1, 2, 1, 2),         # non-square kernel, Csp = 1
    (1, 6, 15, 15, 20, 3, 3, 2, 1, 6, 32),      # stride 2
    (1, 3, 39, 39, 24, 11, 11, 4, 0, 3, 128),   # conv1-like: stride 4, M = 1
    (1, 8, 1, 1, 4, 1, 1, 1, 0, 4, 1),          # 1x1 map, K = 1
    (3, 8, 4, 70, 65, 3, 3, 1, 1, 4, 32),       # map wider than one warp slot
    (1, 8, 58, 3, 16, 3, 3, 1, 1, 8, 16),       # tall, narrow map
    (1, 8, 6, 7, 12, 1, 1, 1, 1, 4, 16),        # padding wider than the kernel: Wo > W + pad
    (2, 8, 5, 6, 20, 3, 3, 1, 3, 4, 32),        # pad 3 around a 3x3 kernel
    (1, 8, 9, 10, 18, 1, 5, 1, 2, 4, 16),       # 1x5 kernel, pad 2 on every side
    (2, 8, 17, 19, 40, 5, 5, 3, 2, 4, 64),      # stride 3 with padding: phases of 2x2 .. 1x1
    (1, 16, 23, 23, 130, 3, 3, 2, 0, 8, 256),   # stride 2, K = 256, ragged channel tile
]


@pytest.mark.parametrize("case", CONV_SWEEP, ids=lambda c: "x".join(map(str, c)))
@pytest.mark.parametrize("algo", ["auto", "unfused", "chunked", "phase"])
def test_conv_sweep(case, algo):
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    x, D, codes, b = conv_case(hash(case) % 1000, N, Cs, H, W, Ct, kh, kw, Csp, K)
    ref = oracle.conv_forward(x, D, codes, kh, kw, s, p, b, relu=False)
    got = q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b), algo=algo)
    assert rel(host(got), ref) <= TOL
    ref_r = np.maximum(ref, 0)
    got_r = q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b), relu=True, algo=algo)
    assert rel(host(got_r), ref_r) <= TOL


@pytest.mark.parametrize("case", [c for c in CONV_SWEEP if c[7] == 1], ids=lambda c: "x".join(map(str, c)))
def test_conv_fused_forced(case):
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    x, D, codes, b = conv_case(7, N, Cs, H, W, Ct, kh, kw, Csp, K)
    ref = oracle.conv_forward(x, D, codes, kh, kw, s, p, b)
    got = q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b), algo="fused")
    assert rel(host(got), ref) <= TOL


@pytest.mark.parametrize("algo", ["fused", "unfused", "chunked", "phase"])
def test_conv_integer_bit_exact(algo):
    case = (2, 16, 14, 13, 36, 3, 3, 1, 1, 4, 32)
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    x, D, codes, b = conv_case(3, N, Cs, H, W, Ct, kh, kw, Csp, K, integer=True)
    ref = oracle.conv_forward(x, D, codes, kh, kw, s, p, b)
    got = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b), algo=algo))
    assert np.array_equal(got.astype(np.float64), ref)


def test_conv_codeword_renumbering_is_bit_identical():
    N, Cs, H, W, Ct, kh, kw, Csp, K = 1, 16, 13, 13, 24, 3, 3, 4, 128
    x, D, codes, b = conv_case(5, N, Cs, H, W, Ct, kh, kw, Csp, K)
    M = Cs // Csp
    r = np.random.default_rng(1)
    perm = np.stack([r.permutation(K) for _ in range(M)])
    Dp = np.empty_like(D)
    for m in range(M):
        Dp[m, perm[m]] = D[m]
    cp = perm[np.arange(M)[None, None, :], codes.astype(np.int64)].astype(np.uint8)
    a = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, 1, 1, cuda(b)))
    c = host(q.conv_forward(cuda(x), cuda(Dp), cuda(cp), kh, kw, 1, 1, cuda(b)))
    assert np.array_equal(a, c)


def test_conv_packed_codes_match_canonical():
    N, Cs, H, W, Ct, kh, kw, Csp, K = 2, 24, 27, 27, 48, 5, 5, 4, 128
    x, D, codes, b = conv_case(9, N, Cs, H, W, Ct, kh, kw, Csp, K)
    packed = q.conv_pack_codes(cuda(codes), K, kh, kw)
    a = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, 1, 2, cuda(b)))
    c = host(q.conv_forward(cuda(x), cuda(D), packed, kh, kw, 1, 2, cuda(b), packed=True, Ct=Ct))
    assert np.array_equal(a, c)


def test_conv_is_deterministic():
    N, Cs, H, W, Ct, kh, kw, Csp, K = 2, 32, 27, 27, 64, 5, 5, 4, 128
    x, D, codes, b = conv_case(11, N, Cs, H, W, Ct, kh, kw, Csp, K)
    a = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, 1, 2, cuda(b)))
    c = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, 1, 2, cuda(b)))
    assert np.array_equal(a, c)


def test_out_of_range_codes_are_clamped_not_faulting():
    """Codes >= K are a caller error; the kernels clamp them to K - 1, so the
    result equals the one with clamped codes (and no access leaves the table)."""
    N, Cs, H, W, Ct, kh, kw, Csp, K = 1, 8, 9, 9, 16, 3, 3, 4, 100
    x, D, codes, b = conv_case(13, N, Cs, H, W, Ct, kh, kw, Csp, K)
    bad = codes.copy()
    bad[::3, ::2, :] = 255
    good = np.minimum(bad, K - 1).astype(np.uint8)
    for algo in ("fused", "unfused", "chunked", "phase"):
        a = host(q.conv_forward(cuda(x), cuda(D), cuda(bad), kh, kw, 1, 1, cuda(b), algo=algo))
        c = host(q.conv_forward(cuda(x), cuda(D), cuda(good), kh, kw, 1, 1, cuda(b), algo=algo))
        assert np.array_equal(a, c)
    xf = synth.normal((3, 32), 1.0, 1)
    Df = synth.normal((8, 20, 4), 1.0, 2)
    cf = np.full((8, 10), 200, np.uint8)
    a = host(q.fc_forward(cuda(xf), cuda(Df), cuda(cf)))
    c = host(q.fc_forward(cuda(xf), cuda(Df), cuda(np.full((8, 10), 19, np.uint8))))
    assert np.array_equal(a, c)


# (N, Cs, Ct, Csp, K)
FC_SWEEP = [
    (1, 4, 3, 4, 5),
    (8, 512, 256, 4, 16),       # the single-layer FC workload
    (3, 96, 7, 3, 32),          # Ct not a multiple of 4
    (33, 128, 1030, 4, 32),     # ragged image and output tiles
    (2, 64, 100, 8, 256),       # K = 256 (bank conflicts, still exact)
    (5, 40, 64, 1, 2),          # Csp = 1
    (70, 2304, 513, 4, 32),     # many chunks, splits
    (1, 9216, 4096, 4, 32),     # fc6 at batch 1
    (128, 4096, 1000, 4, 32),   # fc8 at batch 128: 16 images x 4 outputs per lane
    (100, 6144, 1030, 6, 64),   # the same tile, ragged images and outputs, C's = 6
]


@pytest.mark.parametrize("case", FC_SWEEP, ids=lambda c: "x".join(map(str, c)))
def test_fc_sweep(case):
    N, Cs, Ct, Csp, K = case
    M = Cs // Csp
    x = synth.normal((N, Cs), 1.0, 20, *case)
    D = synth.normal((M, K, Csp), 0.5, 21, *case)
    codes = synth.uniform_codes((M, Ct), K, 22, *case)
    b = synth.normal((Ct,), 0.1, 23, *case)
    for relu in (False, True):
        ref = oracle.fc_forward(x, D, codes, b, relu)
        got = q.fc_forward(cuda(x), cuda(D), cuda(codes), cuda(b), relu=relu)
        assert rel(host(got), ref) <= TOL


# Small batches (the sub-spaces split over many CTAs): (N, Cs, Ct, Csp, K)
FC_SMALL = [
    (1, 9216, 4096, 4, 32),    # fc6 at batch 1
    (1, 4096, 1000, 4, 32),    # fc8 at batch 1: ragged last tile
    (8, 512, 256, 4, 16),      # the single-layer FC workload
    (3, 96, 70, 3, 5),         # odd batch, K not a power of two, tiny M
    (5, 64, 1030, 8, 32),      # Ct % 4 == 2: codes copied byte by byte
    (2, 40, 64, 1, 2),         # C's = 1, K = 2
    (7, 2304, 513, 4, 32),     # many sub-spaces
    (1, 12, 3, 4, 32),         # M = 3
]


@pytest.mark.parametrize("case", FC_SMALL, ids=lambda c: "x".join(map(str, c)))
def test_fc_small_batch(case):
    N, Cs, Ct, Csp, K = case
    M = Cs // Csp
    x = synth.normal((N, Cs), 1.0, 24, *case)
    D = synth.normal((M, K, Csp), 0.5, 25, *case)
    codes = synth.uniform_codes((M, Ct), K, 26, *case)
    b = synth.normal((Ct,), 0.1, 27, *case)
    for relu in (False, True):
        ref = oracle.fc_forward(x, D, codes, b, relu)
        got = host(q.fc_forward(cuda(x), cuda(D), cuda(codes), cuda(b), relu=relu))
        assert rel(got, ref) <= TOL
    # bit-packed codes, same plan
    rows = q.fc_pack_codes(cuda(codes), K)
    got = host(q.fc_forward(cuda(x), cuda(D), rows, cuda(b), Ct=Ct))
    assert rel(got, oracle.fc_forward(x, D, codes, b)) <= TOL
    # integer data: exact in any summation order
    xi = synth.small_integers((N, Cs), -8, 8, 28, *case)
    Di = synth.small_integers((M, K, Csp), -8, 8, 29, *case)
    bi = synth.small_integers((Ct,), -8, 8, 30, *case)
    gi = host(q.fc_forward(cuda(xi), cuda(Di), cuda(codes), cuda(bi)))
    assert np.array_equal(gi.astype(np.float64), oracle.fc_forward(xi, Di, codes, bi))
    # deterministic
    again = host(q.fc_forward(cuda(x), cuda(D), cuda(codes), cuda(b)))
    assert np.array_equal(again, host(q.fc_forward(cuda(x), cuda(D), cuda(codes), cuda(b))))


def test_fc_integer_bit_exact():
    N, Cs, Ct, Csp, K = 17, 256, 300, 4, 32
    M = Cs // Csp
    x = synth.small_integers((N, Cs), -8, 8, 30)
    D = synth.small_integers((M, K, Csp), -8, 8, 31)
    codes = synth.uniform_codes((M, Ct), K, 32)
    b = synth.small_integers((Ct,), -8, 8, 33)
    ref = oracle.fc_forward(x, D, codes, b)
    got = host(q.fc_forward(cuda(x), cuda(D), cuda(codes), cuda(b)))
    assert np.array_equal(got.astype(np.float64), ref)


@pytest.mark.parametrize("shape", [(2, 8, 5, 7, 4, 16), (1, 12, 1, 1, 3, 5), (3, 16, 9, 9, 8, 128),
                                   (1, 6, 4, 4, 2, 256)])
def test_lut_build(shape):
    N, Cs, H, W, Csp, K = shape
    M = Cs // Csp
    x = synth.normal((N, Cs, H, W), 1.0, 40, *shape)
    D = synth.normal((M, K, Csp), 1.0, 41, *shape)
    ref = oracle.conv_lut(x, D)
    got = host(q.lut_build(cuda(x), cuda(D)))
    assert rel(got, ref) <= TOL
    xf = x[:, :, 0, 0].copy()
    assert rel(host(q.lut_build(cuda(xf), cuda(D))), oracle.fc_lut(xf, D)[:, :, None, :]) <= TOL


@pytest.mark.parametrize("shape", [(2, 3, 55, 55, 3, 2), (1, 5, 13, 13, 3, 2), (1, 4, 8, 9, 2, 2)])
def test_maxpool(shape):
    N, C, H, W, k, s = shape
    x = synth.normal((N, C, H, W), 1.0, 50, *shape)
    assert np.array_equal(host(q.maxpool(cuda(x), k, s)).astype(np.float64), oracle.maxpool(x, k, s))


# ---------------------------------------------------------------- networks
def build_net(w, params, packed=False):
    layers = []
    for L, P in zip(w.layers, params):
        if isinstance(L, synth.Conv):
            codes = cuda(P["codes"])
            if packed:
                codes = q.conv_pack_codes(codes, L.K, L.kh, L.kw)
            layers.append(q.ConvLayer(cuda(P["D"]), codes, cuda(P["bias"]), L.Ct, L.kh, L.kw,
                                      L.stride, L.pad, L.relu, packed=packed))
        elif isinstance(L, synth.FC):
            layers.append(q.FCLayer(cuda(P["D"]), cuda(P["codes"]), cuda(P["bias"]), L.relu))
        else:
            layers.append(q.PoolLayer(L.k, L.s))
    in_shape = tuple(w.in_shape) if len(w.in_shape) == 3 else (w.in_shape[0], 1, 1)
    return q.Net(layers, in_shape)


def oracle_layers(w, params):
    return [synth.oracle_layer_dict(L, P) for L, P in zip(w.layers, params)]


def oracle_net_images(x, ol, threads=None):
    """The oracle stack on every image of x, one image per task on a thread
    pool (the C oracle releases the interpreter lock while it runs), stacked
    in image order."""
    threads = threads or min(32, os.cpu_count() or 1)
    with cf.ThreadPoolExecutor(threads) as ex:
        outs = list(ex.map(lambda n: oracle.net_forward(x[n:n + 1], ol), range(x.shape[0])))
    return np.concatenate(outs, axis=0)


def run_workload(name, N):
    """The workload's whole stack at batch N through qcnn_net_forward (codes
    packed at load, as the benchmark runs it), against the oracle on every
    image."""
    w = synth.WORKLOADS[name]
    params = w.params()
    x = w.input(N)
    net = build_net(w, params, packed=True)
    xin = x if x.ndim == 4 else x.reshape(N, -1, 1, 1)
    got = host(net.forward(cuda(xin)))
    ref = oracle_net_images(x, oracle_layers(w, params))
    return rel(got.reshape(ref.shape), ref)


@pytest.mark.parametrize("name,N", [
    ("fc_512x256_b8", 8),
    ("conv3x3_64x56x56_b1", 1),
    ("vgg16_conv_stack", 1),
    ("alexnet_fc678", 1),
    ("alexnet_fc678", 64),
    ("alexnet_qcnn", 1),
    ("alexnet_qcnn", 8),
])
def test_workload(name, N):
    assert run_workload(name, N) <= TOL


def test_vgg_stack_batch32_all_images():
    assert run_workload("vgg16_conv_stack", 32) <= TOL


def test_fc678_batch256_all_images():
    assert run_workload("alexnet_fc678", 256) <= TOL


def test_alexnet_batch128_bench_launch_all_images():
    """The benchmark's launch configuration: AlexNet-shaped Q-CNN at batch 128
    with packed codes (stream-K cuts tiles between CTAs at batch-dependent
    points), every one of the 128 images against the oracle."""
    assert run_workload("alexnet_qcnn", 128) <= TOL


@pytest.mark.parametrize("N,cluster", [(1, True), (1, False), (8, True), (2, False)])
def test_net_conv_pool_partials_bit_identical_to_layer_calls(N, cluster):
    """A conv layer whose plan leaves split partial sums hands them to the
    max-pool after it instead of a reduction launch.  The AlexNet conv stack
    (conv1 .. pool5) through qcnn_net_forward equals conv_forward and maxpool
    called layer by layer bit for bit, with one launch fewer per such pair.
    Without clusters the stride-phase conv1 leaves partial sums too."""
    w = synth.alexnet()
    params = w.params()
    n = 8  # conv1 .. pool5
    layers, shapes = w.layers[:n], w.shapes()[:n]
    assert isinstance(layers[-1], synth.Pool) and isinstance(layers[-2], synth.Conv)
    dev_layers = []
    for L, P in zip(layers, params):
        if isinstance(L, synth.Conv):
            codes = q.conv_pack_codes(cuda(P["codes"]), L.K, L.kh, L.kw)
            dev_layers.append(q.ConvLayer(cuda(P["D"]), codes, cuda(P["bias"]), L.Ct, L.kh, L.kw,
                                          L.stride, L.pad, L.relu, packed=True, cluster=cluster))
        else:
            dev_layers.append(q.PoolLayer(L.k, L.s))
    net = q.Net(dev_layers, tuple(w.in_shape))
    x = cuda(w.input(N, 11))
    ws = net.alloc_workspace(N)
    torch.cuda.synchronize()

    before = q.launch_count()
    h = x
    for L, d in zip(layers, dev_layers):
        if isinstance(L, synth.Conv):
            h = q.conv_forward(h, d.D, d.codes, L.kh, L.kw, L.stride, L.pad, d.bias, L.relu,
                               packed=True, Ct=L.Ct, cluster=cluster)
        else:
            h = q.maxpool(h, L.k, L.s)
    torch.cuda.synchronize()
    calls = q.launch_count() - before

    before = q.launch_count()
    y = net.forward(x, workspace=ws)
    torch.cuda.synchronize()
    launches = q.launch_count() - before

    handed = 0
    for i in range(n - 1):
        L, (sin, _) = layers[i], shapes[i]
        if isinstance(L, synth.Conv) and isinstance(layers[i + 1], synth.Pool):
            p = q.conv_plan(N, L.Cs, sin[1], sin[2], L.Ct, L.kh, L.kw, L.stride, L.pad, L.Csp,
                            L.K, cluster=cluster)
            if p["algo"] in ("fused", "phase") and not p["stream_k"] and \
                    p["splits"] // p["cluster"] > 1:
                handed += 1
    if N == 1:
        assert handed >= (3 if not cluster else 2)
    assert torch.equal(y, h)
    assert launches == calls - handed


def test_net_forward_host_matches_device():
    w = synth.alexnet()
    params = w.params()
    net = build_net(w, params, packed=True)
    N = 4
    x = w.input(N, 5)
    dev = host(net.forward(cuda(x)))
    xh = torch.from_numpy(x).pin_memory()
    yh = torch.empty((N, 1000), dtype=torch.float32).pin_memory()
    ws = net.alloc_workspace(N, host_io=True)
    net.forward_host(xh, yh, ws)
    assert np.array_equal(yh.numpy(), dev)


def test_net_forward_host_sliced_input():
    """N = 32: the input is copied in four slices of 8 images and the first
    layer runs per slice while the rest copy; the result matches the device
    path (the first layer's plan can differ at batch 8, so within the fp32
    bar rather than bit for bit)."""
    w = synth.alexnet()
    params = w.params()
    net = build_net(w, params, packed=True)
    N = 32
    x = w.input(N, 6)
    dev = host(net.forward(cuda(x)))
    xh = torch.from_numpy(x).pin_memory()
    yh = torch.empty((N, 1000), dtype=torch.float32).pin_memory()
    ws = net.alloc_workspace(N, host_io=True)
    for _ in range(2):  # the second call reuses the library's copy stream
        yh.zero_()
        net.forward_host(xh, yh, ws)
        assert rel(yh.numpy(), dev) <= TOL


@pytest.mark.parametrize("name", ["conv3x3_64x56x56_b1", "fc_512x256_b8", "alexnet_fc678"])
def test_net_forward_host_sliced_single_layer_and_fc_first(name):
    """Host input in four slices of 8 images for a one-layer stack (the
    first layer's slices are the final output) and for stacks whose first
    layer is FC (slices of flattened rows)."""
    w = synth.WORKLOADS[name]
    params = w.params()
    net = build_net(w, params, packed=True)
    N = 32
    x = w.input(N, 7).reshape((N,) + net.in_shape)
    dev = host(net.forward(cuda(x)))
    xh = torch.from_numpy(x).pin_memory()
    yh = torch.empty(dev.shape, dtype=torch.float32).pin_memory()
    ws = net.alloc_workspace(N, host_io=True)
    net.forward_host(xh, yh, ws)
    assert rel(yh.numpy(), dev) <= TOL


def test_launch_counter_counts_kernels():
    x = cuda(synth.normal((2, 32), 1.0, 1))
    D = cuda(synth.normal((8, 16, 4), 1.0, 2))
    c = cuda(synth.uniform_codes((8, 12), 16, 3))
    before = q.launch_count()
    q.fc_forward(x, D, c)
    torch.cuda.synchronize()
    assert q.launch_count() > before


# Large batches run a stream-K schedule: persistent CTAs take equal runs of
# (tile, sub-space) units, tiles cut between two CTAs are summed by a fix-up
# kernel.  These shapes have more tiles than CTA slots, so they take it.
STREAM_K = [
    (64, 64, 13, 13, 384, 3, 3, 1, 1, 4, 128),   # AlexNet conv3-like, M = 16
    (24, 32, 27, 27, 256, 5, 5, 1, 2, 4, 64),    # conv2-like bands, M = 8
    (160, 16, 13, 13, 256, 3, 3, 1, 1, 8, 32),   # M = 2: one-unit pieces
]


@pytest.mark.parametrize("case", STREAM_K, ids=lambda c: "x".join(map(str, c)))
def test_conv_stream_k(case):
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    x, D, codes, b = conv_case(31, N, Cs, H, W, Ct, kh, kw, Csp, K)
    ref = oracle.conv_forward(x, D, codes, kh, kw, s, p, b, relu=True)
    got = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b), relu=True))
    assert rel(got, ref) <= TOL
    xi, Di, ci, bi = conv_case(32, N, Cs, H, W, Ct, kh, kw, Csp, K, integer=True)
    refi = oracle.conv_forward(xi, Di, ci, kh, kw, s, p, bi)
    goti = host(q.conv_forward(cuda(xi), cuda(Di), cuda(ci), kh, kw, s, p, cuda(bi)))
    assert np.array_equal(goti.astype(np.float64), refi)


# Fewer tiles than CTA slots (but at least half as many): a tile's units
# spread over two or three CTAs, whose pieces (head, middle, tail) the fix-up
# adds in CTA order.
# (case, stream-K tile forced: P, CTW, NW, TC)
STREAM_K_SPREAD = [
    ((48, 32, 13, 13, 384, 3, 3, 1, 1, 4, 64), (6, 16, 12, 0)),    # 96 tiles, M = 8
    ((24, 64, 14, 14, 512, 3, 3, 1, 1, 8, 128), (7, 8, 16, 1)),    # 96 tiles, tensor-core build
    ((40, 8, 13, 13, 256, 3, 3, 1, 1, 4, 32), (6, 8, 16, 0)),      # 80 tiles, M = 2
]


@pytest.mark.parametrize("case,tile", STREAM_K_SPREAD, ids=lambda c: "x".join(map(str, c)))
def test_conv_stream_k_tiles_over_several_ctas(case, tile):
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    v = [i for i, f in enumerate(q.fused_variants())
         if f["SK"] and not f["BF"] and (f["P"], f["CTW"], f["NW"], f["TC"]) == tile
         and f["CSP4"] == (8 if Csp > 4 else 4)][0]
    plan = q.conv_plan(N, Cs, H, W, Ct, kh, kw, s, p, Csp, K, algo=v)
    Ho, Wo = H + 2 * p - kh + 1, W + 2 * p - kw + 1
    pitch = max(W + p, Wo)
    npos = (Ho - 1) * pitch + Wo
    tiles = N * -(-Ct // plan["channels"]) * -(-npos // plan["positions"])
    # fewer tiles than CTAs, at least half as many
    assert plan["stream_k"] == 1 and tiles < plan["ctas"] <= 2 * tiles, (plan, tiles)
    x, D, codes, b = conv_case(33, N, Cs, H, W, Ct, kh, kw, Csp, K)
    ref = oracle.conv_forward(x, D, codes, kh, kw, s, p, b, relu=True)
    got = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b), relu=True,
                              algo=v))
    assert rel(got, ref) <= TOL
    xi, Di, ci, bi = conv_case(34, N, Cs, H, W, Ct, kh, kw, Csp, K, integer=True)
    refi = oracle.conv_forward(xi, Di, ci, kh, kw, s, p, bi)
    goti = host(q.conv_forward(cuda(xi), cuda(Di), cuda(ci), kh, kw, s, p, cuda(bi), algo=v))
    assert np.array_equal(goti.astype(np.float64), refi)


# Small batches split a tile's sub-spaces over several CTAs; the CTAs of one
# tile can form a thread-block cluster that adds their partial tiles in
# distributed shared memory (all of them: no workspace partials and no
# reduction kernel; or groups of them, whose sums the reduction kernel adds).
CLUSTER = [
    (1, 256, 13, 13, 384, 3, 3, 1, 1, 4, 128),    # AlexNet conv3 at batch 1
    (1, 96, 27, 27, 256, 5, 5, 1, 2, 4, 128),     # conv2
    (1, 3, 227, 227, 96, 11, 11, 4, 0, 3, 128),   # conv1 (stride-phase kernel)
    (1, 64, 56, 56, 64, 3, 3, 1, 1, 4, 128),      # the single-layer conv workload
    (1, 512, 14, 14, 512, 3, 3, 1, 1, 8, 128),    # VGG 14x14
    (2, 128, 20, 17, 70, 3, 3, 1, 1, 8, 64),      # ragged tiles and channels
    (1, 64, 9, 9, 40, 5, 5, 2, 2, 4, 32),         # strided, phase kernel
]


@pytest.mark.parametrize("case", CLUSTER, ids=lambda c: "x".join(map(str, c)))
def test_conv_cluster_split_reduction(case):
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    plan = q.conv_plan(N, Cs, H, W, Ct, kh, kw, s, p, Csp, K, packed=False)
    flat = q.conv_plan(N, Cs, H, W, Ct, kh, kw, s, p, Csp, K, packed=False, cluster=False)
    assert flat["cluster"] == 1
    x, D, codes, b = conv_case(41, N, Cs, H, W, Ct, kh, kw, Csp, K)
    ref = oracle.conv_forward(x, D, codes, kh, kw, s, p, b, relu=True)
    got = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b), relu=True))
    assert rel(got, ref) <= TOL, plan
    nocl = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b), relu=True,
                               cluster=False))
    assert rel(nocl, ref) <= TOL, flat
    if plan["cluster"] == plan["splits"] and (plan["variant"], plan["splits"]) == \
            (flat["variant"], flat["splits"]):
        # the cluster adds the splits' tiles in the order the reduction kernel does
        assert np.array_equal(got, nocl)
    xi, Di, ci, bi = conv_case(42, N, Cs, H, W, Ct, kh, kw, Csp, K, integer=True)
    refi = oracle.conv_forward(xi, Di, ci, kh, kw, s, p, bi)
    goti = host(q.conv_forward(cuda(xi), cuda(Di), cuda(ci), kh, kw, s, p, cuda(bi)))
    assert np.array_equal(goti.astype(np.float64), refi), plan


def test_some_small_batch_plans_use_clusters():
    clustered = [q.conv_plan(*c[:9], Csp=c[9], K=c[10], packed=False)["cluster"] > 1
                 for c in CLUSTER]
    assert sum(clustered) >= 4, clustered


# The table build on the tensor cores (tcgen05.mma kind::tf32, 3xTF32 split
# of both operands), forced through the ABI on every tile variant that has
# it: C'_s 5..8, K a multiple of 32, maps of VGG sizes and ragged ones.
TC_CASES = [
    (1, 32, 56, 56, 64, 3, 3, 1, 1, 8, 128),    # VGG 56x56 tile shape
    (2, 48, 28, 28, 80, 3, 3, 1, 1, 8, 64),     # 28x28, ragged channel tile
    (1, 40, 14, 14, 130, 3, 3, 1, 1, 5, 32),    # C'_s = 5 (zero slots), K = 32
    (3, 16, 9, 11, 20, 3, 3, 1, 0, 8, 96),      # small map, K = 96, no padding
]


@pytest.mark.parametrize("case", TC_CASES, ids=lambda c: "x".join(map(str, c)))
def test_tensor_core_table_build(case):
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    x, D, codes, b = conv_case(51, N, Cs, H, W, Ct, kh, kw, Csp, K)
    ref = oracle.conv_forward(x, D, codes, kh, kw, s, p, b, relu=True)
    xi, Di, ci, bi = conv_case(52, N, Cs, H, W, Ct, kh, kw, Csp, K, integer=True)
    refi = oracle.conv_forward(xi, Di, ci, kh, kw, s, p, bi)
    ran = 0
    for v, info in enumerate(q.fused_variants()):
        if not info["TC"]:
            continue
        try:
            got = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b),
                                      relu=True, algo=v))
        except q.QcnnError as e:
            assert e.status == 2, (v, info)  # the variant cannot serve the shape
            continue
        assert rel(got, ref) <= TOL, (v, info)
        goti = host(q.conv_forward(cuda(xi), cuda(Di), cuda(ci), kh, kw, s, p, cuda(bi), algo=v))
        assert np.array_equal(goti.astype(np.float64), refi), (v, info)
        ran += 1
    assert ran >= 1
    assert q.device_check() == 0  # no tensor-core wait gave up


# Every instantiated fused tile variant, forced through the C ABI (the
# planner only ever picks some of them).  Integer inputs with |x|, |D| <= 4
# keep every table entry within 256, so fp32 and bfloat16 tables alike give
# the exact result.  The batches give the stream-K variants at least as many
# tiles as CTA slots.
FORCED = [
    (80, 16, 13, 13, 384, 3, 3, 1, 1, 4, 128),   # C'_s = 4, 13x13 (one- or two-tile maps)
    (32, 16, 27, 27, 256, 5, 5, 1, 2, 8, 64),    # C'_s = 8, 27x27 (several tiles)
]


# Ragged channel and position tiles for the narrow (64-channel) and the
# 12-warp tiles: every forced fp32 variant that can serve the shape, against
# the oracle, on real-valued data (tolerance) -- a channel count that is not a
# multiple of any tile and a map whose positions end mid-slot.
RAGGED = [
    (3, 24, 19, 23, 40, 3, 3, 1, 1, 4, 64),    # Ct = 40 < one 64-channel tile
    (2, 16, 31, 29, 100, 3, 3, 1, 1, 8, 32),   # Ct = 100: two 64-channel tiles, C'_s = 8
]


@pytest.mark.parametrize("case", RAGGED, ids=lambda c: "x".join(map(str, c)))
def test_fused_variants_ragged_tiles(case):
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    x, D, codes, b = conv_case(35, N, Cs, H, W, Ct, kh, kw, Csp, K)
    ref = oracle.conv_forward(x, D, codes, kh, kw, s, p, b, relu=True)
    xd, Dd, cd, bd = cuda(x), cuda(D), cuda(codes), cuda(b)
    ran = 0
    narrow = 0
    for v, info in enumerate(q.fused_variants()):
        if info["BF"]:
            continue
        try:
            got = q.conv_forward(xd, Dd, cd, kh, kw, s, p, bd, relu=True, algo=v)
        except q.QcnnError as e:
            assert e.status == 2, (v, info)
            continue
        assert rel(host(got), ref) <= TOL, (v, info)
        ran += 1
        narrow += info["CTW"] * info["NW"] // info["WP"] == 64
    assert ran >= 10 and narrow >= 1, (ran, narrow)


@pytest.mark.parametrize("case", FORCED, ids=lambda c: "x".join(map(str, c)))
def test_every_fused_variant_is_exact(case):
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    M = Cs // Csp
    x = synth.small_integers((N, Cs, H, W), -4, 4, 61, 0)
    D = synth.small_integers((M, K, Csp), -4, 4, 61, 1)
    b = synth.small_integers((Ct,), -8, 8, 61, 3)
    codes = synth.uniform_codes((Ct, kh * kw, M), K, 61, 2)
    ref = oracle.conv_forward(x, D, codes, kh, kw, s, p, b, relu=True)
    xd, Dd, cd, bd = cuda(x), cuda(D), cuda(codes), cuda(b)
    ran = {"sk": 0, "pipe": 0, "bf": 0, "plain": 0}
    for v, info in enumerate(q.fused_variants()):
        try:
            got = q.conv_forward(xd, Dd, cd, kh, kw, s, p, bd, relu=True, algo=v,
                                 lut="bf16" if info["BF"] else "fp32")
        except q.QcnnError as e:
            assert e.status == 2, (v, info)  # QCNN_ERR_UNSUPPORTED: variant cannot serve it
            continue
        assert np.array_equal(host(got).astype(np.float64), ref), (v, info)
        ran["sk" if info["SK"] else "bf" if info["BF"] else "pipe" if info["PIPE"] else "plain"] += 1
    assert ran["sk"] >= 2 and ran["bf"] >= 2 and ran["plain"] >= 4, ran


def test_smem_load_rate():
    """The roofline's shared-memory peak, measured: a conflict-free 16-byte
    load stream reaches about one 128-byte wavefront per SM per cycle, a
    4-byte one a little less; neither can exceed one."""
    r16 = q.smem_load_rate(16)
    r4 = q.smem_load_rate(4)
    assert 0.8 <= r16 <= 1.01, r16
    assert 0.5 <= r4 <= r16 + 0.01, (r4, r16)
