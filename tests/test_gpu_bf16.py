"""bfloat16 look-up tables (lut="bf16") through the C ABI against the oracle.

The stated bar for reduced-precision tables is max|err| / max|ref| <= 2e-3
against the exact float64 oracle.  Rounding every table entry to bfloat16 (8
significant bits) puts the exact rounding model itself 1.1e-3 - 2.6e-3 from
exact on the benchmark's layers and 1.8e-3 - 5.3e-3 on its stacks, so the
variant meets the bar on some layers and not on others.  The tests say which
(test_benchmark_layers_bf16, test_net_bf16): in tolerance, the GPU result is
held to 2e-3 of the exact oracle; out of tolerance, no claim is made and the
GPU is only checked to implement the rounding model.

Implementation checks on every case:
  * against the oracle's bfloat16 table model (every entry rounded to the
    nearest bfloat16, ties to even, sums exact).  The GPU rounds its fp32
    entry and the model the exact one, so an entry lying within an fp32
    rounding of a bfloat16 rounding boundary can round the other way (a few
    in 10^5): such a "flip" moves the outputs that use the entry by one
    bfloat16 step of the entry.  So every output must be within the fp32 bar
    (1e-5 of the output range) plus two bfloat16 steps of the largest entry,
    and fewer than 1% of the outputs may differ from the model by more than
    the fp32 bar.  A wrong rounding direction, or a wrong copy of the pair
    tables, moves almost every output.
  * against the exact oracle, a bound that holds for any input: rounding an
    entry v to bfloat16 moves it by at most 2^-8 |v| (half a step of 8
    significant bits), so every output is within 2^-8 * (sum of |entries| it
    adds) of the exact one, plus fp32 slack; the sums of |entries| come from a
    float64 conv2d of |LUT| with one-hot code kernels.
Integer data whose entries are exact in bfloat16 must match bit for bit,
and a one-entry table (M = 1, K = 1, D = 1) must return bf16(x) exactly,
ties included."""
import numpy as np
import pytest
import torch

import oracle
import paper_1512_06473_gb300 as q
import synth
from test_gpu_parity import build_net, conv_case, cuda, host, oracle_layers, rel

pytestmark = pytest.mark.gpu


def abs_entry_sums_conv(x, D, codes, kh, kw, s, p):
    """S[n, ct, oy, ox] = sum over the (p_k, m) terms of |LUT entry|."""
    N, Cs, H, W = x.shape
    M, K, Csp = D.shape
    Ct = codes.shape[0]
    T = np.abs(oracle.conv_lut(x, D))  # [N, M, H*W, K]
    T = T.reshape(N, M, H, W, K).transpose(0, 1, 4, 2, 3).reshape(N, M * K, H, W)
    Wk = np.zeros((Ct, M, K, kh * kw))
    ct_i, pk_i, m_i = np.meshgrid(np.arange(Ct), np.arange(kh * kw), np.arange(M), indexing="ij")
    Wk[ct_i, m_i, codes.astype(np.int64), pk_i] = 1.0
    Wk = Wk.reshape(Ct, M * K, kh, kw)
    return torch.nn.functional.conv2d(torch.from_numpy(T), torch.from_numpy(Wk), stride=s,
                                      padding=p).numpy()


def abs_entry_sums_fc(x, D, codes):
    M, K, Csp = D.shape
    T = np.abs(oracle.fc_lut(x, D))  # [N, M, K]
    return T[:, np.arange(M)[:, None], codes.astype(np.int64)].sum(axis=1)


def check_exact(got, exact, S):
    """|got - exact| <= 2^-8 * S (bfloat16 rounding of every entry used) + fp32 slack."""
    got = np.asarray(got, np.float64).reshape(exact.shape)
    bound = 2.0 ** -8 * (1 + 2.0 ** -10) * S + 1e-5 * np.max(np.abs(exact))
    assert np.all(np.abs(got - exact) <= bound), np.max(np.abs(got - exact) - bound)


def check_model(got, model, entry_max, few_flips=True):
    """got against the bfloat16 table model (see the module docstring).
    few_flips=False drops the "fewer than 1% of outputs" part, for layers
    whose few table entries are each summed into many outputs (one flipped
    entry then moves Ct/K of the outputs)."""
    got = np.asarray(got, np.float64).reshape(model.shape)
    d = np.abs(got - model)
    bar = 1e-5 * np.max(np.abs(model))
    flip = 2.0 ** -7 * entry_max  # one bfloat16 step of the largest entry
    assert np.max(d) <= bar + 2 * flip, (np.max(d), bar, flip)
    if few_flips:
        assert np.mean(d > bar) < 0.01, np.mean(d > bar)


# (N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K)
CONV_BF16 = [
    (1, 4, 5, 5, 3, 3, 3, 1, 1, 4, 5),
    (2, 8, 13, 13, 40, 3, 3, 1, 1, 4, 128),     # AlexNet conv3-5 map, ragged Ct
    (1, 16, 27, 27, 70, 5, 5, 1, 2, 4, 128),    # AlexNet conv2 map
    (1, 12, 20, 33, 17, 3, 3, 1, 1, 3, 64),     # odd pitch, Csp = 3
    (2, 16, 9, 11, 9, 3, 3, 1, 0, 8, 256),      # K = 256
    (1, 8, 7, 7, 5, 1, 1, 1, 0, 2, 16),         # 1x1 kernel (only even offsets)
    (1, 8, 6, 9, 33, 3, 5, 1, 2, 1, 2),         # non-square kernel, Csp = 1
    (3, 8, 4, 70, 65, 3, 3, 1, 1, 4, 32),       # map wider than a slot
    (1, 8, 58, 3, 16, 3, 3, 1, 1, 8, 16),       # tall narrow map
    (1, 16, 56, 56, 24, 3, 3, 1, 1, 4, 128),    # 56x56 (VGG / single-layer conv shape)
    (1, 6, 15, 15, 20, 3, 3, 2, 1, 6, 32),      # stride 2 (chunked)
    (1, 3, 39, 39, 24, 11, 11, 4, 0, 3, 128),   # conv1-like, stride 4 (chunked)
]


def _conv_refs(x, D, codes, kh, kw, s, p, b):
    exact = oracle.conv_forward(x, D, codes, kh, kw, s, p, b)
    model = oracle.conv_forward(x, D, codes, kh, kw, s, p, b, lut_bf16=True)
    entry_max = float(np.max(np.abs(oracle.conv_lut(x, D))))
    return exact, model, entry_max, abs_entry_sums_conv(x, D, codes, kh, kw, s, p)


@pytest.mark.parametrize("case", CONV_BF16, ids=lambda c: "x".join(map(str, c)))
@pytest.mark.parametrize("algo", ["auto", "chunked"])
def test_conv_bf16(case, algo):
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    x, D, codes, b = conv_case(hash(case) % 1000 + 1, N, Cs, H, W, Ct, kh, kw, Csp, K)
    exact, model, emax, S = _conv_refs(x, D, codes, kh, kw, s, p, b)
    got = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b), algo=algo,
                              lut="bf16"))
    check_model(got, model, emax)
    check_exact(got, exact, S)


@pytest.mark.parametrize("case", [c for c in CONV_BF16 if c[7] == 1],
                         ids=lambda c: "x".join(map(str, c)))
def test_conv_bf16_fused_forced(case):
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    x, D, codes, b = conv_case(17, N, Cs, H, W, Ct, kh, kw, Csp, K)
    exact, model, emax, S = _conv_refs(x, D, codes, kh, kw, s, p, b)
    got = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b), algo="fused",
                              lut="bf16"))
    check_model(got, model, emax)
    check_exact(got, exact, S)


def _small_int_conv(seed, N, Cs, H, W, Ct, kh, kw, Csp, K):
    """Entries |<x, D>| <= 4 * 4 * Csp <= 128: exact in bfloat16."""
    M = Cs // Csp
    x = synth.small_integers((N, Cs, H, W), -4, 4, seed, 0)
    D = synth.small_integers((M, K, Csp), -4, 4, seed, 1)
    b = synth.small_integers((Ct,), -8, 8, seed, 3)
    codes = synth.uniform_codes((Ct, kh * kw, M), K, seed, 2)
    return x, D, codes, b


@pytest.mark.parametrize("algo,case", [
    ("fused", (2, 16, 14, 13, 36, 3, 3, 1, 1, 4, 32)),
    ("fused", (1, 16, 27, 27, 40, 5, 5, 1, 2, 8, 128)),
    ("chunked", (2, 16, 14, 13, 36, 3, 3, 1, 1, 4, 32)),
    ("chunked", (1, 3, 39, 39, 24, 11, 11, 4, 0, 3, 128)),
])
def test_conv_bf16_integer_bit_exact(algo, case):
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    x, D, codes, b = _small_int_conv(3, N, Cs, H, W, Ct, kh, kw, Csp, K)
    ref = oracle.conv_forward(x, D, codes, kh, kw, s, p, b)
    got = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b), algo=algo,
                              lut="bf16"))
    assert np.array_equal(got.astype(np.float64), ref)


def _tie_values(n, seed):
    """float32 values on, next to and between bfloat16 rounding ties."""
    r = np.random.default_rng(seed)
    mant = r.integers(0, 1 << 7, n)              # 7 stored bits of the bf16 value
    expo = r.integers(-20, 20, n).astype(np.float64)
    base = (1.0 + mant / 128.0) * 2.0 ** expo     # a bfloat16 value
    ulp = 2.0 ** (expo - 7)
    kind = r.integers(0, 4, n)
    frac = np.choose(kind, [0.5, 0.5 - 2.0 ** -16, 0.5 + 2.0 ** -16, r.random(n)])
    v = (base + frac * ulp) * np.where(r.random(n) < 0.5, -1.0, 1.0)
    return v.astype(np.float32)


def test_bf16_rounding_ties_fc_and_conv():
    """One-entry tables: y = bf16(x) exactly, for ties, near-ties and others."""
    x = _tie_values(4096, 5)
    want = oracle.round_bf16(x.astype(np.float64))
    assert np.array_equal(want, torch.from_numpy(x).to(torch.bfloat16).double().numpy())
    D = np.ones((1, 1, 1), np.float32)
    # FC, Cs = Csp = 1: every output is the single entry x * 1
    xf = x.reshape(-1, 1)
    got = host(q.fc_forward(cuda(xf), cuda(D), cuda(np.zeros((1, 3), np.uint8)), lut="bf16"))
    assert np.array_equal(got.astype(np.float64), np.repeat(want.reshape(-1, 1), 3, axis=1))
    # conv, 1x1 kernel, one channel: fused (stride 1) and chunked (stride 2)
    xc = x.reshape(4, 1, 32, 32)
    codes = np.zeros((2, 1, 1), np.uint8)
    wc = want.reshape(4, 1, 32, 32)
    for algo in ("fused", "chunked"):
        got = host(q.conv_forward(cuda(xc), cuda(D), cuda(codes), 1, 1, 1, 0, algo=algo,
                                  lut="bf16"))
        assert np.array_equal(got.astype(np.float64), np.repeat(wc, 2, axis=1)), algo
    got = host(q.conv_forward(cuda(xc), cuda(D), cuda(codes), 1, 1, 2, 0, lut="bf16"))
    assert np.array_equal(got.astype(np.float64), np.repeat(wc[:, :, ::2, ::2], 2, axis=1))


# (N, Cs, Ct, Csp, K)
FC_BF16 = [
    (1, 4, 3, 4, 5),
    (8, 512, 256, 4, 16),       # the single-layer FC workload
    (3, 96, 7, 3, 32),
    (33, 128, 1030, 4, 32),     # odd batch: last image pair half empty
    (2, 64, 100, 8, 256),
    (70, 2304, 513, 4, 32),     # many chunks, splits
    (1, 9216, 4096, 4, 32),     # fc6 at batch 1 (2-byte entries)
    (128, 4096, 1000, 4, 32),   # fc8 at batch 128
    (100, 6144, 1030, 6, 64),   # 16 images per lane, ragged images and outputs
]


@pytest.mark.parametrize("case", FC_BF16, ids=lambda c: "x".join(map(str, c)))
def test_fc_bf16(case):
    N, Cs, Ct, Csp, K = case
    M = Cs // Csp
    x = synth.normal((N, Cs), 1.0, 60, *case)
    D = synth.normal((M, K, Csp), 0.5, 61, *case)
    codes = synth.uniform_codes((M, Ct), K, 62, *case)
    b = synth.normal((Ct,), 0.1, 63, *case)
    exact = oracle.fc_forward(x, D, codes, b)
    model = oracle.fc_forward(x, D, codes, b, lut_bf16=True)
    emax = float(np.max(np.abs(oracle.fc_lut(x, D))))
    got = host(q.fc_forward(cuda(x), cuda(D), cuda(codes), cuda(b), lut="bf16"))
    check_model(got, model, emax)
    check_exact(got, exact, abs_entry_sums_fc(x, D, codes))


@pytest.mark.parametrize("N", [1, 17, 64])
def test_fc_bf16_integer_bit_exact(N):
    Cs, Ct, Csp, K = 256, 300, 4, 32
    M = Cs // Csp
    x = synth.small_integers((N, Cs), -4, 4, 70)
    D = synth.small_integers((M, K, Csp), -4, 4, 71)
    codes = synth.uniform_codes((M, Ct), K, 72)
    b = synth.small_integers((Ct,), -8, 8, 73)
    ref = oracle.fc_forward(x, D, codes, b)
    got = host(q.fc_forward(cuda(x), cuda(D), cuda(codes), cuda(b), lut="bf16"))
    assert np.array_equal(got.astype(np.float64), ref)


@pytest.mark.parametrize("shape", [(2, 8, 5, 7, 4, 16), (3, 16, 9, 9, 8, 128), (1, 6, 4, 4, 2, 256)])
def test_lut_build_bf16(shape):
    """Stand-alone bf16 tables: each entry the bfloat16 rounding of the fp32
    entry, so within one bfloat16 step (2^-8 relative) of the rounded exact
    entry, and equal to it for all but a few."""
    N, Cs, H, W, Csp, K = shape
    M = Cs // Csp
    x = synth.normal((N, Cs, H, W), 1.0, 80, *shape)
    D = synth.normal((M, K, Csp), 1.0, 81, *shape)
    model = oracle.conv_lut(x, D, lut_bf16=True)
    got = host(q.lut_build(cuda(x), cuda(D), lut="bf16").float()).astype(np.float64)
    assert got.shape == model.shape
    diff = np.abs(got - model)
    assert np.all(diff <= 2.0 ** -7 * np.abs(model) + 1e-30)
    assert np.mean(diff > 0) < 1e-3


def test_conv_bf16_deterministic_and_split_consistent():
    """Batch 1 (sub-spaces split over CTAs) gives the same bits on every call."""
    N, Cs, H, W, Ct, kh, kw, Csp, K = 1, 256, 13, 13, 96, 3, 3, 4, 128
    x, D, codes, b = conv_case(23, N, Cs, H, W, Ct, kh, kw, Csp, K)
    a = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, 1, 1, cuda(b), lut="bf16"))
    c = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, 1, 1, cuda(b), lut="bf16"))
    assert np.array_equal(a, c)
    exact, model, emax, S = _conv_refs(x, D, codes, kh, kw, 1, 1, b)
    check_model(a, model, emax)


def _bf16_net(w, params):
    net = build_net(w, params, packed=True)
    for L in net.layers:
        if not isinstance(L, q.PoolLayer):
            L.lut = "bf16"
    return q.Net(net.layers, net.in_shape)


# The stated bar for reduced-precision tables: max|err| / max|ref| <= 2e-3
# against the exact (float64) oracle.
BAR = 2e-3
# A layer or stack is within the bar by construction only when the exact
# bfloat16 table model itself -- every entry rounded exactly, sums exact,
# the best any bfloat16 table can do -- stays clear of it: the GPU rounds its
# fp32 entries, and a few entries within an fp32 rounding of a bfloat16
# boundary round the other way ("flips"), so the model's distance gets a 5%
# margin.  Where the model alone is beyond MODEL_MAX the variant is out of
# tolerance for that layer, whatever the kernel does; there the GPU is only
# checked to implement the rounding model, and no 2e-3 claim is made.
MODEL_MAX = 0.95 * BAR
# Which benchmark layers and stacks fall on which side (seeded inputs, see
# the tests below).  Kept explicit so that the documentation of the variant
# cannot drift from what is measured: (workload, layer index) -> in tolerance.
IN_TOLERANCE_LAYERS = {
    ("alexnet_qcnn", 0): True,    # conv1   model 1.73e-3
    ("alexnet_qcnn", 2): False,   # conv2   model 2.08e-3
    ("alexnet_qcnn", 4): False,   # conv3   model 2.15e-3
    ("alexnet_qcnn", 5): False,   # conv4   model 1.91e-3 (within the margin)
    ("alexnet_qcnn", 6): False,   # conv5   model 2.57e-3
    ("alexnet_qcnn", 8): True,    # fc6     model 1.85e-3
    ("alexnet_qcnn", 9): True,    # fc7     model 1.79e-3
    ("alexnet_qcnn", 10): False,  # fc8     model 2.28e-3
    ("conv3x3_64x56x56_b1", 0): True,   # model 1.83e-3
    ("fc_512x256_b8", 0): True,         # model 1.55e-3
    ("vgg16_conv_stack", 0): True,      # model 1.74e-3
    ("vgg16_conv_stack", 1): True,      # model 1.72e-3
    ("vgg16_conv_stack", 3): False,     # model 1.91e-3 (within the margin)
    ("vgg16_conv_stack", 5): False,     # model 2.04e-3
    ("vgg16_conv_stack", 6): True,      # model 1.87e-3
    ("alexnet_fc678", 0): False,        # fc6 of the fc stack input: 2.00e-3
    ("alexnet_fc678", 1): True,         # model 1.50e-3
    ("alexnet_fc678", 2): True,         # model 1.15e-3
}


@pytest.mark.parametrize("name", ["alexnet_qcnn", "conv3x3_64x56x56_b1", "fc_512x256_b8",
                                  "vgg16_conv_stack", "alexnet_fc678"])
def test_benchmark_layers_bf16(name):
    """Every PQ layer of the workloads with bfloat16 tables, fed the exact
    activations of the layer before it (two images).  Where the rounding
    model is within the margin, the GPU result must be within 2e-3 of the
    exact oracle; elsewhere the variant is out of tolerance by construction
    (the classification is asserted, so it stays true) and the GPU must
    implement the rounding model."""
    w = synth.WORKLOADS[name]
    params = w.params()
    N = 2
    x = w.input(N, 9)
    ol = oracle_layers(w, params)
    acts = [x] + oracle.net_forward(x, ol, return_all=True)
    for i, (L, P) in enumerate(zip(w.layers, params)):
        h = acts[i]
        if isinstance(L, synth.Conv):
            got = q.conv_forward(cuda(h.astype(np.float32)), cuda(P["D"]), cuda(P["codes"]), L.kh,
                                 L.kw, L.stride, L.pad, cuda(P["bias"]), relu=L.relu, lut="bf16")
        elif isinstance(L, synth.FC):
            got = q.fc_forward(cuda(h.reshape(N, -1).astype(np.float32)), cuda(P["D"]),
                               cuda(P["codes"]), cuda(P["bias"]), relu=L.relu, lut="bf16")
        else:
            continue
        ref = acts[i + 1]
        d = synth.oracle_layer_dict(L, P)
        if isinstance(L, synth.Conv):
            model = oracle.conv_forward(h, d["D"], d["codes"], L.kh, L.kw, L.stride, L.pad,
                                        d["bias"], L.relu, lut_bf16=True)
            emax = float(np.max(np.abs(oracle.conv_lut(h, d["D"]))))
        else:
            model = oracle.fc_forward(h.reshape(N, -1), d["D"], d["codes"], d["bias"], L.relu,
                                      lut_bf16=True)
            emax = float(np.max(np.abs(oracle.fc_lut(h.reshape(N, -1), d["D"]))))
        e_model = rel(model.reshape(ref.shape), ref)
        within = e_model <= MODEL_MAX
        assert within == IN_TOLERANCE_LAYERS[(name, i)], (name, i, e_model)
        got = host(got)
        if within:
            assert rel(got.reshape(ref.shape), ref) <= BAR, (name, i)
        else:
            check_model(got.reshape(model.shape), model, emax, few_flips=False)


# whole stacks (batch as in the benchmark configs): in tolerance or not, by
# the same rule as single layers
IN_TOLERANCE_STACKS = {
    "alexnet_qcnn": False,          # model 5.29e-3 after eight PQ layers
    "vgg16_conv_stack": False,      # model 3.86e-3
    "alexnet_fc678": False,         # model 2.25e-3
    "conv3x3_64x56x56_b1": True,    # model 1.76e-3
    "fc_512x256_b8": True,          # model 1.82e-3 at batch 8
}


@pytest.mark.parametrize("name,N", [("alexnet_qcnn", 2), ("vgg16_conv_stack", 1),
                                    ("alexnet_fc678", 2), ("conv3x3_64x56x56_b1", 1),
                                    ("fc_512x256_b8", 8)])
def test_net_bf16(name, N):
    """Whole stacks with bfloat16 tables against the exact oracle: within
    2e-3 where the stack is in tolerance.  Through a stack, rounding flips in
    one layer change the next layer's entries, so a GPU stack and the model
    stack drift apart by about the size of the bfloat16 error itself: out of
    tolerance, only the classification is asserted and no claim is made."""
    w = synth.WORKLOADS[name]
    params = w.params()
    x = w.input(N)
    net = _bf16_net(w, params)
    xin = x if x.ndim == 4 else x.reshape(N, -1, 1, 1)
    got = host(net.forward(cuda(xin)))
    ol = oracle_layers(w, params)
    exact = oracle.net_forward(x, ol)
    model = oracle.net_forward(x, [dict(d, lut_bf16=True) if d["kind"] != "maxpool" else d
                                   for d in ol])
    within = rel(model, exact) <= MODEL_MAX
    assert within == IN_TOLERANCE_STACKS[name], (name, rel(model, exact))
    if within:
        assert rel(got.reshape(exact.shape), exact) <= BAR


@pytest.mark.parametrize("case", [(64, 64, 13, 13, 384, 3, 3, 1, 1, 4, 128),
                                  (40, 32, 27, 27, 256, 5, 5, 1, 2, 4, 64)],
                         ids=lambda c: "x".join(map(str, c)))
def test_conv_bf16_stream_k(case):
    """bf16 tables under the stream-K schedule (more tiles than CTA slots)."""
    N, Cs, H, W, Ct, kh, kw, s, p, Csp, K = case
    x, D, codes, b = conv_case(33, N, Cs, H, W, Ct, kh, kw, Csp, K)
    exact, model, emax, S = _conv_refs(x, D, codes, kh, kw, s, p, b)
    got = host(q.conv_forward(cuda(x), cuda(D), cuda(codes), kh, kw, s, p, cuda(b), lut="bf16"))
    check_model(got, model, emax)
    check_exact(got, exact, S)
