"""Pins for the float64 oracle: facts fixed by the paper and by mathematics,
each computed by a route that does not go through the oracle's own code.

Every pin takes an ``oracle.Oracle`` instance and returns a list of failure
messages (empty = pinned).  ``test_oracle_pins.py`` runs them on the oracle;
``test_oracle_mutants.py`` runs them on copies of the oracle's C file with a
planted mistake and checks that at least one pin fails for each.

Independent routes used here:
  * Eq. 4 / Eq. 6 give the meaning of the codes: the m-th sub-vector of weight
    vector c_t (at kernel offset p_k) is replaced by sub-codeword
    D^(m)_{k_m}.  Building that dense weight tensor W_hat by indexing and
    running torch's float64 conv2d / matmul (Eq. 1 / Eq. 2) must give the
    same response as the look-up-table route of Eq. 5 / Eq. 7.
  * Exactness (the approximation in Eq. 3 is an equality when every weight
    sub-vector is itself a sub-codeword): a dense W is drawn first, from a
    set of K sub-vectors per sub-space; its codes are recovered by an exact
    nearest-sub-codeword search (Eq. 4 / Eq. 6 solved with zero error); the
    Q-CNN response must equal conv2d(x, W).
  * Linearity in the input, invariance under renumbering sub-codewords,
    the K = 1 closed form, 1x1 conv == FC, and one-hot codebooks that make
    the look-up table a copy of the input.
"""
from __future__ import annotations

import numpy as np
import torch
import torch.nn.functional as F




def _rng(seed):
    return np.random.default_rng(seed)


def w_hat_conv(D, codes, kh, kw):
    """Dense kernels from Eq. 6: W[ct, m*Csp + j, ky, kx] = D[m, codes[ct, ky*kw+kx, m], j]."""
    M, K, Csp = D.shape
    Ct = codes.shape[0]
    sel = D[np.arange(M)[None, None, :], codes.astype(np.int64)]  # (Ct, kk, M, Csp)
    return sel.reshape(Ct, kh, kw, M * Csp).transpose(0, 3, 1, 2)


def w_hat_fc(D, codes):
    """Dense weights from Eq. 4: W[ct, m*Csp + j] = D[m, codes[m, ct], j]."""
    M, K, Csp = D.shape
    sel = D[np.arange(M)[:, None], codes.astype(np.int64)]  # (M, Ct, Csp)
    return sel.transpose(1, 0, 2).reshape(codes.shape[1], M * Csp)


def torch_conv(x, W, bias, stride, pad, relu):
    y = F.conv2d(torch.from_numpy(np.asarray(x, np.float64)), torch.from_numpy(W),
                 None if bias is None else torch.from_numpy(np.asarray(bias, np.float64)),
                 stride=stride, padding=pad)
    if relu:
        y = F.relu(y)
    return y.numpy()


def torch_fc(x, W, bias, relu):
    y = torch.from_numpy(np.asarray(x, np.float64)) @ torch.from_numpy(W).T
    if bias is not None:
        y = y + torch.from_numpy(np.asarray(bias, np.float64))
    if relu:
        y = F.relu(y)
    return y.numpy()


def relerr(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    den = max(np.max(np.abs(b)), 1e-300)
    return float(np.max(np.abs(a - b)) / den) if a.size else 0.0


def rand_conv_case(seed, N, Cs, H, W, Ct, kh, kw, Csp, K, bias=True):
    r = _rng(seed)
    M = Cs // Csp
    x = r.standard_normal((N, Cs, H, W))
    D = r.standard_normal((M, K, Csp))
    codes = r.integers(0, K, (Ct, kh * kw, M), dtype=np.uint8)
    b = r.standard_normal(Ct) if bias else None
    return x, D, codes, b


def rand_fc_case(seed, N, Cs, Ct, Csp, K, bias=True):
    r = _rng(seed)
    M = Cs // Csp
    x = r.standard_normal((N, Cs))
    D = r.standard_normal((M, K, Csp))
    codes = r.integers(0, K, (M, Ct), dtype=np.uint8)
    b = r.standard_normal(Ct) if bias else None
    return x, D, codes, b


# (N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K, relu)
CONV_CASES = [
    (1, 4, 5, 5, 3, 3, 3, 1, 1, 4, 5, False),
    (2, 6, 7, 6, 5, 3, 3, 1, 1, 2, 16, True),
    (1, 6, 9, 8, 4, 5, 5, 1, 2, 3, 7, False),
    (2, 8, 11, 10, 3, 3, 3, 2, 1, 8, 2, True),
    (1, 3, 23, 19, 4, 11, 11, 4, 0, 3, 128, False),
    (1, 4, 8, 9, 2, 1, 1, 1, 0, 1, 256, False),
    (1, 8, 6, 7, 3, 2, 3, 1, 0, 4, 1, False),
    (2, 12, 7, 7, 5, 3, 1, 2, 2, 4, 33, True),
    (1, 16, 6, 6, 6, 3, 3, 1, 1, 8, 128, True),
]

# (N, Cs, Ct, Csp, K, relu)
FC_CASES = [
    (1, 4, 3, 4, 5, False),
    (3, 12, 7, 3, 16, True),
    (2, 16, 9, 1, 2, False),
    (4, 32, 17, 4, 32, True),
    (1, 24, 5, 8, 256, False),
    (2, 10, 4, 2, 1, False),
]


def pin_conv_vs_dense(o, cases=CONV_CASES, tol=1e-12):
    fails = []
    for i, (N, Cs, H, W, Ct, kh, kw, s, p, Csp, K, relu) in enumerate(cases):
        x, D, codes, b = rand_conv_case(100 + i, N, Cs, H, W, Ct, kh, kw, Csp, K)
        got = o.conv_forward(x, D, codes, kh, kw, s, p, b, relu)
        ref = torch_conv(x, w_hat_conv(D, codes, kh, kw), b, s, p, relu)
        if got.shape != ref.shape or relerr(got, ref) > tol:
            fails.append(f"conv case {i}: shape {got.shape} vs {ref.shape}, "
                         f"err {relerr(got, ref) if got.shape == ref.shape else 'n/a'}")
    return fails


def pin_fc_vs_dense(o, cases=FC_CASES, tol=1e-12):
    fails = []
    for i, (N, Cs, Ct, Csp, K, relu) in enumerate(cases):
        x, D, codes, b = rand_fc_case(200 + i, N, Cs, Ct, Csp, K)
        got = o.fc_forward(x, D, codes, b, relu)
        ref = torch_fc(x, w_hat_fc(D, codes), b, relu)
        if relerr(got, ref) > tol:
            fails.append(f"fc case {i}: err {relerr(got, ref)}")
    return fails


def pin_integer_exact(o):
    """Small-integer inputs and codebooks: every partial sum is an exact
    integer, so the look-up route and conv2d must agree bit for bit."""
    fails = []
    r = _rng(7)
    N, Cs, H, W, Ct, kh, kw, Csp, K = 2, 8, 7, 6, 5, 3, 3, 4, 9
    M = Cs // Csp
    x = r.integers(-8, 9, (N, Cs, H, W)).astype(np.float64)
    D = r.integers(-8, 9, (M, K, Csp)).astype(np.float64)
    codes = r.integers(0, K, (Ct, kh * kw, M), dtype=np.uint8)
    b = r.integers(-8, 9, Ct).astype(np.float64)
    got = o.conv_forward(x, D, codes, kh, kw, 1, 1, b, False)
    ref = torch_conv(x, w_hat_conv(D, codes, kh, kw), b, 1, 1, False)
    if not np.array_equal(got, ref):
        fails.append("integer conv not bit-exact")
    xf = r.integers(-8, 9, (3, 12)).astype(np.float64)
    Df = r.integers(-8, 9, (3, 6, 4)).astype(np.float64)
    cf = r.integers(0, 6, (3, 10), dtype=np.uint8)
    if not np.array_equal(o.fc_forward(xf, Df, cf), torch_fc(xf, w_hat_fc(Df, cf), None, False)):
        fails.append("integer fc not bit-exact")
    return fails


def _exact_codes(Wsub, D):
    """Recover the sub-codeword index of every weight sub-vector by an exact
    nearest-neighbour search: Wsub [..., M, Csp], D [M, K, Csp]."""
    d2 = ((Wsub[..., None, :] - D) ** 2).sum(-1)  # [..., M, K]
    idx = d2.argmin(-1)
    assert np.all(np.take_along_axis(d2, idx[..., None], -1) == 0)
    return idx.astype(np.uint8)


def pin_exactness(o):
    """Eq. 3 / Eq. 4: with K covering every distinct weight sub-vector the
    response is the exact dense response of the original weights."""
    fails = []
    r = _rng(11)
    # conv: W drawn first from K prototypes per sub-space
    N, Cs, H, Wd, Ct, kh, kw, Csp, K, s, p = 2, 12, 9, 8, 6, 3, 3, 4, 5, 1, 1
    M = Cs // Csp
    D = r.standard_normal((M, K, Csp))
    pick = r.integers(0, K, (Ct, kh, kw, M))
    Wsub = D[np.arange(M), pick]                       # (Ct, kh, kw, M, Csp)
    Wt = Wsub.reshape(Ct, kh, kw, Cs).transpose(0, 3, 1, 2).copy()
    codes = _exact_codes(Wsub.reshape(Ct, kh * kw, M, Csp), D)
    x = r.standard_normal((N, Cs, H, Wd))
    got = o.conv_forward(x, D, codes, kh, kw, s, p)
    ref = torch_conv(x, Wt, None, s, p, False)
    if relerr(got, ref) > 1e-12:
        fails.append(f"conv exactness err {relerr(got, ref)}")
    # fc
    N, Cs, Ct, Csp, K = 3, 20, 11, 5, 4
    M = Cs // Csp
    D = r.standard_normal((M, K, Csp))
    pick = r.integers(0, K, (Ct, M))
    Wf = D[np.arange(M), pick].reshape(Ct, Cs)
    codes = _exact_codes(Wf.reshape(Ct, M, Csp), D).T.copy()  # [M, Ct]
    x = r.standard_normal((N, Cs))
    got = o.fc_forward(x, D, codes)
    ref = torch_fc(x, Wf, None, False)
    if relerr(got, ref) > 1e-12:
        fails.append(f"fc exactness err {relerr(got, ref)}")
    return fails


def pin_linearity(o):
    """The response minus the bias is linear in the input."""
    fails = []
    a, c = 0.75, -1.5
    x, D, codes, b = rand_conv_case(31, 1, 8, 7, 7, 4, 3, 3, 4, 16)
    x2 = _rng(32).standard_normal(x.shape)
    f = lambda z: o.conv_forward(z, D, codes, 3, 3, 1, 1, b) - b[None, :, None, None]
    lhs = f(a * x + c * x2)
    rhs = a * f(x) + c * f(x2)
    if relerr(lhs, rhs) > 1e-12:
        fails.append(f"conv linearity err {relerr(lhs, rhs)}")
    x, D, codes, b = rand_fc_case(33, 2, 16, 6, 4, 8)
    x2 = _rng(34).standard_normal(x.shape)
    g = lambda z: o.fc_forward(z, D, codes, b) - b
    if relerr(g(a * x + c * x2), a * g(x) + c * g(x2)) > 1e-12:
        fails.append("fc linearity")
    return fails


def pin_permutation(o):
    """Renumbering the sub-codewords of each sub-space (and the codes with
    them) leaves the response bit-identical."""
    fails = []
    r = _rng(41)
    x, D, codes, b = rand_conv_case(42, 1, 8, 6, 6, 5, 3, 3, 4, 12)
    M, K, _ = D.shape
    perm = np.stack([r.permutation(K) for _ in range(M)])   # new index of old k
    Dp = np.empty_like(D)
    for m in range(M):
        Dp[m, perm[m]] = D[m]
    cp = perm[np.arange(M)[None, None, :], codes.astype(np.int64)].astype(np.uint8)
    if not np.array_equal(o.conv_forward(x, D, codes, 3, 3, 1, 1, b),
                          o.conv_forward(x, Dp, cp, 3, 3, 1, 1, b)):
        fails.append("conv permutation")
    x, D, codes, b = rand_fc_case(43, 2, 12, 7, 3, 10)
    M, K, _ = D.shape
    perm = np.stack([r.permutation(K) for _ in range(M)])
    Dp = np.empty_like(D)
    for m in range(M):
        Dp[m, perm[m]] = D[m]
    cp = perm[np.arange(M)[:, None], codes.astype(np.int64)].astype(np.uint8)
    if not np.array_equal(o.fc_forward(x, D, codes, b), o.fc_forward(x, Dp, cp, b)):
        fails.append("fc permutation")
    return fails


def pin_k1_closed_form(o):
    """K = 1: every weight sub-vector is the single sub-codeword, so the FC
    response is <x, concat_m D[m, 0]> for every output (a textbook dot
    product) and the conv response is a conv with identical kernels."""
    fails = []
    r = _rng(51)
    x = r.standard_normal((3, 12))
    D = r.standard_normal((4, 1, 3))
    codes = np.zeros((4, 5), np.uint8)
    got = o.fc_forward(x, D, codes)
    ref = np.repeat((x @ D[:, 0, :].reshape(-1))[:, None], 5, axis=1)
    if relerr(got, ref) > 1e-12:
        fails.append("fc K=1")
    xc = r.standard_normal((1, 6, 5, 5))
    Dc = r.standard_normal((2, 1, 3))
    cc = np.zeros((3, 9, 2), np.uint8)
    got = o.conv_forward(xc, Dc, cc, 3, 3, 1, 1)
    # the same 3x3 kernel for every output channel: box-sum over the window of
    # the per-position dot product <x[:, p], concat_m D[m, 0]>
    v = np.einsum("nchw,c->nhw", xc, Dc[:, 0, :].reshape(-1))
    vp = np.pad(v, ((0, 0), (1, 1), (1, 1)))
    box = sum(vp[:, dy:dy + 5, dx:dx + 5] for dy in range(3) for dx in range(3))
    if relerr(got, np.repeat(box[:, None], 3, axis=1)) > 1e-12:
        fails.append("conv K=1")
    return fails


def pin_conv_fc_equivalence(o):
    """A 1x1 conv is the FC layer applied at every position, and an FC layer
    is a conv on a 1x1 map (Sec. 2: both are sums of inner products)."""
    fails = []
    r = _rng(61)
    N, Cs, H, W, Ct, Csp, K = 2, 12, 4, 5, 7, 3, 9
    M = Cs // Csp
    x = r.standard_normal((N, Cs, H, W))
    D = r.standard_normal((M, K, Csp))
    codes_fc = r.integers(0, K, (M, Ct), dtype=np.uint8)
    b = r.standard_normal(Ct)
    codes_conv = codes_fc.T.reshape(Ct, 1, M).copy()
    yc = o.conv_forward(x, D, codes_conv, 1, 1, 1, 0, b, True)
    yf = o.fc_forward(x.transpose(0, 2, 3, 1).reshape(-1, Cs), D, codes_fc, b, True)
    yf = yf.reshape(N, H, W, Ct).transpose(0, 3, 1, 2)
    if relerr(yc, yf) > 1e-13:
        fails.append("1x1 conv != fc per position")
    y1 = o.conv_forward(x[:, :, :1, :1], D, codes_conv, 1, 1, 1, 0, b)[:, :, 0, 0]
    y2 = o.fc_forward(x[:, :, 0, 0], D, codes_fc, b)
    if relerr(y1, y2) > 1e-13:
        fails.append("fc != conv on 1x1 map")
    return fails


def pin_lut_one_hot(o):
    """One-hot sub-codebooks D[m][k][j] = (k+1) [j == k mod Csp] turn the
    look-up table into scaled copies of single input channels:
    LUT[n, m, p, k] = (k+1) x[n, m*Csp + (k mod Csp), p]."""
    fails = []
    r = _rng(71)
    N, Cs, H, W, Csp, K = 2, 12, 3, 4, 4, 10
    M = Cs // Csp
    x = r.standard_normal((N, Cs, H, W))
    D = np.zeros((M, K, Csp))
    for k in range(K):
        D[:, k, k % Csp] = k + 1
    lut = o.conv_lut(x, D)
    xr = x.reshape(N, M, Csp, H * W)
    for k in range(K):
        if not np.array_equal(lut[:, :, :, k], (k + 1) * xr[:, :, k % Csp, :]):
            fails.append(f"conv lut one-hot k={k}")
            break
    xf = r.standard_normal((3, Cs))
    lf = o.fc_lut(xf, D)
    xfr = xf.reshape(3, M, Csp)
    for k in range(K):
        if not np.array_equal(lf[:, :, k], (k + 1) * xfr[:, :, k % Csp]):
            fails.append(f"fc lut one-hot k={k}")
            break
    return fails


def pin_maxpool(o):
    fails = []
    r = _rng(81)
    for (N, C, H, W, k, s) in [(2, 3, 9, 8, 3, 2), (1, 2, 13, 13, 3, 2), (1, 4, 8, 8, 2, 2),
                               (1, 1, 5, 7, 1, 1)]:
        x = r.standard_normal((N, C, H, W))
        ref = F.max_pool2d(torch.from_numpy(x), k, s).numpy()
        got = o.maxpool(x, k, s)
        if got.shape != ref.shape or not np.array_equal(got, ref):
            fails.append(f"maxpool {(N, C, H, W, k, s)}")
    return fails


def pin_tiny_net(o):
    """A conv -> pool -> conv -> FC -> FC stack equals the same stack built
    from torch's float64 conv2d / max_pool2d / linear with W_hat weights
    (flatten in C*H*W order)."""
    r = _rng(91)
    x = r.standard_normal((2, 6, 15, 15))
    spec = [("conv", 6, 8, 3, 3, 2, 1, 3, 7), ("pool", 3, 2),
            ("conv", 8, 6, 3, 3, 1, 1, 4, 16), ("fc", 6 * 3 * 3, 10, 3, 8, True),
            ("fc", 10, 5, 2, 4, False)]
    layers, h = [], torch.from_numpy(x)
    for t in spec:
        if t[0] == "conv":
            _, Cs, Ct, kh, kw, s, p, Csp, K = t
            D = r.standard_normal((Cs // Csp, K, Csp))
            c = r.integers(0, K, (Ct, kh * kw, Cs // Csp), dtype=np.uint8)
            b = r.standard_normal(Ct)
            layers.append(dict(kind="conv", D=D, codes=c, bias=b, kh=kh, kw=kw,
                               stride=s, pad=p, relu=True))
            h = F.relu(F.conv2d(h, torch.from_numpy(w_hat_conv(D, c, kh, kw)),
                                torch.from_numpy(b), stride=s, padding=p))
        elif t[0] == "pool":
            layers.append(dict(kind="maxpool", k=t[1], s=t[2]))
            h = F.max_pool2d(h, t[1], t[2])
        else:
            _, Cs, Ct, Csp, K, relu = t
            D = r.standard_normal((Cs // Csp, K, Csp))
            c = r.integers(0, K, (Cs // Csp, Ct), dtype=np.uint8)
            b = r.standard_normal(Ct)
            layers.append(dict(kind="fc", D=D, codes=c, bias=b, relu=relu))
            h = h.reshape(h.shape[0], -1) @ torch.from_numpy(w_hat_fc(D, c)).T + torch.from_numpy(b)
            if relu:
                h = F.relu(h)
    got = o.net_forward(x, layers)
    return [] if relerr(got, h.numpy()) < 1e-12 else [f"tiny net err {relerr(got, h.numpy())}"]


def torch_bf16(v):
    """torch's CPU float32 -> bfloat16 conversion (round to nearest even)."""
    t = torch.from_numpy(np.asarray(v, np.float32)).to(torch.bfloat16)
    return t.to(torch.float64).numpy()


def pin_bf16_rounding(o):
    """The bfloat16 rounding of the reduced-precision table model: equal to
    torch's float32 -> bfloat16 conversion on float32 values of every scale,
    and to hand-worked ties (8 significant bits, ties to even)."""
    fails = []
    r = _rng(31)
    v = (r.standard_normal(3000) * 2.0 ** r.integers(-40, 40, 3000)).astype(np.float32)
    v = np.concatenate([v, np.float32([0.0, 1.0, -1.0, 255.0, 1e30, -3e-30])])
    got, ref = o.round_bf16(v.astype(np.float64)), torch_bf16(v)
    if not np.array_equal(got, ref):
        bad = int(np.sum(got != ref))
        fails.append(f"{bad} values differ from torch's bfloat16 conversion")
    e8 = 2.0 ** -8
    worked = [
        (1 + e8, 1.0),                         # tie: 1 has an even last bit
        (1 + 3 * e8, 1 + 4 * e8),              # tie: 1 + 2^-7 has an odd last bit
        (-(1 + e8), -1.0),
        (1 + e8 + 2.0 ** -40, 1 + 2 * e8),     # just above the tie (not a float32)
        (257.0, 256.0), (259.0, 260.0), (258.0, 258.0),
        (0.1, 0.10009765625),                  # 0x3DCD
        (-1000.0, -1000.0), (1001.0, 1000.0), (1003.0, 1004.0),
    ]
    for x, want in worked:
        g = float(o.round_bf16(np.float64([x]))[0])
        if g != want:
            fails.append(f"round_bf16({x!r}) = {g!r}, expected {want!r}")
    return fails


def pin_bf16_tables(o):
    """Reduced-precision tables, on integer data whose table entries (up to a
    few thousand) are exact in double and in float32 but not in bfloat16:
    the FC response must equal (rounded tables) @ (one-hot code matrix) and the
    conv response a float64 conv2d of the rounded table maps with one-hot
    code kernels (Eq. 7 read as a convolution over the (m, k) table
    channels); tables built by torch, rounded by torch."""
    fails = []
    r = _rng(37)
    for (N, Cs, Ct, Csp, K) in [(3, 24, 7, 4, 16), (2, 16, 5, 8, 3)]:
        M = Cs // Csp
        x = r.integers(-20, 21, (N, Cs)).astype(np.float64)
        D = r.integers(-20, 21, (M, K, Csp)).astype(np.float64)
        codes = r.integers(0, K, (M, Ct), dtype=np.uint8)
        T = torch.einsum("nmj,mkj->nmk", torch.from_numpy(x.reshape(N, M, Csp)),
                         torch.from_numpy(D)).numpy()
        Tr = torch_bf16(T)
        if np.array_equal(Tr, T):
            fails.append("test data too small to exercise rounding")
        onehot = np.zeros((M, K, Ct))
        onehot[np.arange(M)[:, None], codes.astype(np.int64), np.arange(Ct)[None, :]] = 1.0
        ref = Tr.reshape(N, M * K) @ onehot.reshape(M * K, Ct)
        got = o.fc_forward(x, D, codes, lut_bf16=True)
        if not np.array_equal(got, ref):
            fails.append(f"fc bf16 tables: err {relerr(got, ref)}")
    for (N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K) in [
            (2, 8, 6, 7, 3, 3, 3, 1, 1, 4, 6), (1, 6, 9, 8, 2, 5, 3, 2, 2, 3, 5)]:
        M = Cs // Csp
        x = r.integers(-20, 21, (N, Cs, H, W)).astype(np.float64)
        D = r.integers(-20, 21, (M, K, Csp)).astype(np.float64)
        codes = r.integers(0, K, (Ct, kh * kw, M), dtype=np.uint8)
        T = torch.einsum("nmjhw,mkj->nmkhw",
                         torch.from_numpy(x.reshape(N, M, Csp, H, W)),
                         torch.from_numpy(D)).numpy()
        Tr = torch_bf16(T).reshape(N, M * K, H, W)
        Wk = np.zeros((Ct, M, K, kh * kw))
        ct_i, pk_i, m_i = np.meshgrid(np.arange(Ct), np.arange(kh * kw), np.arange(M),
                                      indexing="ij")
        Wk[ct_i, m_i, codes.astype(np.int64), pk_i] = 1.0
        Wk = Wk.reshape(Ct, M * K, kh, kw)
        ref = F.conv2d(torch.from_numpy(Tr), torch.from_numpy(Wk), stride=stride,
                       padding=pad).numpy()
        got = o.conv_forward(x, D, codes, kh, kw, stride, pad, lut_bf16=True)
        if got.shape != ref.shape or not np.array_equal(got, ref):
            fails.append(f"conv bf16 tables: err {relerr(got, ref)}")
    return fails


# ----------------------------------------------------------- quantizer
def _clustered(seed, K, d, per, spread=10.0, noise=0.3):
    """K well-separated centres on a grid, `per` points each (shuffled)."""
    r = _rng(seed)
    grid = np.stack(np.meshgrid(*[np.arange(3)] * d, indexing="ij"), -1).reshape(-1, d)
    centres = grid[r.choice(len(grid), K, replace=False)] * spread
    labels = np.repeat(np.arange(K), per)
    pts = centres[labels] + r.uniform(-noise, noise, (K * per, d))
    order = r.permutation(K * per)
    return pts[order].astype(np.float32), labels[order]


def pin_kmeans_separated(o):
    """Well-separated clusters: from one point of each cluster, Lloyd's
    iterations find the true labels and each centroid is its cluster's mean."""
    fails = []
    for d, K in [(4, 16), (3, 9), (8, 5)]:
        pts, labels = _clustered(41 + d, K, d, 37)
        first = np.array([np.flatnonzero(labels == k)[0] for k in range(K)])
        for iters in (1, 3):
            cen, a = o.kmeans(pts, pts[first], iters)
            if not np.array_equal(a, labels.astype(np.uint8)):
                fails.append(f"d={d} K={K} iters={iters}: labels not recovered")
                continue
            want = np.stack([pts[labels == k].astype(np.float64).mean(0) for k in range(K)])
            if np.max(np.abs(cen - want)) > 1e-6 * np.max(np.abs(want)):
                fails.append(f"d={d} K={K} iters={iters}: centroids are not the cluster means")
        # a duplicated initial centroid: exact distance ties go to the first
        # index, and the copy, left without points, keeps its value
        init = np.concatenate([pts[first], pts[first[:1]]])
        _, a0 = o.kmeans(pts, init, 0)          # assignment to the initial centroids
        cen1, _ = o.kmeans(pts, init, 1)        # one round: the copy had no points
        if not np.array_equal(a0, labels.astype(np.uint8)):
            fails.append(f"d={d} K={K}: an exact distance tie did not go to the first index")
        if not np.array_equal(cen1[K], init[K]):
            fails.append(f"d={d} K={K}: a centroid without points did not keep its value")
    return fails


def pin_kmeans_scipy(o):
    """Lloyd's algorithm as scipy runs it (kmeans2 with a given initial
    codebook, float64): same centroids after T rounds, and the same final
    assignment as scipy's vq against them, on points whose nearest and
    second-nearest centroids are not near-tied."""
    import warnings

    from scipy.cluster import vq as spvq
    fails = []
    r = _rng(43)
    for (P, d, K, T) in [(600, 4, 8, 3), (400, 3, 16, 4), (300, 8, 4, 2), (64, 2, 256, 1)]:
        pts = r.standard_normal((P, d)).astype(np.float32)
        init = pts[r.choice(P, K, replace=K > P)] if K <= P else \
            r.standard_normal((K, d)).astype(np.float32)
        with warnings.catch_warnings():
            warnings.simplefilter("ignore")  # empty clusters keep their centroid
            ref_cb, _ = spvq.kmeans2(pts.astype(np.float64), init.astype(np.float64), iter=T,
                                     minit="matrix", missing="warn")
        ref_a, _ = spvq.vq(pts.astype(np.float64), ref_cb)
        cen, a = o.kmeans(pts, init, T)
        if np.max(np.abs(cen - ref_cb)) > 1e-6 * max(1.0, np.max(np.abs(ref_cb))):
            fails.append(f"P={P} d={d} K={K} T={T}: centroids differ from scipy")
            continue
        dist = ((pts[:, None, :].astype(np.float64) - ref_cb[None]) ** 2).sum(-1)
        two = np.sort(dist, axis=1)[:, :2]
        clear = two[:, 1] - two[:, 0] > 1e-4 * (1 + two[:, 1])
        if np.mean(clear) < 0.95 or not np.array_equal(a[clear], ref_a[clear]):
            fails.append(f"P={P} d={d} K={K} T={T}: assignment differs from scipy")
    return fails


def pin_kmeans_distortion_monotone(o):
    """Each Lloyd round can only lower sum ||x - c(x)||^2."""
    r = _rng(47)
    pts = r.standard_normal((500, 4)).astype(np.float32)
    init = pts[:32]
    prev, fails = np.inf, []
    for T in range(6):
        cen, a = o.kmeans(pts, init, T)
        dist = float(((pts.astype(np.float64) - cen[a].astype(np.float64)) ** 2).sum())
        if dist > prev * (1 + 1e-9):
            fails.append(f"distortion rose at T={T}: {dist} > {prev}")
        prev = dist
    return fails


def pin_pq_quantize_exact(o):
    """Eq. 4 / Eq. 6 solved with zero error: a dense W whose sub-vectors are
    drawn from K prototypes per sub-space.  Started from the prototypes, the
    quantizer returns them and the codes W was built from; the PQ response
    then equals the dense conv / FC of W (torch)."""
    fails = []
    r = _rng(53)
    for (Ct, Cs, kh, kw, Csp, K) in [(12, 8, 3, 3, 4, 16), (7, 6, 1, 2, 3, 5), (5, 16, 2, 2, 8, 8)]:
        M = Cs // Csp
        D0 = r.standard_normal((M, K, Csp)).astype(np.float32)
        c0 = r.integers(0, K, (Ct, kh * kw, M), dtype=np.uint8)
        c0[:K, 0, :] = np.arange(K)[:, None] % K if Ct >= K else c0[:K, 0, :]
        W = w_hat_conv(D0, c0, kh, kw).astype(np.float32)
        D, codes = o.pq_quantize_conv(W, Csp, K, D0, 2)
        used = np.zeros((M, K), bool)
        used[np.arange(M)[None, None, :], c0.astype(np.int64)] = True
        if not np.array_equal(codes, c0) or not np.array_equal(D[used], D0[used]):
            fails.append(f"conv {Ct}x{Cs}x{kh}x{kw}: prototypes/codes not recovered")
            continue
        x = r.standard_normal((1, Cs, 6, 7))
        got = o.conv_forward(x, D, codes, kh, kw, 1, 1)
        ref = torch_conv(x, W.astype(np.float64), None, 1, 1, False)
        if relerr(got, ref) > 1e-12:
            fails.append(f"conv {Ct}x{Cs}: response differs from the dense conv")
    for (Ct, Cs, Csp, K) in [(40, 12, 4, 8), (33, 16, 2, 32)]:
        M = Cs // Csp
        D0 = r.standard_normal((M, K, Csp)).astype(np.float32)
        c0 = r.integers(0, K, (M, Ct), dtype=np.uint8)
        W = w_hat_fc(D0, c0).astype(np.float32)
        D, codes = o.pq_quantize_fc(W, Csp, K, D0, 2)
        used = np.zeros((M, K), bool)
        used[np.arange(M)[:, None], c0.astype(np.int64)] = True
        if not np.array_equal(codes, c0) or not np.array_equal(D[used], D0[used]):
            fails.append(f"fc {Ct}x{Cs}: prototypes/codes not recovered")
            continue
        x = r.standard_normal((3, Cs))
        if relerr(o.fc_forward(x, D, codes), torch_fc(x, W.astype(np.float64), None, False)) > 1e-12:
            fails.append(f"fc {Ct}x{Cs}: response differs from the dense FC")
    return fails


def pin_pq_quantize_conv_1x1_is_fc(o):
    """A 1x1 conv kernel set quantizes like the FC matrix it equals."""
    r = _rng(59)
    Ct, Cs, Csp, K = 50, 12, 3, 8
    W = r.standard_normal((Ct, Cs)).astype(np.float32)
    init = r.standard_normal((Cs // Csp, K, Csp)).astype(np.float32)
    Dc, cc = o.pq_quantize_conv(W[:, :, None, None], Csp, K, init, 3)
    Df, cf = o.pq_quantize_fc(W, Csp, K, init, 3)
    if not (np.array_equal(Dc, Df) and np.array_equal(cc[:, 0, :].T, cf)):
        return ["1x1 conv quantization differs from the FC quantization"]
    return []


# ---------------------------------------------------------------- bit codes
def pin_bits(o):
    """Bit packing (oracle/bits.py) against hand-worked streams, numpy's
    little-endian packbits of the bit expansion, and the round trip."""
    from oracle import bits
    fails = []
    worked = [
        (([1, 2, 3], 2), bytes([0b00111001])),           # 01 | 10 | 11, LSB first
        (([5, 31, 0, 17], 5), bytes([0xE5, 0x83, 0x08])),  # 17 -> stream bits 15 and 19
        (([255, 1], 8), bytes([255, 1])),
        (([1, 0, 1, 1, 0, 0, 0, 1, 1], 1), bytes([0b10001101, 0b1])),
        (([7, 7, 7], 3), bytes([0xFF, 0x01])),
    ]
    for (codes, b), want in worked:
        if bits.pack(codes, b) != want:
            fails.append(f"pack({codes}, {b}) = {bits.pack(codes, b).hex()}, want {want.hex()}")
    if [bits.bits_for(K) for K in (1, 2, 3, 4, 5, 16, 17, 32, 128, 129, 256)] != \
            [1, 1, 2, 2, 3, 4, 5, 5, 7, 8, 8]:
        fails.append("bits_for")
    r = _rng(83)
    for b in range(1, 9):
        c = r.integers(0, 1 << b, 1000)
        expand = ((c[:, None] >> np.arange(b)[None, :]) & 1).astype(np.uint8).ravel()
        ref = np.packbits(expand, bitorder="little").tobytes()
        got = bits.pack(c, b)
        if got != ref:
            fails.append(f"b={b}: differs from numpy packbits")
        if not np.array_equal(bits.unpack(got, len(c), b), c.astype(np.uint8)):
            fails.append(f"b={b}: round trip")
    return fails


ALL_PINS = [pin_conv_vs_dense, pin_fc_vs_dense, pin_integer_exact, pin_exactness,
            pin_linearity, pin_permutation, pin_k1_closed_form, pin_conv_fc_equivalence,
            pin_lut_one_hot, pin_maxpool, pin_tiny_net, pin_bf16_rounding, pin_bf16_tables,
            pin_kmeans_separated, pin_kmeans_scipy, pin_kmeans_distortion_monotone,
            pin_pq_quantize_exact, pin_pq_quantize_conv_1x1_is_fc, pin_bits]


def run_all(o):
    fails = []
    for p in ALL_PINS:
        try:
            fails += [f"{p.__name__}: {m}" for m in p(o)]
        except Exception as e:  # a crash inside a pin also counts as caught
            fails.append(f"{p.__name__}: raised {type(e).__name__}: {e}")
    return fails
