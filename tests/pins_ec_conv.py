"""Pins for the error-corrected conv quantizer oracle (oracle/ec_conv.py,
Appendix B).

Independent routes (none goes through the oracle's shifted-view einsums):
  * dense responses: torch float64 conv2d of W_hat (Eq. 6 meaning of the
    codes), and of W_hat restricted to one codeword's (c_t, p_k) entries;
  * Z_k by conv2d of each input channel of the sub-space with the 0/1 mask
    of the offsets assigned to k, and the codeword update by numpy lstsq on
    the stacked rows;
  * the assignment update by trying every codeword at (c_t, p_k) and
    evaluating the whole objective through the dense response;
  * block coordinate descent never raises the objective, zero-error data is
    a fixed point, and a 1x1 conv is the FC layer applied at every position
    (so its error correction equals oracle/ec.py on the flattened samples).
"""
from __future__ import annotations

import numpy as np
import torch
import torch.nn.functional as F

from pins import w_hat_conv


def dense(S, D, codes, kh, kw, stride, pad):
    W = w_hat_conv(np.asarray(D, np.float64), codes, kh, kw)
    return F.conv2d(torch.from_numpy(np.asarray(S, np.float64)), torch.from_numpy(W),
                    stride=stride, padding=pad).numpy()


def dense_obj(S, T, D, codes, kh, kw, stride, pad):
    return float(np.sum((T - dense(S, D, codes, kh, kw, stride, pad)) ** 2))


def _problem(seed, N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K):
    r = np.random.default_rng(seed)
    M = Cs // Csp
    S = r.standard_normal((N, Cs, H, W))
    Wt = r.standard_normal((Ct, Cs, kh, kw)) * 0.3
    T = F.conv2d(torch.from_numpy(S), torch.from_numpy(Wt), stride=stride, padding=pad).numpy()
    D0 = r.standard_normal((M, K, Csp)) * 0.3
    c0 = r.integers(0, K, (Ct, kh * kw, M)).astype(np.uint8)
    return S, T, D0, c0


def _z(S, m, Csp, mask, kh, kw, stride, pad):
    """Z[n, c_t, j, p_t] = sum over offsets p_k with mask[c_t, p_k] of the
    input sub-vector at p_s(p_t, p_k), by conv2d."""
    Ct = mask.shape[0]
    Wm = torch.from_numpy(mask.reshape(Ct, 1, kh, kw).astype(np.float64))
    cols = [F.conv2d(torch.from_numpy(S[:, m * Csp + j:m * Csp + j + 1]), Wm, stride=stride,
                     padding=pad).numpy() for j in range(Csp)]
    return np.stack(cols, axis=2)                       # [N, Ct, Csp, Ho, Wo]


def _replay(S, T, D0, c0, kh, kw, stride, pad, inner):
    """One sweep of Appendix B replayed with the independent primitives."""
    D, codes = D0.copy(), c0.copy()
    M, K, Csp = D.shape
    Ct, kk, _ = codes.shape
    for m in range(M):
        for _ in range(inner):
            for k in range(K):
                mask = (codes[:, :, m] == k)
                if not mask.any():
                    continue
                Z = _z(S, m, Csp, mask.astype(np.float64), kh, kw, stride, pad)
                # Q_k: T minus everything but codeword k of sub-space m
                Dk0 = D.copy()
                Dk0[m, k] = 0.0
                Q = T - dense(S, Dk0, codes, kh, kw, stride, pad)
                rows = Z.transpose(0, 1, 3, 4, 2).reshape(-1, Csp)
                D[m, k] = np.linalg.lstsq(rows, Q.reshape(-1), rcond=None)[0]
            for pk in range(kk):
                for ct in range(Ct):
                    best, best_e = 0, None
                    for k in range(K):
                        trial = codes.copy()
                        trial[ct, pk, m] = k
                        e = dense_obj(S, T, D, trial, kh, kw, stride, pad)
                        if best_e is None or e < best_e * (1 - 1e-12):
                            best, best_e = k, e
                    codes[ct, pk, m] = best
    return D, codes


def pin_ecc_replayed(ecc, ec):
    """Two sub-spaces, one sweep: the oracle equals the replay."""
    fails = []
    for (N, Cs, H, W, Ct, kh, kw, s, p, Csp, K, inner) in [
            (2, 4, 5, 6, 3, 2, 2, 1, 1, 2, 3, 1),
            (2, 6, 7, 5, 2, 3, 3, 2, 1, 3, 4, 2)]:
        S, T, D0, c0 = _problem(89 + H, N, Cs, H, W, Ct, kh, kw, s, p, Csp, K)
        D, codes = ecc.ec_quantize_conv(S, T, D0, c0, kh, kw, s, p, 1, inner)
        Dr, cr = _replay(S, T, D0, c0, kh, kw, s, p, inner)
        if not np.array_equal(codes, cr) or np.max(np.abs(D - Dr)) > 1e-8:
            fails.append(f"{(N, Cs, H, W, Ct, kh, kw, s, p)}: differs from the replay")
    return fails


def pin_ecc_monotone(ecc, ec):
    S, T, D0, c0 = _problem(97, 3, 8, 7, 7, 6, 3, 3, 1, 1, 4, 8)
    trace = []
    D, codes = ecc.ec_quantize_conv(S, T, D0, c0, 3, 3, 1, 1, 2, 2, trace=trace)
    seq = [dense_obj(S, T, D0, c0, 3, 3, 1, 1)] + trace
    fails = []
    if any(b > a * (1 + 1e-12) for a, b in zip(seq, seq[1:])):
        fails.append("objective rose during block coordinate descent")
    if abs(dense_obj(S, T, D, codes, 3, 3, 1, 1) - trace[-1]) > 1e-9 * max(1.0, trace[-1]):
        fails.append("objective disagrees with the dense response")
    return fails


def pin_ecc_fixed_point(ecc, ec):
    r = np.random.default_rng(101)
    N, Cs, H, W, Ct, kh, kw, Csp, K = 2, 6, 6, 6, 5, 3, 3, 3, 4
    M = Cs // Csp
    S = r.standard_normal((N, Cs, H, W))
    D0 = r.standard_normal((M, K, Csp))
    c0 = r.integers(0, K, (Ct, kh * kw, M)).astype(np.uint8)
    c0[0, :K, :] = np.arange(K)[:, None]                 # every codeword used
    T = dense(S, D0, c0, kh, kw, 1, 1)
    D, codes = ecc.ec_quantize_conv(S, T, D0, c0, kh, kw, 1, 1, 1, 2)
    if not np.array_equal(codes, c0) or np.max(np.abs(D - D0)) > 1e-9:
        return ["zero-error parameters moved"]
    return []


def pin_ecc_1x1_is_fc(ecc, ec):
    """A 1x1 conv is the FC layer at every position: error correction on the
    maps equals the FC error correction on the flattened (n, y, x) samples."""
    r = np.random.default_rng(103)
    N, Cs, H, W, Ct, Csp, K = 2, 8, 5, 4, 9, 4, 5
    M = Cs // Csp
    S = r.standard_normal((N, Cs, H, W))
    T = r.standard_normal((N, Ct, H, W))
    D0 = r.standard_normal((M, K, Csp))
    c0 = r.integers(0, K, (Ct, 1, M)).astype(np.uint8)
    D, codes = ecc.ec_quantize_conv(S, T, D0, c0, 1, 1, 1, 0, 2, 2)
    Sf = S.transpose(0, 2, 3, 1).reshape(-1, Cs)
    Tf = T.transpose(0, 2, 3, 1).reshape(-1, Ct)
    Df, cf = ec.ec_quantize_fc(Sf, Tf, D0, c0[:, 0, :].T.copy(), 2, 2)
    if not np.array_equal(codes[:, 0, :].T, cf) or np.max(np.abs(D - Df)) > 1e-9:
        return ["1x1 conv error correction differs from the FC one"]
    return []


ALL_ECC_PINS = [pin_ecc_replayed, pin_ecc_monotone, pin_ecc_fixed_point, pin_ecc_1x1_is_fc]


def run_all(ecc, ec):
    fails = []
    for p in ALL_ECC_PINS:
        try:
            fails += [f"{p.__name__}: {m}" for m in p(ecc, ec)]
        except Exception as e:
            fails.append(f"{p.__name__}: raised {type(e).__name__}: {e}")
    return fails
