"""Pins for the error-corrected FC quantizer oracle (oracle/ec.py, Eq. 8 - 12).

Independent routes:
  * single-step ground truth: for one sub-space the D update is checked
    against numpy's lstsq on the stacked system (every (n, c_t in L_k) pair a
    row) and the B update against a brute-force evaluation of
    sum_n [R_n(c_t) - D_k^T S_n]^2 for every k -- neither goes through the
    oracle's Gram-matrix form;
  * two sub-spaces, one sweep, replayed with those primitives and residuals
    built from the dense response (torch matmul of W_hat, Eq. 4);
  * block coordinate descent never raises the objective (Eq. 8, evaluated
    through W_hat and torch);
  * zero-error data (T made by a PQ layer) is a fixed point;
  * identity inputs (S = I, T = W^T) turn the objective into the k-means
    objective of Eq. 4: one alternation equals one k-means round of the C
    oracle.
Every pin takes the EC module and the C oracle and returns failure messages.
"""
from __future__ import annotations

import numpy as np
import torch

from pins import _clustered, relerr, w_hat_fc


def _dense_response(S, D, codes):
    W = w_hat_fc(np.asarray(D, np.float64), codes)          # [Ct, Cs]
    return (torch.from_numpy(np.asarray(S, np.float64)) @ torch.from_numpy(W).T).numpy()


def _problem(seed, N, Cs, Ct, Csp, K):
    r = np.random.default_rng(seed)
    M = Cs // Csp
    S = r.standard_normal((N, Cs))
    Wt = r.standard_normal((Ct, Cs)) * 0.3
    T = S @ Wt.T
    D0 = r.standard_normal((M, K, Csp)) * 0.3
    c0 = r.integers(0, K, (M, Ct)).astype(np.uint8)
    return S, T, D0, c0


def _lstsq_codeword(A, R, cts):
    rows = np.concatenate([A] * len(cts))
    rhs = np.concatenate([R[:, c] for c in cts])
    return np.linalg.lstsq(rows, rhs, rcond=None)[0]


def _bruteforce_assign(A, R, Dm):
    err = np.stack([((R - (A @ Dm[k])[:, None]) ** 2).sum(0) for k in range(len(Dm))])
    return np.argmin(err, axis=0), np.sort(err, axis=0)


def pin_ec_single_subspace(ec, o):
    """M = 1: R = T.  One alternation = least squares per codeword, then the
    brute-force best codeword per output."""
    fails = []
    for (N, Csp, Ct, K) in [(40, 3, 30, 5), (25, 4, 17, 8), (12, 1, 9, 3)]:
        S, T, D0, c0 = _problem(61 + N, N, Csp, Ct, Csp, K)
        D, codes = ec.ec_quantize_fc(S, T, D0, c0, 1, 1)
        want = D0[0].copy()
        for k in range(K):
            cts = np.flatnonzero(c0[0] == k)
            if cts.size:
                want[k] = _lstsq_codeword(S, T, cts)
        if np.max(np.abs(D[0] - want)) > 1e-9 * max(1.0, np.max(np.abs(want))):
            fails.append(f"N={N}: D update is not the per-codeword least-squares solution")
            continue
        best, _ = _bruteforce_assign(S, T, want)
        if not np.array_equal(codes[0], best):
            fails.append(f"N={N}: B update is not the best codeword per output")
    return fails


def pin_ec_two_subspaces_replayed(ec, o):
    """M = 2, one sweep, two alternations: replay Eq. 9 - 12 with lstsq, brute
    force and residuals from the dense response of the current parameters."""
    S, T, D0, c0 = _problem(67, 50, 6, 14, 3, 4)
    D, codes = ec.ec_quantize_fc(S, T, D0, c0, 1, 2)
    Dw, cw = D0.copy(), c0.copy()
    for m in range(2):
        A = S[:, 3 * m:3 * m + 3]
        mine = (torch.from_numpy(A) @ torch.from_numpy(Dw[m][cw[m]]).T).numpy()
        R = T - (_dense_response(S, Dw, cw) - mine)        # Eq. 9
        for _ in range(2):
            for k in range(4):
                cts = np.flatnonzero(cw[m] == k)
                if cts.size:
                    Dw[m, k] = _lstsq_codeword(A, R, cts)
            cw[m], _ = _bruteforce_assign(A, R, Dw[m])
    if not np.array_equal(codes, cw) or np.max(np.abs(D - Dw)) > 1e-9:
        return ["two-sub-space sweep differs from the replayed block coordinate descent"]
    return []


def pin_ec_monotone(ec, o):
    """Each sub-space step can only lower the Eq. 8 objective (checked through
    the dense response), and the oracle's own objective agrees with it."""
    S, T, D0, c0 = _problem(71, 80, 16, 24, 4, 8)
    trace = []
    D, codes = ec.ec_quantize_fc(S, T, D0, c0, 2, 2, trace=trace)
    dense = float(np.sum((T - _dense_response(S, D, codes)) ** 2))
    fails = []
    start = float(np.sum((T - _dense_response(S, D0, c0)) ** 2))
    seq = [start] + trace
    if any(b > a * (1 + 1e-12) for a, b in zip(seq, seq[1:])):
        fails.append("objective rose during block coordinate descent")
    if abs(dense - trace[-1]) > 1e-9 * max(1.0, dense):
        fails.append("objective disagrees with the dense response")
    return fails


def pin_ec_fixed_point(ec, o):
    """T produced by a PQ layer (zero error): its parameters stay put."""
    r = np.random.default_rng(73)
    N, Cs, Ct, Csp, K = 60, 12, 20, 4, 6
    M = Cs // Csp
    S = r.standard_normal((N, Cs))
    D0 = r.standard_normal((M, K, Csp))
    c0 = r.integers(0, K, (M, Ct)).astype(np.uint8)
    for m in range(M):
        c0[m, :K] = np.arange(K)        # every codeword used
    T = _dense_response(S, D0, c0)
    D, codes = ec.ec_quantize_fc(S, T, D0, c0, 2, 2)
    if not np.array_equal(codes, c0) or np.max(np.abs(D - D0)) > 1e-9:
        return ["zero-error parameters moved"]
    return []


def pin_ec_identity_is_kmeans(ec, o):
    """S = I, T = W^T: the Eq. 8 objective becomes ||W - W_hat||_F^2 (Eq. 4),
    G = I, U = the sub-vectors.  From codes that assign every sub-vector to
    its nearest initial centroid, one alternation (D update, B update) is one
    k-means round of the C oracle (centroid means, then nearest centroid)."""
    fails = []
    for (d, K) in [(4, 8), (3, 6)]:
        pts, labels = _clustered(79 + d, K, d, 9)            # [P, d] sub-vectors of one sub-space
        P = len(pts)
        W = pts.astype(np.float64)                           # Ct = P weight vectors, Cs = d (M = 1)
        init = pts[[np.flatnonzero(labels == k)[0] for k in range(K)]][::-1].copy()
        _, a0 = o.kmeans(pts, init, 0)
        cen1, a1 = o.kmeans(pts, init, 1)
        D, codes = ec.ec_quantize_fc(np.eye(d), W.T.copy(), init[None].astype(np.float64),
                                     a0[None], 1, 1)
        if not np.array_equal(codes[0], a1) or np.max(np.abs(D[0] - cen1)) > 1e-6:
            fails.append(f"d={d}: S = I alternation differs from a k-means round")
    return fails


ALL_EC_PINS = [pin_ec_single_subspace, pin_ec_two_subspaces_replayed, pin_ec_monotone,
               pin_ec_fixed_point, pin_ec_identity_is_kmeans]


def run_all(ec, o):
    fails = []
    for p in ALL_EC_PINS:
        try:
            fails += [f"{p.__name__}: {m}" for m in p(ec, o)]
        except Exception as e:  # a crash inside a pin also counts as caught
            fails.append(f"{p.__name__}: raised {type(e).__name__}: {e}")
    return fails
