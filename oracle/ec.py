"""Error-corrected quantization of an FC layer (Sec. 3.3.1, Eq. 8 - 12), float64.

TEST INFRASTRUCTURE ONLY (see the package docstring): plain numpy, one step
per line of the method, written to be read against the paper.

Objective (Eq. 8), with S_n the layer input and T_n the desired response of
calibration vector n:
    min_{D, B} sum_n || T_n - sum_m (D^(m) B^(m))^T S_n^(m) ||^2
Block coordinate descent over the sub-spaces m, in order; for sub-space m the
residual with its own term removed (Eq. 9)
    R_n^(m) = T_n - sum_{m' != m} (D^(m') B^(m'))^T S_n^(m')
is fixed while D^(m) and B^(m) are updated alternately (Eq. 10):
  * D update (Eq. 11): with the assignment fixed, L_k = {c_t : k(c_t) = k}
    and each sub-codeword solves its own least-squares problem
        min_{D_k} sum_n sum_{c_t in L_k} [R_n(c_t) - D_k^T S_n^(m)]^2,
    whose normal equations are  G D_k = mean_{c_t in L_k} U[:, c_t]  with
    G = sum_n S_n S_n^T and U = sum_n S_n R_n^T (C'_s x C_t);
  * B update (Eq. 12): k(c_t) = argmin_k sum_n [R_n(c_t) - D_k^T S_n]^2,
    i.e. argmin_k (D_k^T G D_k - 2 D_k^T U[:, c_t]) (the dropped term does
    not depend on k).
Readings (the paper leaves them open):
  * the initial D and codes are inputs (e.g. the plain k-means result);
  * `outer` sweeps over m = 0 .. M-1, `inner` alternations per sub-space,
    each a D update followed by a B update (the order the paper lists);
  * a sub-codeword whose L_k is empty keeps its value;
  * G is solved by Cholesky; calibration data with rank-deficient G
    (fewer than C'_s independent sub-vectors) is rejected;
  * argmin ties go to the smallest k.
Layouts: S [N, Cs], T [N, Ct], D [M, K, Csp], codes [M, Ct] (as qcnn_fc_forward).
"""
from __future__ import annotations

import numpy as np


class ECError(ValueError):
    pass


def _approx_response(S, D, codes):
    """sum_m (D^(m) B^(m))^T S_n^(m) for every n: [N, Ct]."""
    N, Cs = S.shape
    M, K, Csp = D.shape
    Y = np.zeros((N, codes.shape[1]))
    for m in range(M):
        A = S[:, m * Csp:(m + 1) * Csp]           # S^(m): [N, Csp]
        Y += A @ D[m][codes[m]].T                  # D^(m) B^(m) picks D_k(c_t) per column
    return Y


def objective(S, T, D, codes):
    """Eq. 8: sum_n ||T_n - approx_n||^2."""
    S = np.asarray(S, np.float64)
    T = np.asarray(T, np.float64)
    return float(np.sum((T - _approx_response(S, np.asarray(D, np.float64), codes)) ** 2))


def _cholesky_solve(G, b):
    L = np.linalg.cholesky(G)                      # raises on a non-SPD G
    y = np.linalg.solve(L, b)
    return np.linalg.solve(L.T, y)


def ec_quantize_fc(S, T, D0, codes0, outer, inner, trace=None):
    """Returns (D [M, K, Csp] float64, codes [M, Ct] uint8).  `trace`, if a
    list, receives the objective after every sub-space step."""
    S = np.asarray(S, np.float64)
    T = np.asarray(T, np.float64)
    D = np.array(D0, np.float64)
    codes = np.array(codes0, np.uint8)
    N, Cs = S.shape
    M, K, Csp = D.shape
    Ct = codes.shape[1]
    if M * Csp != Cs or T.shape != (N, Ct) or codes.shape != (M, Ct):
        raise ECError("shape mismatch")
    if np.any(codes >= K):
        raise ECError("code >= K")
    E = T - _approx_response(S, D, codes)          # residual of the whole approximation
    for _ in range(outer):
        for m in range(M):
            A = S[:, m * Csp:(m + 1) * Csp]
            old = D[m][codes[m]].copy()            # [Ct, Csp]: this sub-space's terms
            R = E + A @ old.T                      # Eq. 9
            G = A.T @ A
            try:
                np.linalg.cholesky(G)
            except np.linalg.LinAlgError:
                raise ECError(f"sub-space {m}: calibration data is rank deficient")
            U = A.T @ R                            # [Csp, Ct]
            for _ in range(inner):
                for k in range(K):                 # Eq. 11, one least-squares problem per k
                    Lk = np.flatnonzero(codes[m] == k)
                    if Lk.size:
                        D[m, k] = _cholesky_solve(G, U[:, Lk].mean(axis=1))
                cost = np.einsum("kj,ji,ki->k", D[m], G, D[m])[:, None] - 2.0 * (D[m] @ U)
                codes[m] = np.argmin(cost, axis=0)  # Eq. 12; first index on ties
            E = R - A @ D[m][codes[m]].T
            if trace is not None:
                trace.append(objective(S, T, D, codes))
    return D, codes
