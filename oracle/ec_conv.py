"""Error-corrected quantization of a conv layer (Sec. 3.3.2, Appendix B), float64.

TEST INFRASTRUCTURE ONLY (see the package docstring): plain numpy, one step
per line of the method, written to be read against the paper.

Objective (Eq. B.1), S_n the layer input and T_n the desired response:
    min_{D, B} sum_{n, p_t} || sum_{(p_k, p_s)} sum_m (D^(m) B_pk^(m))^T S_{n,p_s}^(m)
                               - T_{n,p_t} ||^2
Block coordinate descent over the sub-spaces m, in order.  For sub-space m,
R = T - (every other sub-space's contribution) (Eq. B.2) is fixed, and
`inner` alternations run, each
  * D update: the sub-codewords one after another, k = 0 .. K-1.  With every
    other codeword of the sub-space in place, codeword k explains what is
    left (Q_k, Eq. B.5): its contribution to output (n, c_t, p_t) is
    D_k^T Z_k(n, c_t, p_t), Z_k the sum of the input sub-vectors at the
    offsets p_k with k(c_t, p_k) = k; D_k solves the least-squares problem
    of Eq. B.6 through its normal equations (sum Z Z^T) D_k = sum Z Q_k;
  * B update: the kernel offsets one after another, p_k = 0 .. kh*kw-1.
    With the other offsets' contributions in place, the residual P (Eq. B.7)
    is explained by offset p_k alone, and each output channel takes the
    codeword that minimises sum_{n,p_t} (D_k^T S_{n,p_s(p_t,p_k)} - P)^2
    (Eq. B.8), i.e. argmin_k D_k^T G D_k - 2 D_k^T U[:, c_t] with
    G = sum S S^T and U = sum S P^T over (n, p_t).
Readings (the paper leaves them open):
  * initial D and codes are inputs; `outer` sweeps over m = 0 .. M-1;
  * in an alternation the D update comes first, as the paper lists it;
  * T is the response before the bias (the bias is not quantized);
  * positions outside the input map contribute zero (zero padding), as in
    the forward response;
  * a codeword with no (c_t, p_k) assigned keeps its value; a singular
    least-squares problem with some terms, or a singular G, is rejected;
  * argmin ties go to the smallest k.
Layouts: S [N, Cs, H, W], T [N, Ct, Ho, Wo], D [M, K, Csp], codes
[Ct, kh*kw, M] (the layouts of qcnn_conv_forward).
"""
from __future__ import annotations

import numpy as np


class ECConvError(ValueError):
    pass


def _shifted(S, m, Csp, kh, kw, stride, pad, Ho, Wo):
    """X[p_k][n, j, oy, ox] = S[n, m*Csp + j, oy*s - pad + ky, ox*s - pad + kx]
    (zero outside the map), p_k = ky*kw + kx."""
    A = S[:, m * Csp:(m + 1) * Csp]
    N, _, H, W = A.shape
    Ap = np.zeros((N, Csp, H + 2 * pad, W + 2 * pad))
    Ap[:, :, pad:pad + H, pad:pad + W] = A
    X = np.empty((kh * kw, N, Csp, Ho, Wo))
    for ky in range(kh):
        for kx in range(kw):
            X[ky * kw + kx] = Ap[:, :, ky:ky + stride * (Ho - 1) + 1:stride,
                                 kx:kx + stride * (Wo - 1) + 1:stride]
    return X


def _contribution(X, Dm, codes_m):
    """sum_{p_k} D_{k(c_t, p_k)}^T X[p_k] -> [N, Ct, Ho, Wo]."""
    out = 0.0
    for pk in range(X.shape[0]):
        out = out + np.einsum("cj,njyx->ncyx", Dm[codes_m[:, pk]], X[pk])
    return out


def approx_response(S, D, codes, kh, kw, stride, pad):
    S = np.asarray(S, np.float64)
    D = np.asarray(D, np.float64)
    N, Cs, H, W = S.shape
    M, K, Csp = D.shape
    Ho, Wo = (H + 2 * pad - kh) // stride + 1, (W + 2 * pad - kw) // stride + 1
    Y = np.zeros((N, codes.shape[0], Ho, Wo))
    for m in range(M):
        Y += _contribution(_shifted(S, m, Csp, kh, kw, stride, pad, Ho, Wo), D[m], codes[:, :, m])
    return Y


def objective(S, T, D, codes, kh, kw, stride, pad):
    """Eq. B.1."""
    return float(np.sum((np.asarray(T, np.float64) -
                         approx_response(S, D, codes, kh, kw, stride, pad)) ** 2))


def _solve_spd(G, b, what):
    try:
        L = np.linalg.cholesky(G)
    except np.linalg.LinAlgError:
        raise ECConvError(f"{what}: singular least-squares problem")
    return np.linalg.solve(L.T, np.linalg.solve(L, b))


def ec_quantize_conv(S, T, D0, codes0, kh, kw, stride, pad, outer, inner, trace=None):
    """Returns (D [M, K, Csp] float64, codes [Ct, kh*kw, M] uint8).  `trace`, if
    a list, receives the objective after every sub-space step."""
    S = np.asarray(S, np.float64)
    T = np.asarray(T, np.float64)
    D = np.array(D0, np.float64)
    codes = np.array(codes0, np.uint8)
    N, Cs, H, W = S.shape
    M, K, Csp = D.shape
    Ct, kk, Mc = codes.shape
    Ho, Wo = (H + 2 * pad - kh) // stride + 1, (W + 2 * pad - kw) // stride + 1
    if M * Csp != Cs or Mc != M or kk != kh * kw or T.shape != (N, Ct, Ho, Wo):
        raise ECConvError("shape mismatch")
    if np.any(codes >= K):
        raise ECConvError("code >= K")
    E = T - approx_response(S, D, codes, kh, kw, stride, pad)
    for _ in range(outer):
        for m in range(M):
            X = _shifted(S, m, Csp, kh, kw, stride, pad, Ho, Wo)
            cm = codes[:, :, m]                               # [Ct, kk] view
            R = E + _contribution(X, D[m], cm)                # Eq. B.2
            Ecur = R - _contribution(X, D[m], cm)             # what sub-space m leaves
            for _ in range(inner):
                for k in range(K):                           # D update, Eq. B.4 - B.6
                    mask = (cm == k).astype(np.float64)       # [Ct, kk]
                    if not mask.any():
                        continue
                    Z = np.einsum("cq,qnjyx->ncjyx", mask, X)  # Z_k [N, Ct, Csp, Ho, Wo]
                    Q = Ecur + np.einsum("j,ncjyx->ncyx", D[m, k], Z)   # Eq. B.5
                    Gk = np.einsum("ncjyx,nclyx->jl", Z, Z)
                    rhs = np.einsum("ncjyx,ncyx->j", Z, Q)
                    D[m, k] = _solve_spd(Gk, rhs, f"sub-space {m}, codeword {k}")
                    Ecur = Q - np.einsum("j,ncjyx->ncyx", D[m, k], Z)
                for pk in range(kk):                         # B update, Eq. B.7 - B.8
                    Xp = X[pk]                                # [N, Csp, Ho, Wo]
                    P = Ecur + np.einsum("cj,njyx->ncyx", D[m][cm[:, pk]], Xp)   # Eq. B.7
                    G = np.einsum("njyx,nlyx->jl", Xp, Xp)
                    try:
                        np.linalg.cholesky(G)
                    except np.linalg.LinAlgError:
                        raise ECConvError(f"sub-space {m}, offset {pk}: singular G")
                    U = np.einsum("njyx,ncyx->jc", Xp, P)     # [Csp, Ct]
                    cost = np.einsum("kj,jl,kl->k", D[m], G, D[m])[:, None] - 2.0 * (D[m] @ U)
                    cm[:, pk] = np.argmin(cost, axis=0)      # Eq. B.8, first index on ties
                    Ecur = P - np.einsum("cj,njyx->ncyx", D[m][cm[:, pk]], Xp)
            E = Ecur
            if trace is not None:
                trace.append(objective(S, T, D, codes, kh, kw, stride, pad))
    return D, codes
