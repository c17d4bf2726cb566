"""float64 CPU oracle for the Q-CNN test-phase layer response.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The CUDA library never calls it, and it shares no code, header, table
or helper with that library.

The arithmetic lives in ``qcnn_oracle.c`` (plain loops in IEEE double, one loop
per symbol of the paper's equations); this module only builds that file with
gcc, marshals numpy arrays to it, and composes layers into a network.

Paper: Wu et al., "Quantized Convolutional Neural Networks for Mobile Devices"
(arXiv 1512.06473).
  - FC layer response: Sec. 3.1, Eq. 5 and the look-up-table paragraph after it.
  - Conv layer response: Sec. 3.2, Eq. 7 and the paragraph after it.
  - Whole network (conv/pool/FC stack): Sec. 4.2.3, Table 8.
  - ``lut_bf16=True``: every table entry rounded to bfloat16 (nearest, ties to
    even) before the sums, the rounding model of the library's reduced-precision
    table variant; ``round_bf16`` exposes that rounding.
  - Quantizer: k-means in every sub-space (Eq. 4 for FC, Eq. 6 for conv),
    ``kmeans``, ``pq_quantize_fc``, ``pq_quantize_conv`` (float32 in and out;
    distances in binary32, centroid sums in double, see the C file).

Array conventions (all numpy):
  fc:   x [N, Cs], codebooks D [M, K, Csp], codes [M, Ct] uint8, bias [Ct]
  conv: x [N, Cs, H, W], D [M, K, Csp], codes [Ct, kh*kw, M] uint8, bias [Ct]
Every function returns float64 arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(_HERE, "qcnn_oracle.c")
_SO = os.path.join(_HERE, "_build", "libqcnn_oracle.so")
_lock = threading.Lock()

_D = ctypes.POINTER(ctypes.c_double)
_F = ctypes.POINTER(ctypes.c_float)
_U8 = ctypes.POINTER(ctypes.c_uint8)
GCC_FLAGS = ["-O2", "-std=c99", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]


def compile_c(src: str, out: str) -> str:
    """Compile one C file of the oracle into a shared library (IEEE double,
    no fast-math, no fused multiply-add contraction, so x86 and Arm agree)."""
    os.makedirs(os.path.dirname(out) or ".", exist_ok=True)
    tmp = out + f".tmp{os.getpid()}"
    subprocess.run(["gcc", *GCC_FLAGS, "-o", tmp, src, "-lm"], check=True)
    os.replace(tmp, out)
    return out


def build(force: bool = False) -> str:
    """Build ``qcnn_oracle.c`` (only when the source is newer)."""
    with _lock:
        if (force or not os.path.exists(_SO)
                or os.path.getmtime(_SO) < os.path.getmtime(SOURCE)):
            compile_c(SOURCE, _SO)
    return _SO


class OracleError(RuntimeError):
    pass


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


def _f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


def _u8(a):
    a = np.asarray(a)
    if a.dtype != np.uint8:
        raise TypeError("codes must be uint8")
    return np.ascontiguousarray(a)


def _p(a, t):
    return a.ctypes.data_as(t)


def _check(rc, what):
    if rc != 0:
        raise OracleError(f"{what}: oracle returned {rc}")


class Oracle:
    """numpy front-end of one build of the C oracle."""

    def __init__(self, so_path: str):
        lib = ctypes.CDLL(so_path)
        i = ctypes.c_int
        lib.qo_fc_lut.argtypes = [_D, i, i, _D, i, i, i, _D]
        lib.qo_fc_forward.argtypes = [_D, i, i, i, _D, i, i, _U8, _D, i, i, _D]
        lib.qo_conv_lut.argtypes = [_D, i, i, i, i, _D, i, i, i, _D]
        lib.qo_conv_forward.argtypes = [_D, i, i, i, i, i, i, i, i, i, _D,
                                        i, i, _U8, _D, i, i, _D]
        lib.qo_round_bf16.argtypes = [ctypes.c_double]
        lib.qo_round_bf16.restype = ctypes.c_double
        lib.qo_maxpool.argtypes = [_D, i, i, i, i, i, i, _D]
        i64 = ctypes.c_longlong
        lib.qo_kmeans.argtypes = [_F, i64, i, i, _F, i, _F, _U8]
        lib.qo_pq_quantize_fc.argtypes = [_F, i, i, i, i, _F, i, _F, _U8]
        lib.qo_pq_quantize_conv.argtypes = [_F, i, i, i, i, i, i, _F, i, _F, _U8]
        for f in (lib.qo_fc_lut, lib.qo_fc_forward, lib.qo_conv_lut,
                  lib.qo_conv_forward, lib.qo_maxpool, lib.qo_kmeans,
                  lib.qo_pq_quantize_fc, lib.qo_pq_quantize_conv):
            f.restype = ctypes.c_int
        self.lib = lib

    def round_bf16(self, v):
        """Each value rounded to the nearest bfloat16 (ties to even)."""
        v = _f64(v)
        return np.array([self.lib.qo_round_bf16(float(e)) for e in v.ravel()],
                        np.float64).reshape(v.shape)

    def fc_lut(self, x, D, lut_bf16=False):
        """LUT[n, m, k] = <x[n, m*Csp:(m+1)*Csp], D[m, k, :]> (Sec. 3.1)."""
        x, D = _f64(x), _f64(D)
        N, Cs = x.shape
        M, K, Csp = D.shape
        out = np.empty((N, M, K), np.float64)
        _check(self.lib.qo_fc_lut(_p(x, _D), N, Cs, _p(D, _D), Csp, K,
                                  int(bool(lut_bf16)), _p(out, _D)), "fc_lut")
        return out

    def fc_forward(self, x, D, codes, bias=None, relu=False, lut_bf16=False):
        """Eq. 5: y[n, ct] = bias[ct] + sum_m LUT[n, m, codes[m, ct]]."""
        x, D, codes = _f64(x), _f64(D), _u8(codes)
        N, Cs = x.shape
        M, K, Csp = D.shape
        if M * Csp != Cs or codes.ndim != 2 or codes.shape[0] != M:
            raise OracleError("fc_forward: shape mismatch")
        Ct = codes.shape[1]
        b = None if bias is None else _f64(bias)
        y = np.empty((N, Ct), np.float64)
        _check(self.lib.qo_fc_forward(
            _p(x, _D), N, Cs, Ct, _p(D, _D), Csp, K, _p(codes, _U8),
            None if b is None else _p(b, _D), int(bool(relu)),
            int(bool(lut_bf16)), _p(y, _D)), "fc_forward")
        return y

    def conv_lut(self, x, D, lut_bf16=False):
        """LUT[n, m, iy*W+ix, k] = <x[n, m*Csp:(m+1)*Csp, iy, ix], D[m, k]>
        (Sec. 3.2: one table per input position)."""
        x, D = _f64(x), _f64(D)
        N, Cs, H, W = x.shape
        M, K, Csp = D.shape
        out = np.empty((N, M, H * W, K), np.float64)
        _check(self.lib.qo_conv_lut(_p(x, _D), N, Cs, H, W, _p(D, _D), Csp, K,
                                    int(bool(lut_bf16)), _p(out, _D)), "conv_lut")
        return out

    def conv_forward(self, x, D, codes, kh, kw, stride=1, pad=0, bias=None,
                     relu=False, lut_bf16=False):
        """Eq. 7: y[n, ct, oy, ox] = bias[ct] + sum_{(pk, ps)} sum_m
        LUT[n, m, ps, codes[ct, pk, m]], ps = (oy*s - pad + ky, ox*s - pad + kx)."""
        x, D, codes = _f64(x), _f64(D), _u8(codes)
        N, Cs, H, W = x.shape
        M, K, Csp = D.shape
        if M * Csp != Cs or codes.ndim != 3 or codes.shape[1] != kh * kw \
                or codes.shape[2] != M:
            raise OracleError("conv_forward: shape mismatch")
        Ct = codes.shape[0]
        Ho, Wo = conv_out_size(H, W, kh, kw, stride, pad)
        b = None if bias is None else _f64(bias)
        y = np.empty((N, Ct, Ho, Wo), np.float64)
        _check(self.lib.qo_conv_forward(
            _p(x, _D), N, Cs, H, W, Ct, kh, kw, stride, pad, _p(D, _D), Csp, K,
            _p(codes, _U8), None if b is None else _p(b, _D), int(bool(relu)),
            int(bool(lut_bf16)), _p(y, _D)), "conv_forward")
        return y

    def maxpool(self, x, k, s):
        """k x k max-pool, stride s, no padding, floor mode."""
        x = _f64(x)
        N, C, H, W = x.shape
        Ho, Wo = (H - k) // s + 1, (W - k) // s + 1
        y = np.empty((N, C, Ho, Wo), np.float64)
        _check(self.lib.qo_maxpool(_p(x, _D), N, C, H, W, k, s, _p(y, _D)),
               "maxpool")
        return y

    def kmeans(self, points, init, iters):
        """Lloyd's k-means of points [P, d] from centroids init [K, d]:
        returns (centroids [K, d] float32, assignment [P] uint8)."""
        pts, ini = _f32(points), _f32(init)
        P, d = pts.shape
        K = ini.shape[0]
        if ini.shape[1] != d:
            raise OracleError("kmeans: dimension mismatch")
        cen = np.empty((K, d), np.float32)
        a = np.empty(P, np.uint8)
        _check(self.lib.qo_kmeans(_p(pts, _F), P, d, K, _p(ini, _F), int(iters),
                                  _p(cen, _F), _p(a, _U8)), "kmeans")
        return cen, a

    def pq_quantize_fc(self, W, Csp, K, init, iters):
        """Eq. 4 for W [Ct, Cs]: returns D [M, K, Csp] and codes [M, Ct]."""
        W, ini = _f32(W), _f32(init)
        Ct, Cs = W.shape
        M = Cs // Csp
        if ini.shape != (M, K, Csp):
            raise OracleError("pq_quantize_fc: init must be [M, K, Csp]")
        D = np.empty((M, K, Csp), np.float32)
        codes = np.empty((M, Ct), np.uint8)
        _check(self.lib.qo_pq_quantize_fc(_p(W, _F), Ct, Cs, Csp, K, _p(ini, _F), int(iters),
                                          _p(D, _F), _p(codes, _U8)), "pq_quantize_fc")
        return D, codes

    def pq_quantize_conv(self, W, Csp, K, init, iters):
        """Eq. 6 for W [Ct, Cs, kh, kw]: returns D [M, K, Csp] and codes
        [Ct, kh*kw, M]."""
        W, ini = _f32(W), _f32(init)
        Ct, Cs, kh, kw = W.shape
        M = Cs // Csp
        if ini.shape != (M, K, Csp):
            raise OracleError("pq_quantize_conv: init must be [M, K, Csp]")
        D = np.empty((M, K, Csp), np.float32)
        codes = np.empty((Ct, kh * kw, M), np.uint8)
        _check(self.lib.qo_pq_quantize_conv(_p(W, _F), Ct, Cs, kh, kw, Csp, K, _p(ini, _F),
                                            int(iters), _p(D, _F), _p(codes, _U8)),
               "pq_quantize_conv")
        return D, codes

    def net_forward(self, x, layers, return_all=False):
        """Compose the oracle layers into a network (Sec. 4.2.3).

        ``layers`` is a list of dicts:
          {"kind": "conv", "D", "codes", "bias", "kh", "kw", "stride", "pad", "relu"}
          {"kind": "maxpool", "k", "s"}
          {"kind": "fc", "D", "codes", "bias", "relu"}
        plus an optional "lut_bf16" on conv and fc layers.
        A conv/pool output feeding an FC layer is flattened in C*H*W order.
        """
        h = _f64(x)
        outs = []
        for L in layers:
            kind = L["kind"]
            if kind == "conv":
                h = self.conv_forward(h, L["D"], L["codes"], L["kh"], L["kw"],
                                      L.get("stride", 1), L.get("pad", 0),
                                      L.get("bias"), L.get("relu", False),
                                      L.get("lut_bf16", False))
            elif kind == "maxpool":
                h = self.maxpool(h, L["k"], L["s"])
            elif kind == "fc":
                if h.ndim != 2:
                    h = h.reshape(h.shape[0], -1)
                h = self.fc_forward(h, L["D"], L["codes"], L.get("bias"),
                                    L.get("relu", False), L.get("lut_bf16", False))
            else:
                raise OracleError(f"unknown layer kind {kind!r}")
            outs.append(h)
        return outs if return_all else h


_default = None


def default() -> Oracle:
    global _default
    if _default is None:
        so = build()
        with _lock:
            if _default is None:
                _default = Oracle(so)
    return _default


def round_bf16(v):
    return default().round_bf16(v)


def fc_lut(x, D, lut_bf16=False):
    return default().fc_lut(x, D, lut_bf16)


def fc_forward(x, D, codes, bias=None, relu=False, lut_bf16=False):
    return default().fc_forward(x, D, codes, bias, relu, lut_bf16)


def conv_lut(x, D, lut_bf16=False):
    return default().conv_lut(x, D, lut_bf16)


def conv_forward(x, D, codes, kh, kw, stride=1, pad=0, bias=None, relu=False,
                 lut_bf16=False):
    return default().conv_forward(x, D, codes, kh, kw, stride, pad, bias, relu,
                                  lut_bf16)


def maxpool(x, k, s):
    return default().maxpool(x, k, s)


def net_forward(x, layers, return_all=False):
    return default().net_forward(x, layers, return_all)


def kmeans(points, init, iters):
    return default().kmeans(points, init, iters)


def pq_quantize_fc(W, Csp, K, init, iters):
    return default().pq_quantize_fc(W, Csp, K, init, iters)


def pq_quantize_conv(W, Csp, K, init, iters):
    return default().pq_quantize_conv(W, Csp, K, init, iters)


def conv_out_size(H, W, kh, kw, stride, pad):
    return (H + 2 * pad - kh) // stride + 1, (W + 2 * pad - kw) // stride + 1
