"""GB300 (sm_103a) implementation of the test-phase response of
product-quantized conv and FC layers (Q-CNN, Wu et al., arXiv 1512.06473).

This module only marshals arguments: every step of the path runs in the CUDA
kernels of libqcnn.so behind the C ABI of include/qcnn.h.  PyTorch provides
device memory and the current stream.  There is no CPU fallback: if the
library cannot be built or loaded, every call raises.

Layouts (fp32 unless stated, all CUDA tensors, contiguous):
  FC   : x [N, Cs], D [M, K, Csp], codes [M, Ct] uint8, bias [Ct]  -> [N, Ct]
  conv : x [N, Cs, H, W], D [M, K, Csp], codes [Ct, kh*kw, M] uint8 -> [N, Ct, Ho, Wo]

``lut="bf16"`` rounds every table entry to bfloat16 (nearest, ties to even)
and still sums in fp32; ``lut="fp32"`` (default) keeps fp32 entries.
"""
from __future__ import annotations

import ctypes
from dataclasses import dataclass
from typing import List, Optional, Sequence

import torch

from . import _lib
from ._lib import QcnnError, load, set_debug  # noqa: F401

__all__ = ["lut_build", "fc_forward", "conv_forward", "conv_pack_codes", "maxpool",
           "kmeans", "pq_quantize_fc", "pq_quantize_conv", "ec_quantize_fc", "ec_quantize_conv",
           "code_bits", "pack_bits", "unpack_bits", "fc_pack_codes", "serialize_model",
           "model_info", "load_model",
           "ConvLayer", "FCLayer", "PoolLayer", "Net", "launch_count", "QcnnError", "load",
           "set_debug", "debug_checks", "device_check", "smem_load_rate"]


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _need(t: torch.Tensor, name: str, dtype, ndim: int):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if t.dim() != ndim or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous {ndim}-d tensor, got shape {tuple(t.shape)}")


def _workspace(nbytes: int, device, workspace: Optional[torch.Tensor]):
    if nbytes == 0:
        return None, 0
    if workspace is not None:
        return workspace, workspace.numel() * workspace.element_size()
    ws = torch.empty(nbytes + 256, dtype=torch.uint8, device=device)
    off = (-ws.data_ptr()) % 256
    return ws[off:off + nbytes], nbytes


def debug_checks() -> bool:
    """True when the binding calls the debug build (set_debug(True))."""
    return bool(load().qcnn_debug_checks())


def device_check(stream=None) -> int:
    """Synchronize the stream and return the debug build's device-check flags
    since the last check (QCNN_CHECK_CODE 1: a code >= K was read;
    QCNN_CHECK_TABLE 2: a table read outside the built table;
    QCNN_CHECK_GLOBAL 4: a device-memory access outside its array), clearing
    them.  Always 0 with the release build."""
    flags = ctypes.c_uint(0)
    st = load().qcnn_device_check(_stream(stream), ctypes.byref(flags))
    if st not in (_lib.OK, _lib.ERR_DEVICE_CHECK):
        _lib.check(st, "qcnn_device_check")
    return int(flags.value)


def smem_load_rate(vec_bytes: int = 16, stream=None) -> float:
    """Shared-memory load wavefronts (128 B) per SM per cycle this GPU
    sustains with conflict-free loads of vec_bytes (4 or 16) per lane
    (qcnn_smem_load_rate): the peak of the look-up stage's roofline."""
    r = ctypes.c_double(0.0)
    _lib.check(load().qcnn_smem_load_rate(int(vec_bytes), ctypes.byref(r), _stream(stream)),
               "qcnn_smem_load_rate")
    return float(r.value)


def launch_count() -> int:
    """Kernels launched by libqcnn in this process so far."""
    return int(load().qcnn_launch_count())


def lut_build(x: torch.Tensor, D: torch.Tensor, out: Optional[torch.Tensor] = None, stream=None,
              lut: str = "fp32"):
    """Tables lut[n, m, p, k] = <x[n, m*Csp:(m+1)*Csp, p], D[m, k]> (Sec. 3.1 / 3.2).
    x is [N, Cs] (FC input) or [N, Cs, H, W]; returns [N, M, H*W, K], float32
    or (lut="bf16") bfloat16."""
    if x.dim() == 2:
        N, Cs = x.shape
        H = W = 1
    else:
        _need(x, "x", torch.float32, 4)
        N, Cs, H, W = x.shape
    _need(x, "x", torch.float32, x.dim())
    _need(D, "D", torch.float32, 3)
    M, K, Csp = D.shape
    lt = _lib.LUT[lut]
    dt = torch.bfloat16 if lt else torch.float32
    if out is None:
        out = torch.empty((N, M, H * W, K), dtype=dt, device=x.device)
    _need(out, "out", dt, 4)
    _lib.check(load().qcnn_lut_build(_ptr(x), N, Cs, H, W, _ptr(D), Csp, K, _ptr(out), lt,
                                     _stream(stream)), "qcnn_lut_build")
    return out


def fc_forward(x, D, codes, bias=None, relu=False, out=None, workspace=None, stream=None,
               lut="fp32", Ct=None):
    """Eq. 5: y[n, ct] = bias[ct] + sum_m LUT_n[m, codes[m, ct]] (then ReLU).
    ``codes`` is [M, Ct] uint8, or the 1-d output of fc_pack_codes (then
    ``Ct`` is required)."""
    _need(x, "x", torch.float32, 2)
    _need(D, "D", torch.float32, 3)
    packed = codes.dim() == 1
    _need(codes, "codes", torch.uint8, 1 if packed else 2)
    N, Cs = x.shape
    M, K, Csp = D.shape
    if packed:
        if Ct is None:
            raise ValueError("Ct is required with packed codes")
    else:
        Ct = codes.shape[1]
    if bias is not None:
        _need(bias, "bias", torch.float32, 1)
    lib = load()
    lt = _lib.LUT[lut]
    nb = ctypes.c_size_t()
    _lib.check(lib.qcnn_fc_workspace_size(N, Cs, Ct, Csp, K, lt, ctypes.byref(nb)),
               "qcnn_fc_workspace_size")
    ws, wsb = _workspace(nb.value, x.device, workspace)
    if out is None:
        out = torch.empty((N, Ct), dtype=torch.float32, device=x.device)
    fn = lib.qcnn_fc_forward_packed if packed else lib.qcnn_fc_forward
    _lib.check(fn(_ptr(x), N, Cs, Ct, _ptr(D), Csp, K, _ptr(codes), _ptr(bias), _ptr(out),
                  int(bool(relu)), lt, _ptr(ws), wsb, _stream(stream)), "qcnn_fc_forward")
    return out


def _aligned_bytes(nbytes, device, align=256):
    raw = torch.empty(nbytes + align, dtype=torch.uint8, device=device)
    off = (-raw.data_ptr()) % align
    return raw[off:off + nbytes]


def code_bits(K: int) -> int:
    """Bits per stored code, ceil(log2 K) (at least 1)."""
    return int(load().qcnn_code_bits(K))


def pack_bits(codes: torch.Tensor, bits: int, stream=None) -> torch.Tensor:
    """Codes (any shape, uint8) -> the packed stream, ceil(n*bits/8) bytes."""
    _need(codes, "codes", torch.uint8, codes.dim())
    n = codes.numel()
    out = torch.empty((n * bits + 7) // 8, dtype=torch.uint8, device=codes.device)
    _lib.check(load().qcnn_pack_bits(_ptr(codes), n, bits, _ptr(out), _stream(stream)),
               "qcnn_pack_bits")
    return out


def unpack_bits(stream_bytes: torch.Tensor, n: int, bits: int, stream=None) -> torch.Tensor:
    _need(stream_bytes, "stream_bytes", torch.uint8, 1)
    out = torch.empty(n, dtype=torch.uint8, device=stream_bytes.device)
    _lib.check(load().qcnn_unpack_bits(_ptr(stream_bytes), n, bits, _ptr(out), _stream(stream)),
               "qcnn_unpack_bits")
    return out


def fc_pack_codes(codes: torch.Tensor, K: int, stream=None) -> torch.Tensor:
    """FC codes [M, Ct] -> bit-packed rows (16-byte pitch) for fc_forward."""
    _need(codes, "codes", torch.uint8, 2)
    M, Ct = codes.shape
    lib = load()
    out = _aligned_bytes(lib.qcnn_fc_packed_codes_bytes(M, Ct, K), codes.device)
    _lib.check(lib.qcnn_fc_pack_codes(_ptr(codes), M, Ct, K, _ptr(out), _stream(stream)),
               "qcnn_fc_pack_codes")
    return out


def conv_pack_codes(codes: torch.Tensor, K: int, kh: int, kw: int, stream=None) -> torch.Tensor:
    """Model-load-time re-layout of conv codes [Ct, kh*kw, M] for the fused kernels."""
    _need(codes, "codes", torch.uint8, 3)
    Ct, kk, M = codes.shape
    if kk != kh * kw:
        raise ValueError("codes.shape[1] must be kh*kw")
    lib = load()
    nbytes = lib.qcnn_conv_packed_codes_bytes(Ct, kh, kw, M)
    packed = torch.empty(nbytes + 256, dtype=torch.uint8, device=codes.device)
    off = (-packed.data_ptr()) % 256
    packed = packed[off:off + nbytes]
    _lib.check(lib.qcnn_conv_pack_codes(_ptr(codes), Ct, kh, kw, M, K, _ptr(packed),
                                        _stream(stream)), "qcnn_conv_pack_codes")
    return packed


def fused_variants():
    """The fused conv kernel's tile variants: a list of dicts (index = the
    variant number accepted by conv_forward's ``algo``)."""
    lib = load()
    keys = ("P", "CTW", "WP", "CSP4", "NW", "MINB", "PIPE", "BF", "SK", "TC")
    out = []
    for v in range(lib.qcnn_conv_fused_variant_count()):
        info = (ctypes.c_int * 10)()
        _lib.check(lib.qcnn_conv_fused_variant_info(v, info), "qcnn_conv_fused_variant_info")
        out.append(dict(zip(keys, list(info))))
    return out


_ALGO_NAMES = {v: k for k, v in _lib.ALGO.items()}


def conv_plan(N, Cs, H, W, Ct, kh, kw, stride=1, pad=0, Csp=4, K=128, algo="auto",
              packed=True, lut="fp32", cluster=True):
    """The plan conv_forward would run for these sizes (qcnn_conv_plan_info),
    worked out on the host: a dict with the algorithm's name, its kernel
    variant, positions per tile, channels per CTA, splits, stream-K, CTAs and
    the CTAs per cluster among the splits (1: none)."""
    a = _lib.ALGO[algo] if isinstance(algo, str) else _lib.ALGO_FUSED_VARIANT + int(algo)
    if not cluster:
        a |= _lib.ALGO_NO_CLUSTER
    info = (ctypes.c_int * 8)()
    _lib.check(load().qcnn_conv_plan_info(N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K,
                                          _lib.CODES_PACKED if packed else _lib.CODES_CANONICAL,
                                          a, _lib.LUT[lut], info), "qcnn_conv_plan_info")
    keys = ("algo", "variant", "positions", "channels", "splits", "stream_k", "ctas", "cluster")
    d = dict(zip(keys, list(info)))
    d["algo"] = _ALGO_NAMES[d["algo"]]
    return d


def fc_plan(N, Cs, Ct, Csp=4, K=32, lut="fp32"):
    """The plan fc_forward would run (qcnn_fc_plan_info): images and outputs
    per CTA, splits, sub-spaces per chunk, CTAs and CTAs per cluster (1: none)."""
    info = (ctypes.c_int * 6)()
    _lib.check(load().qcnn_fc_plan_info(N, Cs, Ct, Csp, K, _lib.LUT[lut], info),
               "qcnn_fc_plan_info")
    return dict(zip(("images", "outputs", "splits", "chunk", "ctas", "cluster"), list(info)))


def conv_forward(x, D, codes, kh, kw, stride=1, pad=0, bias=None, relu=False, algo="auto",
                 packed=False, Ct=None, out=None, workspace=None, stream=None, lut="fp32",
                 cluster=True):
    """Eq. 7 conv response.  ``codes`` is [Ct, kh*kw, M] uint8, or (packed=True,
    then ``Ct`` is required) the output of conv_pack_codes.  ``algo`` is
    "auto", "fused", "unfused", "chunked", "phase", or an int v: fused tile variant v
    of fused_variants().  cluster=False keeps split sub-space ranges out of
    thread-block clusters (QCNN_ALGO_NO_CLUSTER)."""
    _need(x, "x", torch.float32, 4)
    _need(D, "D", torch.float32, 3)
    N, Cs, H, W = x.shape
    M, K, Csp = D.shape
    if packed:
        if Ct is None:
            raise ValueError("Ct is required with packed codes")
        _need(codes, "codes", torch.uint8, 1)
    else:
        _need(codes, "codes", torch.uint8, 3)
        Ct = codes.shape[0]
    if bias is not None:
        _need(bias, "bias", torch.float32, 1)
    layout = _lib.CODES_PACKED if packed else _lib.CODES_CANONICAL
    a = _lib.ALGO[algo] if isinstance(algo, str) else _lib.ALGO_FUSED_VARIANT + int(algo)
    if not cluster:
        a |= _lib.ALGO_NO_CLUSTER
    lt = _lib.LUT[lut]
    lib = load()
    nb = ctypes.c_size_t()
    _lib.check(lib.qcnn_conv_workspace_size(N, Cs, H, W, Ct, kh, kw, stride, pad, Csp, K, layout,
                                            a, lt, ctypes.byref(nb)), "qcnn_conv_workspace_size")
    ws, wsb = _workspace(nb.value, x.device, workspace)
    Ho = (H + 2 * pad - kh) // stride + 1
    Wo = (W + 2 * pad - kw) // stride + 1
    if out is None:
        out = torch.empty((N, Ct, Ho, Wo), dtype=torch.float32, device=x.device)
    _lib.check(lib.qcnn_conv_forward(_ptr(x), N, Cs, H, W, Ct, kh, kw, stride, pad, _ptr(D), Csp,
                                     K, _ptr(codes), layout, _ptr(bias), _ptr(out),
                                     int(bool(relu)), a, lt, _ptr(ws), wsb, _stream(stream)),
               "qcnn_conv_forward")
    return out


def maxpool(x, k, s, out=None, stream=None):
    _need(x, "x", torch.float32, 4)
    N, C, H, W = x.shape
    if out is None:
        out = torch.empty((N, C, (H - k) // s + 1, (W - k) // s + 1), dtype=torch.float32,
                          device=x.device)
    _lib.check(load().qcnn_maxpool(_ptr(x), N, C, H, W, k, s, _ptr(out), _stream(stream)),
               "qcnn_maxpool")
    return out


# ---------------------------------------------------------------- quantizer
def kmeans(points, init, iters, stream=None):
    """k-means in each of M sub-spaces (Eq. 4 / Eq. 6): points [M, P, Csp],
    init [M, K, Csp] -> (D [M, K, Csp] float32, assign [M, P] uint8)."""
    _need(points, "points", torch.float32, 3)
    _need(init, "init", torch.float32, 3)
    M, P, Csp = points.shape
    K = init.shape[1]
    if init.shape != (M, K, Csp):
        raise ValueError("init must be [M, K, Csp]")
    lib = load()
    nb = ctypes.c_size_t()
    _lib.check(lib.qcnn_kmeans_workspace_size(M, P, Csp, K, ctypes.byref(nb)),
               "qcnn_kmeans_workspace_size")
    ws, wsb = _workspace(nb.value, points.device, None)
    D = torch.empty((M, K, Csp), dtype=torch.float32, device=points.device)
    a = torch.empty((M, P), dtype=torch.uint8, device=points.device)
    _lib.check(lib.qcnn_kmeans(_ptr(points), M, P, Csp, K, _ptr(init), int(iters), _ptr(D),
                               _ptr(a), _ptr(ws), wsb, _stream(stream)), "qcnn_kmeans")
    return D, a


def _pq_quantize(kind, W, Csp, K, init, iters, stream):
    _need(init, "init", torch.float32, 3)
    if kind == _lib.LAYER_FC:
        _need(W, "W", torch.float32, 2)
        (Ct, Cs), kh, kw = W.shape, 1, 1
    else:
        _need(W, "W", torch.float32, 4)
        Ct, Cs, kh, kw = W.shape
    M = Cs // Csp
    if init.shape != (M, K, Csp):
        raise ValueError("init must be [M, K, Csp]")
    lib = load()
    nb = ctypes.c_size_t()
    _lib.check(lib.qcnn_pq_quantize_workspace_size(kind, Ct, Cs, kh, kw, Csp, K,
                                                   ctypes.byref(nb)),
               "qcnn_pq_quantize_workspace_size")
    ws, wsb = _workspace(nb.value, W.device, None)
    D = torch.empty((M, K, Csp), dtype=torch.float32, device=W.device)
    shape = (M, Ct) if kind == _lib.LAYER_FC else (Ct, kh * kw, M)
    codes = torch.empty(shape, dtype=torch.uint8, device=W.device)
    _lib.check(lib.qcnn_pq_quantize(kind, _ptr(W), Ct, Cs, kh, kw, Csp, K, _ptr(init),
                                    int(iters), _ptr(D), _ptr(codes), _ptr(ws), wsb,
                                    _stream(stream)), "qcnn_pq_quantize")
    return D, codes


def pq_quantize_fc(W, Csp, K, init, iters, stream=None):
    """Eq. 4: W [Ct, Cs] -> (D [M, K, Csp], codes [M, Ct])."""
    return _pq_quantize(_lib.LAYER_FC, W, Csp, K, init, iters, stream)


def pq_quantize_conv(W, Csp, K, init, iters, stream=None):
    """Eq. 6: W [Ct, Cs, kh, kw] -> (D [M, K, Csp], codes [Ct, kh*kw, M])."""
    return _pq_quantize(_lib.LAYER_CONV, W, Csp, K, init, iters, stream)


def ec_quantize_fc(S, T, D, codes, outer, inner, stream=None):
    """Error-corrected FC quantization (Eq. 8 - 12) from the starting point
    (D [M, K, Csp], codes [M, Ct]) on calibration pairs S [N, Cs], T [N, Ct].
    Returns new (D, codes); the inputs are not modified."""
    _need(S, "S", torch.float32, 2)
    _need(T, "T", torch.float32, 2)
    _need(D, "D", torch.float32, 3)
    _need(codes, "codes", torch.uint8, 2)
    N, Cs = S.shape
    Ct = T.shape[1]
    M, K, Csp = D.shape
    lib = load()
    nb = ctypes.c_size_t()
    _lib.check(lib.qcnn_ec_quantize_fc_workspace_size(N, Cs, Ct, Csp, K, ctypes.byref(nb)),
               "qcnn_ec_quantize_fc_workspace_size")
    ws, wsb = _workspace(nb.value, S.device, None)
    D2, c2 = D.clone(), codes.clone()
    _lib.check(lib.qcnn_ec_quantize_fc(_ptr(S), _ptr(T), N, Cs, Ct, Csp, K, _ptr(D2), _ptr(c2),
                                       int(outer), int(inner), _ptr(ws), wsb, _stream(stream)),
               "qcnn_ec_quantize_fc")
    return D2, c2


def ec_quantize_conv(S, T, D, codes, kh, kw, stride, pad, outer, inner, stream=None):
    """Error-corrected conv quantization (Appendix B) from (D [M, K, Csp],
    codes [Ct, kh*kw, M]) on calibration maps S [N, Cs, H, W] and pre-bias
    responses T [N, Ct, Ho, Wo].  Returns new (D, codes)."""
    _need(S, "S", torch.float32, 4)
    _need(T, "T", torch.float32, 4)
    _need(D, "D", torch.float32, 3)
    _need(codes, "codes", torch.uint8, 3)
    N, Cs, H, W = S.shape
    Ct = T.shape[1]
    M, K, Csp = D.shape
    lib = load()
    nb = ctypes.c_size_t()
    _lib.check(lib.qcnn_ec_quantize_conv_workspace_size(N, Cs, H, W, Ct, kh, kw, stride, pad, Csp,
                                                        K, ctypes.byref(nb)),
               "qcnn_ec_quantize_conv_workspace_size")
    ws, wsb = _workspace(nb.value, S.device, None)
    D2, c2 = D.clone(), codes.clone()
    _lib.check(lib.qcnn_ec_quantize_conv(_ptr(S), _ptr(T), N, Cs, H, W, Ct, kh, kw, stride, pad,
                                         Csp, K, _ptr(D2), _ptr(c2), int(outer), int(inner),
                                         _ptr(ws), wsb, _stream(stream)), "qcnn_ec_quantize_conv")
    return D2, c2


# ------------------------------------------------------------------ network
@dataclass
class ConvLayer:
    D: torch.Tensor
    codes: torch.Tensor         # [Ct, kh*kw, M] (canonical) or packed bytes
    bias: Optional[torch.Tensor]
    Ct: int
    kh: int
    kw: int
    stride: int = 1
    pad: int = 0
    relu: bool = True
    algo: str = "auto"
    packed: bool = False
    lut: str = "fp32"
    cluster: bool = True        # False: QCNN_ALGO_NO_CLUSTER (as conv_forward's cluster)


@dataclass
class FCLayer:
    D: torch.Tensor
    codes: torch.Tensor         # [M, Ct], or fc_pack_codes rows (packed=True, Ct given)
    bias: Optional[torch.Tensor]
    relu: bool = True
    lut: str = "fp32"
    packed: bool = False
    Ct: Optional[int] = None


@dataclass
class PoolLayer:
    k: int
    s: int


class Net:
    """A stack of PQ conv / PQ FC / max-pool layers run by qcnn_net_forward."""

    def __init__(self, layers: Sequence, in_shape: Sequence[int]):
        self.layers = list(layers)
        self.in_shape = tuple(in_shape)
        arr = (_lib.Layer * len(self.layers))()
        for i, L in enumerate(self.layers):
            d = arr[i]
            if isinstance(L, ConvLayer):
                M, K, Csp = L.D.shape
                d.kind, d.Ct, d.kh, d.kw, d.stride, d.pad = _lib.LAYER_CONV, L.Ct, L.kh, L.kw, L.stride, L.pad
                d.Csp, d.K, d.relu, d.algo = Csp, K, int(L.relu), _lib.ALGO[L.algo]
                if not L.cluster:
                    d.algo |= _lib.ALGO_NO_CLUSTER
                d.codes_layout = _lib.CODES_PACKED if L.packed else _lib.CODES_CANONICAL
                d.lut_type = _lib.LUT[L.lut]
                d.D, d.codes, d.bias = _ptr(L.D), _ptr(L.codes), _ptr(L.bias)
            elif isinstance(L, FCLayer):
                M, K, Csp = L.D.shape
                ct = L.Ct if L.packed else L.codes.shape[1]
                d.kind, d.Ct, d.Csp, d.K, d.relu = _lib.LAYER_FC, ct, Csp, K, int(L.relu)
                d.codes_layout = _lib.CODES_PACKED if L.packed else _lib.CODES_CANONICAL
                d.lut_type = _lib.LUT[L.lut]
                d.D, d.codes, d.bias = _ptr(L.D), _ptr(L.codes), _ptr(L.bias)
            elif isinstance(L, PoolLayer):
                d.kind, d.kh, d.kw, d.stride = _lib.LAYER_MAXPOOL, L.k, L.k, L.s
            else:
                raise TypeError(f"unknown layer {L!r}")
        self._arr = arr
        C, H, W = self.in_shape
        oc, oh, ow = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
        _lib.check(load().qcnn_net_output_shape(arr, len(arr), C, H, W, ctypes.byref(oc),
                                                ctypes.byref(oh), ctypes.byref(ow)),
                   "qcnn_net_output_shape")
        self.out_shape = (oc.value, oh.value, ow.value)

    def _out(self, N, device):
        C, H, W = self.out_shape
        shape = (N, C) if (H, W) == (1, 1) else (N, C, H, W)
        return torch.empty(shape, dtype=torch.float32, device=device)

    def workspace_bytes(self, N: int, host_io: bool = False) -> int:
        nb = ctypes.c_size_t()
        C, H, W = self.in_shape
        _lib.check(load().qcnn_net_workspace_size(self._arr, len(self._arr), N, C, H, W,
                                                  int(host_io), ctypes.byref(nb)),
                   "qcnn_net_workspace_size")
        return nb.value

    def plan_info(self, N: int, host_io: bool = False):
        """Per layer, whether qcnn_net_forward (host_io: qcnn_net_forward_host)
        at batch N hands its split partial sums to the next layer instead of
        a reduction launch (qcnn_net_plan_info): a list of dicts with
        "leaves_partials" and "takes_partials"."""
        n = len(self._arr)
        info = (ctypes.c_int * (2 * n))()
        C, H, W = self.in_shape
        _lib.check(load().qcnn_net_plan_info(self._arr, n, N, C, H, W, int(host_io), info),
                   "qcnn_net_plan_info")
        return [{"leaves_partials": bool(info[2 * i]), "takes_partials": bool(info[2 * i + 1])}
                for i in range(n)]

    def alloc_workspace(self, N: int, device="cuda", host_io: bool = False):
        nb = self.workspace_bytes(N, host_io)
        ws, _ = _workspace(max(nb, 1), torch.device(device), None)
        return ws

    def forward(self, x: torch.Tensor, out=None, workspace=None, stream=None):
        _need(x, "x", torch.float32, 4)
        N, C, H, W = x.shape
        if (C, H, W) != self.in_shape:
            raise ValueError(f"input shape {(C, H, W)} != {self.in_shape}")
        if workspace is None:
            workspace = self.alloc_workspace(N, x.device)
        if out is None:
            out = self._out(N, x.device)
        wsb = workspace.numel()
        _lib.check(load().qcnn_net_forward(self._arr, len(self._arr), _ptr(x), N, C, H, W,
                                           _ptr(out), _ptr(workspace), wsb, _stream(stream)),
                   "qcnn_net_forward")
        return out

    def forward_host(self, x_host: torch.Tensor, out_host: torch.Tensor, workspace: torch.Tensor,
                     stream=None):
        """x_host / out_host are CPU tensors (pinned for speed); workspace must be
        alloc_workspace(N, host_io=True).  Synchronizes the stream."""
        if x_host.is_cuda or out_host.is_cuda:
            raise TypeError("forward_host takes CPU tensors")
        if not (x_host.is_contiguous() and out_host.is_contiguous()):
            raise ValueError("host tensors must be contiguous")
        N, C, H, W = x_host.shape
        _lib.check(load().qcnn_net_forward_host(self._arr, len(self._arr), _ptr(x_host), N, C, H,
                                                W, _ptr(out_host), _ptr(workspace),
                                                workspace.numel(), _stream(stream)),
                   "qcnn_net_forward_host")
        return out_host


# ------------------------------------------------------------- model blob
def _host_layers(layers):
    """(qcnn_layer array with host pointers, arrays kept alive)."""
    import numpy as np
    arr = (_lib.Layer * len(layers))()
    keep = []
    for i, L in enumerate(layers):
        d = arr[i]
        kind = L["kind"]
        if kind == "maxpool":
            d.kind, d.kh, d.kw, d.stride = _lib.LAYER_MAXPOOL, L["k"], L["k"], L["s"]
            continue
        D = np.ascontiguousarray(L["D"], np.float32)
        codes = np.ascontiguousarray(L["codes"], np.uint8)
        bias = None if L.get("bias") is None else np.ascontiguousarray(L["bias"], np.float32)
        keep += [D, codes, bias]
        M, K, Csp = D.shape
        if kind == "conv":
            d.kind, d.Ct, d.kh, d.kw = _lib.LAYER_CONV, codes.shape[0], L["kh"], L["kw"]
            d.stride, d.pad = L.get("stride", 1), L.get("pad", 0)
        else:
            d.kind, d.Ct = _lib.LAYER_FC, codes.shape[1]
        d.Csp, d.K, d.relu = Csp, K, int(bool(L.get("relu", False)))
        d.D, d.codes = D.ctypes.data, codes.ctypes.data
        d.bias = None if bias is None else bias.ctypes.data
    return arr, keep


def serialize_model(layers, in_shape) -> bytes:
    """A stack (list of dicts: {"kind": "conv"|"fc"|"maxpool", "D", "codes" in
    the canonical layout, "bias", "kh", "kw", "stride", "pad", "relu"} or
    {"kind": "maxpool", "k", "s"}, numpy arrays) -> the model blob."""
    arr, keep = _host_layers(layers)
    C, H, W = in_shape
    lib = load()
    need = ctypes.c_size_t()
    _lib.check(lib.qcnn_model_serialize(arr, len(arr), C, H, W, None, 0, ctypes.byref(need)),
               "qcnn_model_serialize")
    buf = ctypes.create_string_buffer(need.value)
    _lib.check(lib.qcnn_model_serialize(arr, len(arr), C, H, W, buf, need.value,
                                        ctypes.byref(need)), "qcnn_model_serialize")
    return buf.raw[:need.value]


def model_info(blob: bytes):
    """(n_layers, (C, H, W), device bytes) of a blob."""
    n, C, H, W = ctypes.c_int(), ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    nb = ctypes.c_size_t()
    _lib.check(load().qcnn_model_info(blob, len(blob), ctypes.byref(n), ctypes.byref(C),
                                      ctypes.byref(H), ctypes.byref(W), ctypes.byref(nb)),
               "qcnn_model_info")
    return n.value, (C.value, H.value, W.value), nb.value


class LoadedNet(Net):
    """A Net whose parameters live in one device buffer filled from a blob."""

    def __init__(self, blob: bytes, device="cuda", stream=None):
        n, in_shape, nbytes = model_info(blob)
        self.buffer = _aligned_bytes(max(nbytes, 1), torch.device(device))
        arr = (_lib.Layer * n)()
        _lib.check(load().qcnn_model_upload(blob, len(blob), _ptr(self.buffer), nbytes, arr,
                                            _stream(stream)), "qcnn_model_upload")
        self.layers = [None] * n
        self.in_shape = tuple(in_shape)
        self._arr = arr
        C, H, W = self.in_shape
        oc, oh, ow = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
        _lib.check(load().qcnn_net_output_shape(arr, n, C, H, W, ctypes.byref(oc),
                                                ctypes.byref(oh), ctypes.byref(ow)),
                   "qcnn_net_output_shape")
        self.out_shape = (oc.value, oh.value, ow.value)

    def set_lut(self, lut: str):
        """Table precision of every PQ layer ("fp32" or "bf16")."""
        for d in self._arr:
            if d.kind != _lib.LAYER_MAXPOOL:
                d.lut_type = _lib.LUT[lut]


def load_model(blob_or_path, device="cuda", stream=None) -> LoadedNet:
    """Load a model blob (bytes, or a file path) onto the GPU."""
    blob = blob_or_path
    if not isinstance(blob, (bytes, bytearray)):
        with open(blob_or_path, "rb") as f:
            blob = f.read()
    return LoadedNet(bytes(blob), device, stream)
