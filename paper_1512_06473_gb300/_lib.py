"""ctypes view of libqcnn.so (include/qcnn.h).  Loading fails loudly: there is
no CPU fallback and no other backend."""
from __future__ import annotations

import ctypes
import os
import re
import threading

from . import build as _build

c_int, c_size_t, c_void_p, c_uint64 = ctypes.c_int, ctypes.c_size_t, ctypes.c_void_p, ctypes.c_uint64

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_WORKSPACE, ERR_CUDA, ERR_DATA = 0, 1, 2, 3, 4, 5
ERR_DEVICE_CHECK = 6
CHECK_CODE, CHECK_TABLE, CHECK_GLOBAL = 1, 2, 4  # qcnn_device_check flag bits
ALGO = {"auto": 0, "fused": 1, "unfused": 2, "chunked": 3, "phase": 4}
ALGO_FUSED_VARIANT = 256  # + v: fused tile variant v
ALGO_NO_CLUSTER = 1 << 16  # flag: no thread-block clusters for split sub-spaces
CODES_CANONICAL, CODES_PACKED = 0, 1
LUT = {"fp32": 0, "bf16": 1}
LAYER_CONV, LAYER_FC, LAYER_MAXPOOL = 0, 1, 2


class QcnnError(RuntimeError):
    def __init__(self, status: int, what: str, msg: str):
        super().__init__(f"{what}: {msg} (status {status})")
        self.status = status


class Layer(ctypes.Structure):
    """Mirror of qcnn_layer."""
    _fields_ = [("kind", c_int), ("Ct", c_int), ("kh", c_int), ("kw", c_int),
                ("stride", c_int), ("pad", c_int), ("Csp", c_int), ("K", c_int),
                ("relu", c_int), ("algo", c_int), ("codes_layout", c_int),
                ("lut_type", c_int), ("D", c_void_p), ("codes", c_void_p), ("bias", c_void_p)]


_SIGS = {
    "qcnn_status_string": (ctypes.c_char_p, [c_int]),
    "qcnn_last_cuda_error": (c_int, []),
    "qcnn_launch_count": (c_uint64, []),
    "qcnn_debug_checks": (c_int, []),
    "qcnn_smem_load_rate": (c_int, [c_int, ctypes.POINTER(ctypes.c_double), c_void_p]),
    "qcnn_device_check": (c_int, [c_void_p, ctypes.POINTER(ctypes.c_uint)]),
    "qcnn_lut_build": (c_int, [c_void_p, c_int, c_int, c_int, c_int, c_void_p, c_int, c_int,
                               c_void_p, c_int, c_void_p]),
    "qcnn_fc_workspace_size": (c_int, [c_int, c_int, c_int, c_int, c_int, c_int,
                                       ctypes.POINTER(c_size_t)]),
    "qcnn_fc_forward": (c_int, [c_void_p, c_int, c_int, c_int, c_void_p, c_int, c_int, c_void_p,
                                c_void_p, c_void_p, c_int, c_int, c_void_p, c_size_t, c_void_p]),
    "qcnn_fc_forward_noalloc": (c_int, [c_void_p, c_int, c_int, c_int, c_void_p, c_int, c_int,
                                        c_void_p, c_void_p, c_void_p, c_int, c_void_p]),
    "qcnn_conv_packed_codes_bytes": (c_size_t, [c_int, c_int, c_int, c_int]),
    "qcnn_conv_pack_codes": (c_int, [c_void_p, c_int, c_int, c_int, c_int, c_int, c_void_p,
                                     c_void_p]),
    "qcnn_conv_fused_variant_count": (c_int, []),
    "qcnn_conv_fused_variant_info": (c_int, [c_int, ctypes.POINTER(c_int)]),
    "qcnn_conv_plan_info": (c_int, [c_int] * 14 + [ctypes.POINTER(c_int)]),
    "qcnn_fc_plan_info": (c_int, [c_int] * 6 + [ctypes.POINTER(c_int)]),
    "qcnn_conv_workspace_size": (c_int, [c_int] * 14 + [ctypes.POINTER(c_size_t)]),
    "qcnn_conv_forward": (c_int, [c_void_p, c_int, c_int, c_int, c_int, c_int, c_int, c_int,
                                  c_int, c_int, c_void_p, c_int, c_int, c_void_p, c_int,
                                  c_void_p, c_void_p, c_int, c_int, c_int, c_void_p, c_size_t,
                                  c_void_p]),
    "qcnn_maxpool": (c_int, [c_void_p, c_int, c_int, c_int, c_int, c_int, c_int, c_void_p,
                             c_void_p]),
    "qcnn_net_output_shape": (c_int, [ctypes.POINTER(Layer), c_int, c_int, c_int, c_int,
                                      ctypes.POINTER(c_int), ctypes.POINTER(c_int),
                                      ctypes.POINTER(c_int)]),
    "qcnn_net_workspace_size": (c_int, [ctypes.POINTER(Layer), c_int, c_int, c_int, c_int, c_int,
                                        c_int, ctypes.POINTER(c_size_t)]),
    "qcnn_net_plan_info": (c_int, [ctypes.POINTER(Layer), c_int, c_int, c_int, c_int, c_int,
                                   c_int, ctypes.POINTER(c_int)]),
    "qcnn_net_forward": (c_int, [ctypes.POINTER(Layer), c_int, c_void_p, c_int, c_int, c_int,
                                 c_int, c_void_p, c_void_p, c_size_t, c_void_p]),
    "qcnn_net_forward_host": (c_int, [ctypes.POINTER(Layer), c_int, c_void_p, c_int, c_int,
                                      c_int, c_int, c_void_p, c_void_p, c_size_t, c_void_p]),
    "qcnn_code_bits": (c_int, [c_int]),
    "qcnn_model_serialize": (c_int, [ctypes.POINTER(Layer), c_int, c_int, c_int, c_int, c_void_p,
                                     c_size_t, ctypes.POINTER(c_size_t)]),
    "qcnn_model_info": (c_int, [c_void_p, c_size_t, ctypes.POINTER(c_int), ctypes.POINTER(c_int),
                                ctypes.POINTER(c_int), ctypes.POINTER(c_int),
                                ctypes.POINTER(c_size_t)]),
    "qcnn_model_upload": (c_int, [c_void_p, c_size_t, c_void_p, c_size_t, ctypes.POINTER(Layer),
                                  c_void_p]),
    "qcnn_pack_bits": (c_int, [c_void_p, ctypes.c_longlong, c_int, c_void_p, c_void_p]),
    "qcnn_unpack_bits": (c_int, [c_void_p, ctypes.c_longlong, c_int, c_void_p, c_void_p]),
    "qcnn_fc_packed_codes_bytes": (c_size_t, [c_int, c_int, c_int]),
    "qcnn_fc_pack_codes": (c_int, [c_void_p, c_int, c_int, c_int, c_void_p, c_void_p]),
    "qcnn_fc_forward_packed": (c_int, [c_void_p, c_int, c_int, c_int, c_void_p, c_int, c_int,
                                       c_void_p, c_void_p, c_void_p, c_int, c_int, c_void_p,
                                       c_size_t, c_void_p]),
    "qcnn_kmeans_workspace_size": (c_int, [c_int, c_int, c_int, c_int, ctypes.POINTER(c_size_t)]),
    "qcnn_kmeans": (c_int, [c_void_p, c_int, c_int, c_int, c_int, c_void_p, c_int, c_void_p,
                            c_void_p, c_void_p, c_size_t, c_void_p]),
    "qcnn_pq_quantize_workspace_size": (c_int, [c_int] * 7 + [ctypes.POINTER(c_size_t)]),
    "qcnn_ec_quantize_fc_workspace_size": (c_int, [c_int] * 5 + [ctypes.POINTER(c_size_t)]),
    "qcnn_ec_quantize_conv_workspace_size": (c_int, [c_int] * 11 + [ctypes.POINTER(c_size_t)]),
    "qcnn_ec_quantize_conv": (c_int, [c_void_p, c_void_p] + [c_int] * 11 +
                              [c_void_p, c_void_p, c_int, c_int, c_void_p, c_size_t, c_void_p]),
    "qcnn_ec_quantize_fc": (c_int, [c_void_p, c_void_p, c_int, c_int, c_int, c_int, c_int,
                                    c_void_p, c_void_p, c_int, c_int, c_void_p, c_size_t,
                                    c_void_p]),
    "qcnn_pq_quantize": (c_int, [c_int, c_void_p, c_int, c_int, c_int, c_int, c_int, c_int,
                                 c_void_p, c_int, c_void_p, c_void_p, c_void_p, c_size_t,
                                 c_void_p]),
}

_lock = threading.Lock()
_lib = None          # the library the binding calls (release unless debug is on)
_release = None
_debug = None


def header_functions(path: str | None = None):
    """Names of the functions include/qcnn.h declares."""
    path = path or os.path.join(_build.INCLUDE, "qcnn.h")
    text = open(path).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(qcnn_[a-z0-9_]+)\s*\(", text)))


def _bind(so: str):
    lib = ctypes.CDLL(so)
    for name, (res, args) in _SIGS.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    return lib


def load(path: str | None = None):
    """The bound library the binding calls: libqcnn.so (built first when the
    sources are newer), or the debug build after set_debug(True).  With a
    path, bind that file and return it without making it current."""
    global _lib, _release
    with _lock:
        if path is not None:
            return _bind(path)
        if _lib is None:
            _release = _bind(_build.build())
            _lib = _release
        return _lib


def set_debug(enabled: bool):
    """Route every later call of the binding to libqcnn_debug.so (the build
    whose kernels record codes >= K and out-of-range indices, read back by
    device_check) or back to libqcnn.so."""
    global _lib, _release, _debug
    with _lock:
        if enabled:
            if _debug is None:
                _debug = _bind(_build.build_debug())
            _lib = _debug
        else:
            if _release is None:
                _release = _bind(_build.build())
            _lib = _release


def check(status: int, what: str):
    if status != OK:
        lib = load()
        msg = lib.qcnn_status_string(status).decode()
        if status == ERR_CUDA:
            msg += f" (cudaError {lib.qcnn_last_cuda_error()})"
        raise QcnnError(status, what, msg)
