"""qcnn_fc_forward_noalloc: the FC response for callers that cannot give the
library device memory (a plugin inside a runtime that owns all memory, or a
foreign-function caller without a device allocator).  Its split partial sums
live in a fixed array inside the library instead of a caller workspace.

Checked through the C ABI against qcnn_fc_forward (which takes a workspace),
on two calls in a row so that leftovers of the first call in the shared array
would show up in the second."""
import ctypes

import numpy as np
import pytest
import torch

import synth
from paper_1512_06473_gb300 import _lib

pytestmark = pytest.mark.gpu
TOL = 1e-5
LIMIT = 16 << 20  # QCNN_FC_NOALLOC_SCRATCH_BYTES


def _ws_bytes(lib, N, Cs, Ct, Csp, K):
    nb = ctypes.c_size_t()
    assert lib.qcnn_fc_workspace_size(N, Cs, Ct, Csp, K, 0, ctypes.byref(nb)) == 0
    return nb.value


def _case(seed, N, Cs, Ct, Csp, K):
    M = Cs // Csp
    x = torch.from_numpy(synth.normal((N, Cs), 1.0, seed, 0)).cuda()
    D = torch.from_numpy(synth.normal((M, K, Csp), 0.5, seed, 1)).cuda()
    codes = torch.from_numpy(synth.uniform_codes((M, Ct), K, seed, 2)).cuda()
    bias = torch.from_numpy(synth.normal((Ct,), 0.1, seed, 3)).cuda()
    return x, D, codes, bias


def _with_workspace(lib, x, D, codes, bias, Ct, relu, stream):
    N, Cs = x.shape
    M, K, Csp = D.shape
    nbytes = _ws_bytes(lib, N, Cs, Ct, Csp, K)
    raw = torch.empty(nbytes + 256, dtype=torch.uint8, device="cuda")
    off = (-raw.data_ptr()) % 256
    y = torch.empty((N, Ct), dtype=torch.float32, device="cuda")
    rc = lib.qcnn_fc_forward(x.data_ptr(), N, Cs, Ct, D.data_ptr(), Csp, K, codes.data_ptr(),
                             bias.data_ptr(), y.data_ptr(), int(relu), 0, raw.data_ptr() + off,
                             nbytes, stream)
    assert rc == 0
    return y


def _noalloc(lib, x, D, codes, bias, Ct, relu, stream):
    N, Cs = x.shape
    M, K, Csp = D.shape
    y = torch.full((N, Ct), float("nan"), dtype=torch.float32, device="cuda")
    rc = lib.qcnn_fc_forward_noalloc(x.data_ptr(), N, Cs, Ct, D.data_ptr(), Csp, K,
                                     codes.data_ptr(), bias.data_ptr(), y.data_ptr(), int(relu),
                                     stream)
    assert rc == 0, lib.qcnn_status_string(rc)
    return y


@pytest.mark.parametrize("shape", [(8, 9216, 4096, 4, 32), (8, 512, 256, 4, 16)])
def test_noalloc_matches_workspace_entry_point_twice(shape):
    lib = _lib.load()
    N, Cs, Ct, Csp, K = shape
    need = _ws_bytes(lib, *shape)
    assert 0 < need <= LIMIT, "the case must use the fixed scratch and fit in it"
    stream = torch.cuda.current_stream().cuda_stream
    for call, seed in enumerate((101, 202)):  # two calls in a row, different data
        x, D, codes, bias = _case(seed, *shape)
        relu = call == 1
        ref = _with_workspace(lib, x, D, codes, bias, Ct, relu, stream)
        got = _noalloc(lib, x, D, codes, bias, Ct, relu, stream)
        torch.cuda.synchronize()
        r, g = ref.cpu().numpy(), got.cpu().numpy()
        assert np.all(np.isfinite(g))
        assert np.max(np.abs(g - r)) / np.max(np.abs(r)) <= TOL


def test_noalloc_runs_cases_whose_split_sums_exceed_its_scratch():
    """fc6 at batch 128: qcnn_fc_forward splits the sub-spaces so far that the
    partial sums outgrow the fixed scratch; the no-alloc call plans fewer
    splits and still matches."""
    lib = _lib.load()
    shape = (128, 9216, 4096, 4, 32)
    assert _ws_bytes(lib, *shape) > LIMIT, "the case must exceed the fixed scratch"
    stream = torch.cuda.current_stream().cuda_stream
    x, D, codes, bias = _case(303, *shape)
    ref = _with_workspace(lib, x, D, codes, bias, shape[2], True, stream)
    got = _noalloc(lib, x, D, codes, bias, shape[2], True, stream)
    torch.cuda.synchronize()
    r, g = ref.cpu().numpy(), got.cpu().numpy()
    assert np.all(np.isfinite(g))
    assert np.max(np.abs(g - r)) / np.max(np.abs(r)) <= TOL
