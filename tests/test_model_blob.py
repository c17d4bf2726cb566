"""Model blob (codes in ceil(log2 K) bits, Table 1 storage) on the CPU:
the C serializer's output read back by an independent Python reader,
storage equal to Table 1's count, and validation of damaged blobs."""
import math
import struct

import numpy as np
import pytest

import paper_1512_06473_gb300 as q
import synth
from oracle import bits
from paper_1512_06473_gb300 import costmodel as cm


def _alexnet_layers():
    w = synth.WORKLOADS["alexnet_qcnn"]
    return w, [synth.oracle_layer_dict(L, P) for L, P in zip(w.layers, w.params())]


def read_blob(blob):
    """Plain reader of the documented layout."""
    assert blob[:8] == b"QCNNMDL1"
    ver, n, C, H, W, _ = struct.unpack_from("<6I", blob, 8)
    recs = []
    for i in range(n):
        f = struct.unpack_from("<12I4Q", blob, 32 + 80 * i)
        recs.append(dict(zip(["kind", "Ct", "kh", "kw", "stride", "pad", "Csp", "K", "relu",
                              "bits", "has_bias", "Cs", "off_D", "off_codes", "off_bias", "r"], f)))
    return ver, (C, H, W), recs, 32 + 80 * n


def test_blob_round_trip_and_storage_model():
    w, layers = _alexnet_layers()
    blob = q.serialize_model(layers, w.in_shape)
    ver, shape, recs, pay = read_blob(blob)
    assert ver == 1 and shape == tuple(w.in_shape) and len(recs) == len(layers)
    for (L, d, r), (sin, sout) in zip(zip(w.layers, layers, recs), w.shapes()):
        if d["kind"] == "maxpool":
            assert (r["kind"], r["kh"], r["stride"]) == (2, L.k, L.s)
            continue
        M, K, Csp = d["D"].shape
        assert r["bits"] == math.ceil(math.log2(K)) and r["K"] == K and r["Csp"] == Csp
        assert r["off_D"] % 16 == 0 and r["off_codes"] % 16 == 0 and r["off_bias"] % 16 == 0
        D = np.frombuffer(blob, np.float32, d["D"].size, pay + r["off_D"]).reshape(d["D"].shape)
        assert np.array_equal(D, d["D"])
        n = d["codes"].size
        nbytes = (n * r["bits"] + 7) // 8
        stream = blob[pay + r["off_codes"]: pay + r["off_codes"] + nbytes]
        assert np.array_equal(bits.unpack(stream, n, r["bits"]), d["codes"].ravel())
        b = np.frombuffer(blob, np.float32, r["Ct"], pay + r["off_bias"])
        assert np.array_equal(b, d["bias"])
        # Table 1: 4 Cs K bytes of sub-codebooks + kk M Ct log2(K) / 8 bytes of codes
        if d["kind"] == "conv":
            c = cm.conv_cost(L.Cs, L.Ct, sin[1], sin[2], L.kh, L.kw, sout[1], sout[2], L.Csp, L.K)
        else:
            c = cm.fc_cost(L.Cs, L.Ct, L.Csp, L.K)
        assert abs((D.nbytes + nbytes) - c.q_bytes) < 1.0


def test_model_info_and_rejections():
    w, layers = _alexnet_layers()
    blob = q.serialize_model(layers, w.in_shape)
    n, shape, dev = q.model_info(blob)
    assert n == len(layers) and shape == tuple(w.in_shape) and dev > len(blob) // 2
    bad = [b"XCNNMDL1" + blob[8:],                     # magic
           blob[:len(blob) - 100],                     # truncated payload
           blob[:40]]                                  # truncated records
    rec0 = bytearray(blob)
    struct.pack_into("<I", rec0, 32 + 9 * 4, 3)        # conv1 bits field (K = 128 needs 7)
    bad.append(bytes(rec0))
    rec1 = bytearray(blob)
    struct.pack_into("<Q", rec1, 32 + 48, 8)           # conv1 off_D not 16-aligned
    bad.append(bytes(rec1))
    rec2 = bytearray(blob)
    struct.pack_into("<I", rec2, 32 + 80 * 2 + 4, 100)  # conv2 Ct changes the chain to fc6
    bad.append(bytes(rec2))
    for b in bad:
        with pytest.raises(q.QcnnError):
            q.model_info(b)


def test_serialize_rejects_bad_layers():
    w, layers = _alexnet_layers()
    broken = [dict(L) for L in layers]
    broken[0]["codes"] = broken[0]["codes"][:, :, :0]    # wrong M
    with pytest.raises((q.QcnnError, ValueError, IndexError)):
        q.serialize_model(broken, (4, 227, 227))          # wrong input channels
