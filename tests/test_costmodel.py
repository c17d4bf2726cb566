"""Table 1 cost model against the speed-up and compression figures the paper
prints (tests/golden/paper_tables.json, each entry cites its table)."""
import json
import os

import pytest

from paper_1512_06473_gb300 import costmodel as cm

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_tables.json")))


def _rows(key):
    return [tuple(r) for r in GOLD[key]["rows"]]


@pytest.mark.parametrize("csp,K,want", _rows("alexnet_conv2_speedup"))
def test_table4_conv2_speedup(csp, K, want):
    c = cm.conv_cost(96, 256, 27, 27, 5, 5, 27, 27, csp, K, groups=2)
    assert round(c.dense_macs / c.q_macs, 2) == want


@pytest.mark.parametrize("csp,K,want", _rows("alexnet_all_conv_speedup"))
def test_table5_alexnet_conv_speedup(csp, K, want):
    assert round(cm.speedup(cm.alexnet_grouped(csp, K, [])), 2) == want


@pytest.mark.parametrize("csp,K,want", _rows("caffenet_fc6_compression"))
def test_table6_fc6_compression(csp, K, want):
    c = cm.fc_cost(9216, 4096, csp, K)
    assert round(c.dense_bytes / c.q_bytes, 2) == want


@pytest.mark.parametrize("csp,K,want", _rows("caffenet_all_fc_compression"))
def test_table7_all_fc_compression(csp, K, want):
    L = [cm.fc_cost(9216, 4096, csp, K), cm.fc_cost(4096, 4096, csp, K), cm.fc_cost(4096, 1000, 1, 16)]
    assert round(cm.compression(L), 2) == want


@pytest.mark.parametrize("csp,K,want", _rows("alexnet_whole_net_speedup"))
def test_table8_whole_net_speedup(csp, K, want):
    L = cm.alexnet_grouped(8, 128, [(csp, K), (csp, K), (1, 16)])
    assert round(cm.speedup(L), 2) == want


def test_layer_counts_are_consistent():
    # look-ups = Ho Wo Ct kh kw M, table entries = H W M K, for one image
    c = cm.conv_cost(64, 64, 56, 56, 3, 3, 56, 56, 4, 128)
    assert c.lookups == 56 * 56 * 64 * 9 * 16
    assert c.lut_entries == 56 * 56 * 16 * 128
    assert c.lut_macs == c.lut_entries * 4
    f = cm.fc_cost(9216, 4096, 4, 32)
    assert f.lookups == 4096 * 2304 and f.lut_entries == 2304 * 32
