"""Plant one plausible mistake at a time in a private copy of the oracle's C
source (on the CPU) and check that at least one pin catches it.  This shows
the pins constrain every index, sign and term of the oracle's arithmetic."""
import os

import pytest

import oracle
import pins

SRC = open(oracle.SOURCE).read()

MUTANTS = {
    "ky_kx_swapped_in_position": (
        "const int ix = ox * stride - pad + kx;", "const int ix = ox * stride - pad + ky;"),
    "kernel_offset_order_transposed": (
        "const int pk = ky * kw + kx;", "const int pk = kx * kh + ky;"),
    "padding_sign_flipped": (
        "const int ix = ox * stride - pad + kx;", "const int ix = ox * stride + pad + kx;"),
    "stride_dropped": (
        "const int ix = ox * stride - pad + kx;", "const int ix = ox - pad + kx;"),
    "subspaces_interleaved": (
        "acc += s[(i64)(m * Csp + j) * s_stride] * dk[j];",
        "acc += s[(i64)(j * M + m) * s_stride] * dk[j];"),
    "codebook_transposed": (
        "acc += s[(i64)(m * Csp + j) * s_stride] * dk[j];",
        "acc += s[(i64)(m * Csp + j) * s_stride] * D[((i64)m * Csp + j) * K + k];"),
    "fc_codes_transposed": (
        "t += lut[(i64)m * K + codes[(i64)m * Ct + ct]];",
        "t += lut[(i64)m * K + codes[(i64)ct * M + m]];"),
    "conv_codes_layout_wrong": (
        "const int k = codes[((i64)ct * KK + pk) * M + m];",
        "const int k = codes[((i64)ct * M + m) * KK + pk];"),
    "codeword_order_reversed": (
        "t += lut[((i64)m * P + ps) * K + k];", "t += lut[((i64)m * P + ps) * K + (K - 1 - k)];"),
    "last_subspace_dropped": (
        "for (int m = 0; m < M; ++m) {\n                                const int k",
        "for (int m = 0; m < M - 1; ++m) {\n                                const int k"),
    "fc_bias_dropped": (
        "            if (bias) t += bias[ct];\n            if (relu",
        "            if (relu"),
    "conv_relu_before_bias": (
        "                    if (bias) t += bias[ct];\n                    if (relu && t < 0.0) t = 0.0;",
        "                    if (relu && t < 0.0) t = 0.0;\n                    if (bias) t += bias[ct];"),
    "first_input_row_skipped": (
        "if (iy < 0 || iy >= H) continue;", "if (iy <= 0 || iy >= H) continue;"),
    "pool_window_short": (
        "for (int dy = 0; dy < k; ++dy)", "for (int dy = 0; dy < k - 1; ++dy)"),
    "bf16_rounding_truncates": (
        "ldexp(nearbyint(ldexp(f, 8)), e - 8)", "ldexp(trunc(ldexp(f, 8)), e - 8)"),
    "bf16_keeps_nine_bits": (
        "ldexp(nearbyint(ldexp(f, 8)), e - 8)", "ldexp(nearbyint(ldexp(f, 9)), e - 9)"),
    "bf16_flag_ignored": (
        "lut[(i64)m * K + k] = lut_bf16 ? qo_round_bf16(acc) : acc;",
        "lut[(i64)m * K + k] = acc;"),
    "kmeans_argmax": (
        "if (k == 0 || dist < best_d) {", "if (k == 0 || dist > best_d) {"),
    "kmeans_ties_to_last": (
        "if (k == 0 || dist < best_d) {", "if (k == 0 || dist <= best_d) {"),
    "kmeans_l1_distance": (
        "const float sq = diff * diff;", "const float sq = diff < 0 ? -diff : diff;"),
    "kmeans_mean_off_by_one": (
        "(float)(sum[(i64)k * d + j] / (double)cnt[k]);",
        "(float)(sum[(i64)k * d + j] / (double)(cnt[k] + 1));"),
    "kmeans_empty_cluster_divided": (
        "        if (cnt[k] > 0)\n", "        if (cnt[k] >= 0)\n"),
    "kmeans_final_assignment_skipped": (
        "    return kmeans_assign(pts, P, d, K, cen, assign);", "    return QO_OK;"),
    "kmeans_one_round_short": (
        "for (int it = 0; it < iters; ++it) {", "for (int it = 0; it < iters - 1; ++it) {"),
    "pq_conv_offsets_reversed": (
        "W[((i64)ct * Cs + m * Csp + j) * KK + pk];",
        "W[((i64)ct * Cs + m * Csp + j) * KK + (KK - 1 - pk)];"),
    "pq_conv_codes_layout": (
        "codes[p * M + m] = a[p];", "codes[m * P + p] = a[p];"),
    "pq_fc_subvectors_interleaved": (
        "pts[(i64)ct * Csp + j] = W[(i64)ct * Cs + m * Csp + j];",
        "pts[(i64)ct * Csp + j] = W[(i64)ct * Cs + j * M + m];"),
    "lut_dot_product_drops_last_dim": (
        "for (int j = 0; j < Csp; ++j)\n                acc +=",
        "for (int j = 0; j < Csp - 1; ++j)\n                acc +="),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    assert SRC.count(old) == 1, f"mutation site for {name} not unique in the source"
    src = tmp_path / "mutant.c"
    src.write_text(SRC.replace(old, new))
    so = oracle.compile_c(str(src), str(tmp_path / "libmutant.so"))
    fails = pins.run_all(oracle.Oracle(so))
    assert fails, f"no pin caught the planted mistake {name!r}"



@pytest.mark.parametrize("name,old,new", [
    ("bits_msb_first", "out[s // 8] |= 1 << (s % 8)", "out[s // 8] |= 1 << (7 - s % 8)"),
    ("bits_code_bits_reversed", "if (c >> t) & 1:", "if (c >> (b - 1 - t)) & 1:"),
    ("bits_rounded_down", "while (1 << b) < K:", "while (1 << b) <= K // 2 + 1:"),
])
def test_bits_mutant_is_caught(name, old, new, tmp_path, monkeypatch):
    import importlib.util
    import sys

    from oracle import bits
    src = open(bits.__file__).read()
    assert src.count(old) == 1, name
    path = tmp_path / "bits.py"
    path.write_text(src.replace(old, new))
    spec = importlib.util.spec_from_file_location("oracle.bits", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    monkeypatch.setitem(sys.modules, "oracle.bits", mod)
    import oracle as pkg
    monkeypatch.setattr(pkg, "bits", mod, raising=False)
    assert pins.pin_bits(oracle.default()), f"no pin caught {name!r}"
