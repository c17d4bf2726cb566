"""The error-corrected conv quantizer oracle (Appendix B) against its pins,
and planted mistakes (in a private copy of oracle/ec_conv.py) that the pins
must catch."""
import importlib.util

import pytest

import oracle.ec as ec
import oracle.ec_conv as ecc
import pins_ec_conv

SRC = open(ecc.__file__).read()

MUTANTS = {
    "codeword_target_ignores_other_codewords": (
        'Q = Ecur + np.einsum("j,ncjyx->ncyx", D[m, k], Z)   # Eq. B.5', "Q = R.copy()"),
    "residual_not_updated_after_codeword": (
        'Ecur = Q - np.einsum("j,ncjyx->ncyx", D[m, k], Z)', "Ecur = Ecur"),
    "assignment_cost_sign": ("- 2.0 * (D[m] @ U)", "+ 2.0 * (D[m] @ U)"),
    "assignment_target_drops_own_offset": (
        'P = Ecur + np.einsum("cj,njyx->ncyx", D[m][cm[:, pk]], Xp)   # Eq. B.7', "P = Ecur"),
    "offset_index_transposed": ("X[ky * kw + kx] = Ap", "X[kx * kh + ky] = Ap"),
    "stride_ignored": ("ky:ky + stride * (Ho - 1) + 1:stride", "ky:ky + Ho"),
    "sweep_residual_not_carried": ("            E = Ecur\n", "            E = R\n"),
    "codeword_update_skipped": ("                    if not mask.any():\n", "                    if True:\n"),
}


@pytest.mark.parametrize("pin", pins_ec_conv.ALL_ECC_PINS, ids=lambda p: p.__name__)
def test_ecc_pin(pin):
    assert pin(ecc, ec) == []


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_ecc_mutant_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    assert SRC.count(old) == 1, name
    path = tmp_path / "ecc_mutant.py"
    path.write_text(SRC.replace(old, new))
    spec = importlib.util.spec_from_file_location("ecc_mutant", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    assert pins_ec_conv.run_all(mod, ec), f"no pin caught {name!r}"
