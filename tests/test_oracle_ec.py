"""The error-corrected FC quantizer oracle against its pins, and planted
mistakes (in a private copy of oracle/ec.py) that the pins must catch."""
import importlib.util

import pytest

import oracle
import oracle.ec as ec
import pins_ec

SRC = open(ec.__file__).read()

MUTANTS = {
    "residual_keeps_own_term": ("R = E + A @ old.T", "R = E"),
    "codeword_from_sum_not_mean": ("U[:, Lk].mean(axis=1)", "U[:, Lk].sum(axis=1)"),
    "cost_sign_flipped": ("- 2.0 * (D[m] @ U)", "+ 2.0 * (D[m] @ U)"),
    "cost_drops_quadratic": (
        'cost = np.einsum("kj,ji,ki->k", D[m], G, D[m])[:, None] - 2.0 * (D[m] @ U)',
        "cost = -2.0 * (D[m] @ U)"),
    "targets_not_residual": ("U = A.T @ R", "U = A.T @ T"),
    "residual_not_updated": ("E = R - A @ D[m][codes[m]].T", "E = E"),
    "argmax_assignment": ("codes[m] = np.argmin(cost, axis=0)", "codes[m] = np.argmax(cost, axis=0)"),
    "b_update_before_d_update_skipped": (
        "                    if Lk.size:\n", "                    if False:\n"),
}


@pytest.mark.parametrize("pin", pins_ec.ALL_EC_PINS, ids=lambda p: p.__name__)
def test_ec_pin(pin):
    assert pin(ec, oracle.default()) == []


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_ec_mutant_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    assert SRC.count(old) == 1, name
    path = tmp_path / "ec_mutant.py"
    path.write_text(SRC.replace(old, new))
    spec = importlib.util.spec_from_file_location("ec_mutant", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    assert pins_ec.run_all(mod, oracle.default()), f"no pin caught {name!r}"
