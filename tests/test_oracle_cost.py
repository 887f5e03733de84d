"""Pins for oracle.cost against the R1 / R2 values the paper prints
(tests/golden/paper_ratios.json: Table 1, Table 2, Sec. 4.1-4.2) -- CPU only."""
import json
import os

import pytest

from oracle import cost

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_ratios.json")))


@pytest.mark.parametrize("row", GOLD["rows"], ids=lambda r: f"{r['method']}-{r['R1']}-{r['R2']}")
def test_printed_ratios(row):
    """The printed R2 fixes r/E; the cost model must then give the printed R1
    (to the table's rounding)."""
    E, L = 4096, 1000
    w_bits, a_bits = row["E_bits"]
    R2 = row["R2"] / 100
    if row["method"] == "qsvd":
        r = 2 * E * R2 * 16 / a_bits                  # eta_qsvd / eta_fp = r / (2E)
        R1m, R2m = cost.ratios_qsvd(E, r, w_bits, a_bits, L)
    elif row["method"] == "kv_only":
        r = E * R2                                    # eta_ind / eta_fp = r / E
        R1m, R2m = cost.ratios_kv_only(E, r, L)
    else:                                             # full KV cache at a_bits
        R1m, R2m = None, cost.eta_fp(E, L) * a_bits / 16 / cost.eta_fp(E, L)
    assert R2m == pytest.approx(R2, abs=5e-5)
    if row["R1"] is not None:
        assert 100 * R1m == pytest.approx(row["R1"], abs=0.051)


def test_cost_identities():
    E, r, L = 4096, 1536, 777
    # Sec. 3.1: the R1 of weights equals the R1 of FLOPs
    assert cost.alpha_qsvd(E, r) / cost.alpha_fp(E) == pytest.approx(
        cost.gamma_qsvd(E, r, L) / cost.gamma_fp(E, L))
    assert cost.alpha_ind(E, r) / cost.alpha_fp(E) == pytest.approx(
        cost.gamma_ind(E, r, L) / cost.gamma_fp(E, L))
    # QSVD beats the original exactly when r < 0.75 E, and always beats per-matrix SVD
    assert cost.alpha_qsvd(E, 3071) < cost.alpha_fp(E) <= cost.alpha_qsvd(E, 3072)
    assert cost.eta_qsvd(r, L) < cost.eta_ind(r, L) and cost.alpha_qsvd(E, r) < cost.alpha_ind(E, r)
