"""The analytic cost model of Sec. 5 against the figures the paper prints in
Tables 2 and 3 and in Sec. 5.1 / 5.3 (tests/golden/paper_cost_figures.json)."""
import json
import math
import os

import pytest

from paper_2010_07565_gb300 import cost_model as cm

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden",
                                     "paper_cost_figures.json")))


def round_sig(x, digits):
    if x == 0:
        return 0.0
    return round(x, -int(math.floor(math.log10(abs(x)))) + (digits - 1))


def dims_of(row):
    d = GOLDEN["datasets"][row["dataset"]]
    return d, [d["features"], row["hidden"], d["classes"]]


@pytest.mark.parametrize("row", GOLDEN["rows"], ids=lambda r: f'{r["dataset"]}-{r["model"]}')
def test_table_figures_reproduce_to_print_precision(row):
    d, dims = dims_of(row)
    dg = row["digits"]
    nw = row.get("weights", 1)
    assert round_sig(cm.model_size_kib(dims, row["binary"], nw), dg["ms"]) == pytest.approx(
        row["ms_kib"], rel=1e-12)
    assert round_sig(cm.data_size_mib(d["N"], d["features"], row["binary"]), dg["ds"]) == \
        pytest.approx(row["ds_mib"], rel=1e-12)
    assert round_sig(cm.cycle_ops(d["N"], d["edges"], dims, row["binary"], nw), dg["co"]) == \
        pytest.approx(row["co"], rel=1e-12)


def test_printed_ratios():
    cora = GOLDEN["datasets"]["Cora"]
    pub = GOLDEN["datasets"]["PubMed"]
    dc_, dp = [cora["features"], 64, 7], [pub["features"], 64, 3]
    co = lambda d, dims, b: cm.cycle_ops(d["N"], d["edges"], dims, b)
    got = {
        "Cora model-size compression, 2 layers":
            cm.model_size_kib(dc_, False) / cm.model_size_kib(dc_, True),
        "Cora S_fe layer 1 (d_in = 1433)": cm.s_fe(1433),
        "Cora S_fe layer 2 (d_in = 64)": cm.s_fe(64),
        "Cora whole-model acceleration (C.O. ratio)": co(cora, dc_, False) / co(cora, dc_, True),
        "Average acceleration over Cora and PubMed":
            0.5 * (co(cora, dc_, False) / co(cora, dc_, True) + co(pub, dp, False) / co(pub, dp, True)),
    }
    for r in GOLDEN["ratios"]:
        assert abs(got[r["what"]] - r["value"]) <= r["tol"], r


def test_closed_forms_agree_with_the_counts():
    """Eq. 16-19's closed forms are the counts' ratios with N cancelled."""
    assert cm.pc(1433) == pytest.approx(cm.model_size_kib([1433, 64], False) /
                                        cm.model_size_kib([1433, 64], True))
    assert cm.dc(500) == pytest.approx(cm.data_size_mib(100, 500, False) /
                                       cm.data_size_mib(100, 500, True))
    N, deg = 1000, 6.0
    full = cm.cycle_ops(N, N * deg / 2, [602, 128], False) / cm.cycle_ops(N, N * deg / 2, [602, 128], True)
    assert cm.s_full(602, deg) == pytest.approx(full)
    assert cm.s_full(602, 0.0) == pytest.approx(cm.s_fe(602))
