"""Algorithm 2 (endpoint selection, Sec. 8.1): the decision rule against the paper's own
Table "policy" (tests/golden/policy_table.json), and the procedure's stop / drop rules."""
import json
import os

import numpy as np
import pytest

from paper_2608_12114_gb300 import build, policy, synth, wt

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "policy_table.json")))


def times(row):
    return {e: row[e] for e in policy.ENDPOINTS}


@pytest.mark.parametrize("row", GOLD["rows"], ids=[r["platform"] for r in GOLD["rows"]])
def test_rule_reproduces_table_policy(row):
    assert policy.select(times(row), GOLD["theta"]) == row["rule"]


@pytest.mark.parametrize("theta", [0.02, 0.05, 0.1, 0.2])
def test_sensitivity_sweep_changes_no_verdict(theta):
    for row in GOLD["rows"]:
        assert policy.select(times(row), theta) == row["rule"]


def test_gh200_tie_resolves_to_copy_below_its_gap():
    gh = [r for r in GOLD["rows"] if r["platform"].startswith("GH200")][0]
    gap = GOLD["gh200_gap_pct"] / 100
    assert policy.select(times(gh), gap * 0.9) == "copy"
    assert policy.select(times(gh), 0.02) == "map (tie)"


def test_map_never_beats_a_resident_lead_larger_than_theta():
    rng = np.random.default_rng(0)
    for _ in range(2000):
        t = {"map": float(rng.uniform(1, 100)), "resident": float(rng.uniform(1, 100)),
             "copy": float(rng.uniform(1, 100))}
        theta = float(rng.uniform(0.0, 0.3))
        d = policy.select(t, theta)
        best = min(t, key=t.get)
        if (t["map"] - t["resident"]) / t["map"] > theta:
            assert not d.startswith("map")
        if d.startswith("map"):
            assert best == "map" or (t["map"] - t[best]) / t["map"] <= theta
        else:
            assert d == best


def _res(seq):
    it = iter(seq)
    return lambda: next(it)


def test_storage_bound_stop():
    out = policy.run(10, _res([(5, 10)]), {e: (lambda: 1.0) for e in policy.ENDPOINTS})
    assert out.decision == "storage-bound" and out.rates_gbs == {}


def test_capacity_gate_drops_resident():
    m = {"map": lambda: 0.050, "resident": lambda: "allocation failed", "copy": lambda: 0.049}
    out = policy.run(10 ** 9, _res([(10, 10), (10, 10)]), m)
    assert out.times_ms["resident"] is None and "resident" in out.dropped
    assert out.decision == "map (tie)"  # 2 % apart: inside the 5 % band


def test_eviction_after_the_arms_drops_resident():
    m = {"map": lambda: 1.0, "resident": lambda: 0.01, "copy": lambda: 0.9}
    out = policy.run(10 ** 9, _res([(10, 10), (9, 10)]), m)
    assert "resident" in out.dropped and out.decision == "copy"
    keep = policy.run(10 ** 9, _res([(10, 10), (10, 10)]), m)
    assert keep.decision == "resident"
    assert keep.rates_gbs["resident"] == pytest.approx(100.0)


def test_residency_of_a_written_file(tmp_path):
    build.build()
    ck = synth.build("mid", str(tmp_path), layers=1, vocab=300)
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY) as h:
        r, t = h.residency()
        assert t == sum(os.path.getsize(p) for p in ck.paths)
        assert 0 <= r <= t
        for p in ck.paths:  # bring every page in, then ask again
            with open(p, "rb") as f:
                f.read()
        r, t = h.residency()
        assert r == t
