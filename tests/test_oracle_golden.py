"""The oracle still reproduces its frozen vectors (tests/golden/oracle_vectors.json).

Those values were written by tests/golden/make_golden.py, which calls only the
oracle; the GEMV case is also checked against exact integer arithmetic here."""
import json
import os

import numpy as np

import oracle
from tests.golden import make_golden

GOLD = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "oracle_vectors.json")


def test_digest_vectors():
    g = json.load(open(GOLD))["digests"]
    for k, b in make_golden.patterns().items():
        assert g[k]["n"] == len(b)
        assert "%016x" % oracle.fnv1a64(b) == g[k]["plain"]
        assert "%016x" % oracle.fnv_tree(b) == g[k]["tree"]


def test_gemv_vector_and_exact_integers():
    g = json.load(open(GOLD))["gemv"]
    W, x = make_golden.gemv_case()
    assert g["W"] == W and g["x"] == x
    exact = [sum(w * v for w, v in zip(row, x)) for row in W]
    assert g["yhat"] == exact
    yhat, a = oracle.gemv(np.frombuffer(make_golden.bf16_bytes(sum(W, [])), np.uint8), 1, 5, 8,
                          np.frombuffer(make_golden.bf16_bytes(x), np.uint8))
    assert list(yhat) == g["yhat"] and list(a) == g["a"]
