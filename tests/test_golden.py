"""The oracle against the hand-worked fixtures under tests/golden/.

Each fixture states its inputs and the value of every intermediate of
Eqs. 1-17 as exact fractions worked by hand (the arithmetic is shown in the
fixture's comments); the paper itself prints no numeric example.
"""

import math
import os
from fractions import Fraction

import numpy as np

import oracle
from oracle import Params

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _number(tok):
    return float(Fraction(tok)) if "/" in tok else float(tok)


def load_fixture(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            key, rhs = (s.strip() for s in line.split("=", 1))
            vals[key] = [_number(t) for t in rhs.split()]
    return vals


def _hand_worked_inputs(fx):
    a, b = np.array(fx["a"]), np.array(fx["b"])
    N, d = a.size, 4
    k = np.zeros((N, d))
    k[:, 0], k[:, 1] = np.log(a), np.log(b)
    q = np.zeros((1, 2, d))
    q[0, 0, 0] = 2.0     # row 0: logit ln a_i
    q[0, 1, 1] = 2.0     # row 1: logit ln b_i
    p = Params(r=int(fx["r"][0]), m=int(fx["m"][0]), rho=int(fx["rho"][0]),
               gamma=fx["gamma"][0], eps=fx["eps"][0], pool_kernel=int(fx["pool"][0]))
    return q, k, p, int(fx["budget"][0])


def _close(got, want, tol=1e-14):
    np.testing.assert_allclose(np.asarray(got, dtype=float), np.asarray(want, dtype=float),
                               rtol=0, atol=tol)


def test_hand_worked_unit_two_layers():
    fx = load_fixture("hand_worked_unit.txt")
    q, k, p, budget = _hand_worked_inputs(fx)
    N, W = k.shape[0], q.shape[1]
    nc = N - W
    prev = []
    for layer in (0, 1):
        out = oracle.score_unit(q, k, prev, p, budget)
        for name in ("B", "Q", "E", "L"):
            _close(out[name], fx[name])
        _close(out["T"], fx[f"layer{layer}.T"])
        _close(out["V"], fx[f"layer{layer}.V"])
        _close(out["Bt"][:nc], fx["Bt"])
        assert abs(out["lambda"] - fx[f"layer{layer}.lambda"][0]) < 1e-13
        _close(out["S"][:nc], fx[f"layer{layer}.S"])
        idx, gap = oracle.select(out["S"], N, W, budget, p)
        assert idx.tolist() == [int(i) for i in fx[f"layer{layer}.idx"]]
        assert abs(gap - fx[f"layer{layer}.gap"][0]) < 1e-13
        prev = [out["E"]]
    # layer 1's lambda is 2 / sqrt(123), worked in closed form
    assert abs(fx["layer1.lambda"][0] - 2 / math.sqrt(123)) < 1e-16


def test_hand_worked_unit_without_calibration():
    fx = load_fixture("hand_worked_unit.txt")
    q, k, p, budget = _hand_worked_inputs(fx)
    p.gamma = 0.0
    out = oracle.score_unit(q, k, [], p, budget)
    idx, _ = oracle.select(out["S"], k.shape[0], q.shape[1], budget, p)
    assert idx.tolist() == [int(i) for i in fx["layer0.idx_gamma0"]]


def test_oracle_regression_record_tiny_workload():
    """The oracle still produces tiny_oracle.json (make_tiny_regression.py)."""
    import json
    import sys
    sys.path.insert(0, GOLDEN)
    import make_tiny_regression as mk

    with open(os.path.join(GOLDEN, "tiny_oracle.json")) as f:
        want = json.load(f)
    got = mk.compute()
    assert got["workload"] == want["workload"]
    assert got["S_positions"] == want["S_positions"]
    assert len(got["units"]) == len(want["units"]) == 8
    for g, w in zip(got["units"], want["units"]):
        key = (w["request"], w["layer"], w["kv_head"])
        assert (g["request"], g["layer"], g["kv_head"]) == key
        assert g["idx"] == w["idx"], key
        assert abs(g["lambda"] - w["lambda"]) <= 1e-12 * abs(w["lambda"]), key
        assert abs(g["gap"] - w["gap"]) <= 1e-12 * max(abs(w["gap"]), 1e-300) + 1e-18, key
        _close(g["S_sample"], w["S_sample"], 1e-15)
