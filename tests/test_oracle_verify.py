"""Oracle verifier against hand-worked schedules (tests/golden/verify_hand.json)."""
import json
import os

import numpy as np

import oracle
import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "verify_hand.json")


def hand_problem(g, case):
    back = np.asarray(case["back"], np.int32).reshape(-1, 3)
    return W.Problem("hand", g["V"], np.array(g["src"], np.int32), np.array(g["dst"], np.int32),
                     np.array(g["lat"], np.int32), np.array(g["cls"], np.int32), g["C"],
                     np.array(g["limit"], np.float64), np.array(g["demand"], np.int32),
                     np.array(g["bits"], np.int32), D=g["D"], II=case["II"],
                     bsrc=back[:, 0].copy(), bdst=back[:, 1].copy(), bdist=back[:, 2].copy())


def test_verify_hand_worked_cases():
    data = json.load(open(GOLDEN))
    for case in data["cases"]:
        p = hand_problem(data["graph"], case)
        rep = oracle.verify(oracle.OracleProblem(p), case["s"])
        for k, v in case["expect"].items():
            assert rep[k] == v, (case["s"], k, rep[k], v)
