"""Pins of the oracle's outer loop of Alg. GauS (Sec. 3.3 Initialization and
Sampling; App. A, reset to the prior best) on a three-node chain whose bounds,
scores and legalizations are worked by hand:

    0 -> 1 -> 2, unit latencies, D = 5, one unlimited class, unit demand
    ASAP = (0, 1, 2), ALAP = (2, 3, 4), slack 2 everywhere.
"""
import numpy as np

import oracle
import workloads as W

TERMS = W.DEP | W.COM | W.RES_OBJ


def chain(D=5):
    i32 = lambda x: np.asarray(x, np.int32)
    return W.Problem(name="chain3", V=3, src=i32([0, 1]), dst=i32([1, 2]), lat=i32([1, 1, 1]),
                     cls=i32([0, 0, 0]), C=1, limit=np.array([np.inf]), demand=i32([1, 1, 1]),
                     bits=i32([1, 1, 1]), D=D)


def fresh(op, mu):
    V, B = mu.shape
    si = np.full((V, B), np.float32(0.5))
    state = dict(mu=mu.astype(np.float32).copy(), sigma=np.full((V, B), np.float32(2.0)),
                 m_mu=np.ones((V, B), np.float32), v_mu=np.ones((V, B), np.float32),
                 m_sigma=np.ones((V, B), np.float32), v_sigma=np.ones((V, B), np.float32),
                 step=np.full(B, 7, np.int32))
    best = dict(sched=np.zeros((V, B), np.int32), score=np.full(B, np.inf), iter=np.full(B, -1, np.int32))
    return state, best, si


def test_init_state_closed_form():
    op = oracle.OracleProblem(chain())
    mu, sg = oracle.init_state(op, 2, 1.0 / 6.0, 0.05)
    # midpoints of [ASAP, ALAP]; sigma = kappa * slack (kappa the float32 1/6, product in double)
    np.testing.assert_array_equal(mu[:, 0], np.float32([1, 2, 3]))
    assert sg[0, 0] == np.float32(float(np.float32(1.0 / 6.0)) * 2.0)
    assert abs(float(sg[0, 0]) - 1.0 / 3.0) < 1e-7
    # a given mu0 is kept
    mu0 = np.float32([[0.25, 1], [1.5, 2], [2.75, 3]])
    mu, _ = oracle.init_state(op, 2, 1.0 / 6.0, 0.05, mu0=mu0)
    np.testing.assert_array_equal(mu, mu0)
    # no slack (D = critical path): sigma falls back to sigma_min
    op3 = oracle.OracleProblem(chain(D=3))
    _, sg = oracle.init_state(op3, 1, 1.0 / 6.0, 0.05)
    np.testing.assert_array_equal(sg[:, 0], np.float32([0.05, 0.05, 0.05]))


def test_legal_first_candidate_becomes_best_without_reset():
    op = oracle.OracleProblem(chain())
    state, best, si = fresh(op, np.float32([[1.2], [2.4], [2.6]]))      # rounds to (1, 2, 3): legal
    moved = oracle.outer_step(op, TERMS, 1.0, 1.0, 1.0, 100, np.int32([[1], [2], [3]]), [1], si, best, state)
    assert moved[0] == 0
    # one node per step: peak usage 1; L_com = (2 - 1) + (3 - 2) = 2; score 3
    assert best["score"][0] == 3.0 and best["iter"][0] == 100
    np.testing.assert_array_equal(best["sched"][:, 0], [1, 2, 3])
    np.testing.assert_array_equal(state["mu"][:, 0], np.float32([1.2, 2.4, 2.6]))  # no reset
    assert state["step"][0] == 7 and state["m_mu"][0, 0] == 1.0


def test_illegal_without_improvement_resets_to_prior_best():
    op = oracle.OracleProblem(chain())
    state, best, si = fresh(op, np.float32([[1.2], [1.4], [2.6]]))      # rounds to (1, 1, 3): node 1 too early
    best["sched"][:, 0] = [0, 2, 4]
    best["score"][0] = 2.0
    best["iter"][0] = 50
    # Alg. 1: clamp to [ASAP, ALAP] keeps (1, 1, 3); the forward pass moves node 1 to 2
    moved = oracle.outer_step(op, TERMS, 1.0, 1.0, 1.0, 100, np.int32([[1], [2], [3]]), [1], si, best, state)
    assert moved[0] == 1
    assert best["score"][0] == 2.0 and best["iter"][0] == 50            # score 3 does not improve on 2
    np.testing.assert_array_equal(state["mu"][:, 0], np.float32([0, 2, 4]))   # the prior best
    np.testing.assert_array_equal(state["sigma"][:, 0], si[:, 0])
    for k in ("m_mu", "v_mu", "m_sigma", "v_sigma"):
        assert not state[k].any()
    assert state["step"][0] == 0


def test_illegal_with_improvement_resets_to_the_legalized_schedule():
    op = oracle.OracleProblem(chain())
    state, best, si = fresh(op, np.float32([[1.2], [1.4], [2.6]]))
    best["score"][0] = 5.0
    best["iter"][0] = 50
    moved = oracle.outer_step(op, TERMS, 1.0, 1.0, 1.0, 100, np.int32([[1], [2], [3]]), [1], si, best, state)
    assert moved[0] == 1
    assert best["score"][0] == 3.0 and best["iter"][0] == 100
    np.testing.assert_array_equal(state["mu"][:, 0], np.float32([1, 2, 3]))
    assert state["step"][0] == 0


def test_failed_legalization_without_best_resets_to_the_midpoint():
    op = oracle.OracleProblem(chain())
    state, best, si = fresh(op, np.float32([[np.nan], [2.0], [3.0]]))
    moved = oracle.outer_step(op, TERMS, 1.0, 1.0, 1.0, 100, np.int32([[0], [1], [2]]), [0], si, best, state)
    assert moved[0] == -1
    assert best["iter"][0] == -1 and np.isinf(best["score"][0])
    np.testing.assert_array_equal(state["mu"][:, 0], np.float32([1, 2, 3]))   # (ASAP + ALAP) / 2


def test_infeasible_candidate_is_not_kept_and_a_legal_rounding_is_not_reset():
    op = oracle.OracleProblem(chain())
    state, best, si = fresh(op, np.float32([[2.0], [3.0], [5.0]]))      # node 2 ends at 6 > D = 5
    moved = oracle.outer_step(op, TERMS, 1.0, 1.0, 1.0, 100, np.int32([[2], [3], [5]]), [1], si, best, state)
    assert moved[0] == 0
    assert best["iter"][0] == -1
    np.testing.assert_array_equal(state["mu"][:, 0], np.float32([2, 3, 5]))
    assert state["step"][0] == 7


def test_score_weights_and_terms():
    # alpha and the weights scale their terms; the ReLU resource term makes an
    # over-limit schedule a non-candidate
    i32 = lambda x: np.asarray(x, np.int32)
    p = W.Problem(name="pair", V=2, src=i32([]), dst=i32([]), lat=i32([1, 1]), cls=i32([0, 0]), C=1,
                  limit=np.array([1.0]), demand=i32([1, 1]), bits=i32([1, 1]), D=3)
    op = oracle.OracleProblem(p)
    mu = np.float32([[0.0], [0.0]])                                      # both at step 0: usage 2 > limit 1
    state, best, si = fresh(op, mu)
    oracle.outer_step(op, W.RES_OBJ | W.COM, 2.5, 1.0, 1.0, 10, np.int32([[0], [0]]), [1], si, best, state)
    assert best["score"][0] == 2.5 * 2                                   # w_res * peak, no edges
    state, best, si = fresh(op, mu)
    oracle.outer_step(op, W.RES_OBJ | W.RES_VIOL, 1.0, 1.0, 1.0, 10, np.int32([[0], [0]]), [1], si, best, state)
    assert best["iter"][0] == -1


def test_illegal_without_best_takes_the_legalized_schedule():
    # Alg. GauS: mu <- legalize(s) when s is illegal; with no prior best to return to,
    # the legalized schedule is taken even when it is no candidate.  Nodes 0 -> 1 and
    # an independent node 2, one step per class of limit 1, D = 4:
    # ASAP = (0, 1, 0), ALAP = (2, 3, 3).  round(mu) = (1, 1, 2) violates 0 -> 1;
    # Alg. 1 gives (1, 2, 2), where nodes 1 and 2 share step 2: usage 2 > 1.
    i32 = lambda x: np.asarray(x, np.int32)
    p = W.Problem(name="tri", V=3, src=i32([0]), dst=i32([1]), lat=i32([1, 1, 1]), cls=i32([0, 0, 0]), C=1,
                  limit=np.array([1.0]), demand=i32([1, 1, 1]), bits=i32([1, 1, 1]), D=4)
    op = oracle.OracleProblem(p)
    rc, order, asap, alap, cp = oracle.asap_alap(op)
    np.testing.assert_array_equal(asap, [0, 1, 0])
    np.testing.assert_array_equal(alap, [2, 3, 3])
    s_legal = oracle.legalize_regular(op, order, asap, alap, np.int32([1, 1, 2]))
    np.testing.assert_array_equal(s_legal, [1, 2, 2])
    state, best, si = fresh(op, np.float32([[1.2], [0.6], [2.4]]))      # rounds to (1, 1, 2)
    terms = W.DEP | W.RES_OBJ | W.RES_VIOL
    moved = oracle.outer_step(op, terms, 1.0, 1.0, 1.0, 100, s_legal[:, None], [1], si, best, state)
    assert moved[0] == 1
    assert best["iter"][0] == -1                                         # over the limit: no candidate
    np.testing.assert_array_equal(state["mu"][:, 0], np.float32([1, 2, 2]))
    assert state["step"][0] == 0
