"""Pins for the routing oracle (CPU): closed forms of the softmax entropy and the decision table of
Sec. 3.3 (Code Generation with a short context and a confident probe goes to the 1B model without
PLD; long contexts and uncertain probes go to the 7B model; General QA and Math go to the 7B model
with PLD)."""
import math

import numpy as np

from oracle import route

CODE, QA, MATH = 0, 1, 2


def test_entropy_closed_forms():
    # the oracle evaluates the definition in double: closed forms hold to a few double ulps
    assert abs(route.entropy([0.0, 0.0, 0.0]) - math.log(3)) < 1e-15          # uniform: ln n
    assert abs(route.entropy([0.0] * 32) - math.log(32)) < 1e-14
    assert route.entropy([0.0, -200.0, -200.0]) < 1e-80                       # one certain category
    h = route.entropy([math.log(3), 0.0])                                     # p = (3/4, 1/4)
    assert abs(h - (-(0.75 * math.log(0.75) + 0.25 * math.log(0.25)))) < 1e-15
    assert route.entropy([5.0, 5.0, 5.0]) == route.entropy([0.0, 0.0, 0.0])   # shift invariant
    # two categories with logit gap g: p = 1 / (1 + e^-g), H = ln(1 + e^-g) + g e^-g / (1 + e^-g)
    for g in (0.5, 2.0, 2.7, 9.0):
        eg = math.exp(-g)
        assert abs(route.entropy([g, 0.0]) - (math.log1p(eg) + g * eg / (1 + eg))) < 1e-15


def test_decision_table():
    confident_code = [4.0, 0.0, 0.0]     # H ~ 0.07 nats
    uncertain_code = [0.5, 0.0, 0.0]     # H ~ 1.07 nats
    assert route.route(confident_code, CODE, 2048)[2:] == (route.MODEL_1B, False)
    assert route.route(confident_code, CODE, 2049)[2:] == (route.MODEL_7B, False)   # long context
    assert route.route(uncertain_code, CODE, 100)[2:] == (route.MODEL_7B, False)    # uncertain
    assert route.route([0.0, 4.0, 0.0], CODE, 100)[2:] == (route.MODEL_7B, True)    # General QA
    assert route.route([0.0, 0.0, 4.0], CODE, 100)[2:] == (route.MODEL_7B, True)    # Math
    assert route.route([0.0, 0.0, 4.0], CODE, 32768)[2:] == (route.MODEL_7B, True)


def test_threshold_is_inclusive():
    # p = (1 - 2e, e, e): find logits whose entropy straddles 0.45
    lo, hi = route.route([2.75, 0.0, 0.0], CODE, 10), route.route([2.65, 0.0, 0.0], CODE, 10)
    assert lo[1] <= route.TAU < hi[1]
    assert lo[2] == route.MODEL_1B and hi[2] == route.MODEL_7B
    c, H, model, pld = route.route([1.0, 1.0, 0.0], CODE, 10)
    assert c == CODE   # ties go to the lowest index
