"""The routing decision of Sec. 3.2 and Sec. 3.3 (TEST INFRASTRUCTURE ONLY).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference leg may import this
module.  It shares no code with the CUDA path.

The probe model emits one categorical token; from its logits over the category tokens:
  * category c = argmax (lowest index among ties);
  * certainty: the Shannon entropy H = -sum_c p_c ln p_c of the softmax p over the category
    logits (natural logarithm: the paper does not state the base, so this is the reading),
    against the threshold tau = 0.45;
  * model: the 1B model if c is Code Generation, L_ctx <= 2K (2048 tokens) and H <= tau; the 7B
    model otherwise (General QA / Math, long contexts, or H > tau);
  * PLD: on for every request that is not Code Generation (they all go to the 7B model), off for
    Code Generation whichever model serves it.
The entropy is the plain definition evaluated in double: p_c = exp(l_c) / sum_j exp(l_j) (shifted
by the largest logit, which leaves p unchanged and keeps exp finite), H = -sum_c p_c ln p_c over the
p_c > 0 (0 ln 0 = 0).  The threshold compares H <= tau in double.

Parity status: pinned by tests/test_oracle_route_pins.py (closed forms of the entropy and the
decision table of Sec. 3.3).
"""
from __future__ import annotations

import numpy as np

TAU = 0.45
SHORT_CONTEXT = 2048
MODEL_1B, MODEL_7B = 1, 7


def entropy(cat_logits) -> float:
    """Softmax entropy in nats, evaluated in double."""
    l = np.asarray(cat_logits, dtype=np.float64)
    e = np.exp(l - l.max())
    p = e / e.sum()
    nz = p[p > 0]
    return float(-np.sum(nz * np.log(nz)))


def route(cat_logits, code_index: int, L_ctx: int, tau: float = TAU):
    """(category, entropy, model, pld) for one request."""
    l = np.asarray(cat_logits, dtype=np.float64)
    c = int(np.argmax(l))
    H = entropy(l)
    code = c == code_index
    model = MODEL_1B if (code and L_ctx <= SHORT_CONTEXT and H <= float(tau)) else MODEL_7B
    return c, H, model, (not code)
