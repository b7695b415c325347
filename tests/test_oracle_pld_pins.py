"""Pins for the prompt-lookup oracle (CPU): hand-worked sequences and brute force.

The paper fixes the matching window N = 6 and the look-ahead L = 2 (Sec. 4.2) and prints no
example, so the oracle is pinned by:
  * sequences worked out by hand (a repeated phrase, a longer match beating a more recent shorter
    one, the most recent of equal matches, a continuation cut by the sequence end, no match);
  * brute force on small random sequences: no suffix longer than the chosen n occurs earlier, the
    chosen occurrence matches, none more recent does, and the draft is its continuation;
  * argmax ties resolved to the lowest index, checked against an explicit scan;
  * the acceptance rule on every prefix length.
"""
import numpy as np
import pytest

from oracle import pld


def test_hand_worked_sequences():
    # "a b c d e a b c" (a=1 ... e=5): the suffix "a b c" (n=3) occurs at 0..2; draft "d e"
    assert pld.draft([1, 2, 3, 4, 5, 1, 2, 3], N=6, L=2) == ([4, 5], 3, 2)
    # a longer match wins over a more recent shorter one: "x y z" at 0..2 (then 7), and "z" alone
    # at 4 (then 8); suffix "x y z"
    assert pld.draft([10, 11, 12, 7, 12, 8, 10, 11, 12], N=6, L=2) == ([7, 12], 3, 2)
    # equal matches: the most recent occurrence of "5 6" (ending at 4, not at 1)
    assert pld.draft([5, 6, 1, 5, 6, 2, 5, 6], N=6, L=2) == ([2, 5], 2, 4)
    # continuation cut by the end of the sequence: "3" last occurs at 2, followed by one token
    assert pld.draft([9, 9, 3, 3], N=6, L=2) == ([3], 1, 2)
    # the window caps n: with N = 2 only the last two tokens are matched
    assert pld.draft([1, 2, 3, 4, 1, 2, 3, 4], N=2, L=2) == ([1, 2], 2, 3)
    # nothing repeats
    assert pld.draft([1, 2, 3, 4], N=6, L=2) == ([], 0, -1)
    # a single token has nothing before it
    assert pld.draft([7], N=6, L=2) == ([], 0, -1)


@pytest.mark.parametrize("seed", range(30))
def test_brute_force_definition(seed):
    rng = np.random.default_rng(seed)
    T = int(rng.integers(2, 60))
    vocab = int(rng.integers(2, 6))
    toks = rng.integers(0, vocab, size=T).tolist()
    N, L = 6, int(rng.integers(1, 4))
    d, n, i = pld.draft(toks, N, L)

    def occurs(m, j):      # the last m tokens occur ending at j (< T - 1)
        return j - m + 1 >= 0 and toks[j - m + 1: j + 1] == toks[T - m:]
    best = max([m for m in range(1, min(N, T - 1) + 1) if any(occurs(m, j) for j in range(T - 1))], default=0)
    assert n == best
    if best == 0:
        assert (d, i) == ([], -1)
        return
    assert occurs(n, i) and not any(occurs(n, j) for j in range(i + 1, T - 1))
    assert d == toks[i + 1: i + 1 + L]


def test_argmax_lowest_index_among_ties():
    x = np.array([[0.0, 3.0, 3.0, -1.0], [5.0, 5.0, 5.0, 5.0], [-2.0, -1.0, -3.0, -1.0]], np.float32)
    got = pld.argmax(x)
    for r, row in enumerate(x):
        best = 0
        for j in range(len(row)):
            if row[j] > row[best]:
                best = j
        assert got[r] == best
    assert got.tolist() == [1, 0, 1]


def test_accept_every_prefix():
    draft = [4, 9]
    assert pld.accept([4, 9, 2], draft) == (2, 2)     # both accepted, then the model's token
    assert pld.accept([4, 7, 2], draft) == (1, 7)     # the second disagrees: the model's 7 follows
    assert pld.accept([3, 9, 2], draft) == (0, 3)     # the first disagrees
    assert pld.accept([5], []) == (0, 5)              # no draft: a plain decode step
