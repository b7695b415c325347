"""Prompt-lookup decoding around the verification pass (TEST INFRASTRUCTURE ONLY).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference leg may import this
module.  It shares no code with the CUDA path.  Plain Python over small integer lists.

What it computes (Sec. 4.2 fixes the n-gram matching window N = 6 and the look-ahead L = 2; the
paper prints no algorithm, so the steps below are the reading):

  draft(tokens, N, L)
      For n = N, N-1, ..., 1: the last n tokens form the query.  Look for an earlier occurrence
      of it: an index i (the occurrence's last token) with i < T - 1 and tokens[i-n+1 .. i] equal
      to tokens[T-n .. T-1].  Among the occurrences of the longest n that has one, take the most
      recent (largest i).  The draft is the up to L tokens that follow it, tokens[i+1 .. i+L],
      cut at the end of the sequence.  No occurrence for any n: an empty draft.

  argmax(logits)  per row, the lowest index among equal maxima.

  accept(argmax_rows, draft)
      The verification pass scores the last committed token followed by the d drafted tokens
      (d + 1 rows; row j predicts the token after position j).  Greedy acceptance keeps the
      longest prefix of the draft that agrees with the model, a = max{k : argmax[j] == draft[j]
      for all j < k}, and the model's own next token argmax[a] follows it: a + 1 tokens commit.

Parity status: pinned by tests/test_oracle_pld_pins.py (hand-worked sequences, brute force over
every suffix length and position on small random sequences, ties, empty drafts).
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

import numpy as np


def suffix_match(tokens: Sequence[int], i: int, N: int) -> int:
    """Length (<= N) of the common suffix of tokens[..i] and the whole sequence."""
    T = len(tokens)
    n = 0
    while n < N and i - n >= 0 and tokens[i - n] == tokens[T - 1 - n]:
        n += 1
    return n


def draft(tokens: Sequence[int], N: int = 6, L: int = 2) -> Tuple[List[int], int, int]:
    """(draft tokens, matched n, index i of the occurrence's last token); ([], 0, -1) if none."""
    T = len(tokens)
    for n in range(N, 0, -1):
        if n > T - 1:
            continue
        for i in range(T - 2, n - 2, -1):          # most recent first; i < T - 1
            if all(tokens[i - k] == tokens[T - 1 - k] for k in range(n)):
                return list(tokens[i + 1: min(i + 1 + L, T)]), n, i
    return [], 0, -1


def argmax(logits: np.ndarray) -> np.ndarray:
    """Row-wise argmax, lowest index among ties (numpy's argmax returns the first maximum)."""
    return np.argmax(np.asarray(logits), axis=-1).astype(np.int32)


def accept(argmax_rows: Sequence[int], draft_tokens: Sequence[int]) -> Tuple[int, int]:
    """(accepted draft tokens a, the model's next token argmax_rows[a])."""
    a = 0
    while a < len(draft_tokens) and argmax_rows[a] == draft_tokens[a]:
        a += 1
    return a, int(argmax_rows[a])
