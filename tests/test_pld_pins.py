"""Pins of the prompt-lookup bottom-draft oracle (PLD, the default bottom draft M_dn of Sec. 4.1 /
Sec. 5.1) against hand-worked histories and a brute force over n-gram slices (no GPU)."""
from __future__ import annotations

import random

import pytest

from oracle import pld_oracle as O


def _slices(x, n_min, n_max, k):
    """Longest n first; the latest earlier start i with x[i:i+n] == x[-n:] and a token after it."""
    L = len(x)
    for n in range(min(n_max, L - 1), n_min - 1, -1):
        starts = [i for i in range(0, L - n) if x[i:i + n] == x[L - n:]]
        if starts:
            i = max(starts)
            return n, x[i + n:i + n + k]
    return 0, []


def test_hand_worked_histories():
    assert O.pld_draft([1, 2, 3, 4, 1, 2, 3], 1, 3, 2) == (3, [4, 1])
    # two earlier occurrences of the final bigram: the later one (followed by 8) wins
    assert O.pld_draft([5, 6, 7, 5, 6, 8, 5, 6], 1, 3, 3) == (2, [8, 5, 6])
    assert O.pld_draft([1, 2, 3], 1, 3, 4) == (0, [])  # the last token never occurred before
    # overlapping occurrences in a run; the draft is cut at the end of the history
    assert O.pld_draft([7, 7, 7, 7], 1, 2, 5) == (2, [7])
    # a match shorter than n_min does not count
    assert O.pld_draft([4, 9, 1, 4], 2, 4, 3) == (0, [])
    assert O.pld_draft([4, 9, 1, 4], 1, 4, 3) == (1, [9, 1, 4])


@pytest.mark.parametrize("seed", range(20))
def test_matches_slice_brute_force(seed):
    r = random.Random(seed)
    L = r.randint(1, 200)
    vocab = r.choice([2, 3, 5, 50])
    x = [r.randrange(vocab) for _ in range(L)]
    n_min = r.randint(1, 3)
    n_max = r.randint(n_min, 6)
    k = r.randint(0, 8)
    assert O.pld_draft(x, n_min, n_max, k) == _slices(x, n_min, n_max, k)
