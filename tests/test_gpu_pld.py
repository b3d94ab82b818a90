"""casspec_pld_draft (the prompt-lookup bottom draft, Sec. 4.1 / 4.2) against the PLD oracle:
bit-exact match length, count and tokens, on seeded histories from empty to 60k tokens."""
from __future__ import annotations

import random

import numpy as np
import pytest
import torch

from oracle import pld_oracle as O

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cs():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2510_26843_gb300 as m

    m.load_library()
    return m


def _run(cs, x, n_min, n_max, k):
    t = torch.tensor(np.asarray(x, dtype=np.int32), device="cuda") if len(x) else torch.zeros(1, dtype=torch.int32,
                                                                                             device="cuda")
    out = torch.full((2 + k,), -7, dtype=torch.int32, device="cuda")
    cs.pld_draft(t, len(x), n_min, n_max, k, out)
    torch.cuda.synchronize()
    o = out.cpu().tolist()
    return o[0], o[2:2 + o[1]], o[2 + o[1]:]


@pytest.mark.parametrize("seed", range(24))
def test_pld_matches_oracle(cs, seed):
    r = random.Random(seed)
    L = r.choice([0, 1, 2, 17, 300, 1023, 1024, 1025, 4096, 60000])
    vocab = r.choice([2, 4, 32, 32000])
    x = [r.randrange(vocab) for _ in range(L)]
    n_min = r.randint(1, 3)
    n_max = r.choice([n_min, 4, 8, 64])
    k = r.choice([0, 1, 5, 64])
    n, toks, rest = _run(cs, x, n_min, n_max, k)
    assert (n, toks) == O.pld_draft(x, n_min, n_max, k)
    assert all(v == -7 for v in rest)  # nothing written past the drafted tokens


def test_pld_on_repeated_text(cs):
    # a history that repeats a 40-token phrase: the draft continues the phrase with the longest match
    r = random.Random(5)
    phrase = [r.randrange(1000) for _ in range(40)]
    x = [r.randrange(1000) for _ in range(200)] + phrase + [r.randrange(1000) for _ in range(50)] + phrase[:25]
    n, toks, _ = _run(cs, x, 1, 8, 10)
    assert n == 8 and toks == phrase[25:35]


def test_pld_rejects_bad_arguments(cs):
    t = torch.zeros(8, dtype=torch.int32, device="cuda")
    out = torch.zeros(4, dtype=torch.int32, device="cuda")
    for args in [(8, 0, 2, 2), (8, 3, 2, 2), (8, 1, 65, 2), (-1, 1, 2, 2), (8, 1, 2, -1)]:
        with pytest.raises(cs.CasspecError):
            cs.pld_draft(t, *args, out)
