"""CPU oracle of the prompt-lookup bottom draft (PLD) -- TEST INFRASTRUCTURE ONLY (see oracle/).

CAS-Spec uses prompt lookup decoding as its default bottom draft M_dn (Sec. 4.1, bottom draft
model; Sec. 5.1 setup): a retrieval draft of negligible cost that proposes, as the next tokens, the
tokens that followed an earlier occurrence of the sequence's latest n-gram; a longer matching n-gram
means a more confident draft (Sec. 4.2, token-level information).

Readings (the paper gives no parameters or tie rules; each is also listed in the design notes):
  * the match is the longest n in [n_min, n_max] for which the last n tokens x[L-n:L] occur earlier,
    ending at some position p < L - 1 (so at least one following token exists);
  * among occurrences of that length the most recent one (largest end position p) is used;
  * the draft is x[p+1 : p+1+k], cut at the end of the history; no match gives an empty draft.
"""
from __future__ import annotations


def pld_draft(x: list[int], n_min: int, n_max: int, k: int) -> tuple[int, list[int]]:
    """(match length, drafted tokens) for history x.  A plain scan: for every candidate end
    position p, the length of the common suffix of x[:p+1] and x, capped at n_max."""
    L = len(x)
    best_n, best_p = 0, -1
    for p in range(L - 1):  # p = L - 1 is the suffix itself
        s = 0
        while s < n_max and s <= p and x[p - s] == x[L - 1 - s]:
            s += 1
        if s >= n_min and (s > best_n or (s == best_n and p > best_p)):
            best_n, best_p = s, p
    if best_n == 0:
        return 0, []
    return best_n, list(x[best_p + 1: best_p + 1 + k])
