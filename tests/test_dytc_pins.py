"""Pins of the DyTC scheduler oracle (Sec. 3 EWIF closed forms, Sec. 4.2 EMA / Eq. 5 / Algorithm 1,
App. D Algorithm 2) against what the paper prints and what exact enumeration gives (no GPU).

Each check compares the oracle with something other than its own formula: the paper's worked
example (Sec. 4.2: EWIF 1.554 greedy vs 1.615 horizontal cascade, local speedups 2.25 and 2.67),
exact enumeration of the Bernoulli acceptance processes with rational arithmetic, the closed form of
an EMA under a constant outcome stream, and invariants of the tree construction.
"""
from __future__ import annotations

import itertools
import math
from fractions import Fraction

import pytest

from oracle import dytc_oracle as D


# ------------------------------------------------------------------------------------------------
# Sec. 4.2 worked example
# ------------------------------------------------------------------------------------------------
def test_worked_example_greedy_vs_horizontal_cascade():
    # two drafts: d1 (alpha 0.9, c 0.4), d2 (alpha 0.8, c 0.3)
    t_d2, k_d2 = D.best_sd(0.8, 0.3, 16)
    assert round(t_d2, 3) == 1.554 and k_d2 == 3
    t_hc, k1, k2 = D.best_hc(0.9, 0.4, 0.8, 0.3, 16)
    assert round(t_hc, 3) == 1.615 and (k1, k2) == (2, 2)
    # local speedups of the first step at k = 1 (no future term): 0.9 / 0.4 and 0.8 / 0.3
    assert D.step_objective(0.9, 0.4, 1, 0.0, 0.0) == pytest.approx(2.25)
    assert round(D.step_objective(0.8, 0.3, 1, 0.0, 0.0), 2) == 2.67
    # the greedy local choice is d2 (at k = 1), as the paper states
    s, k, _ = D.find_best_config([0.9, 0.8], [0.4, 0.3], 0.0, 0.0, 8)
    assert (s, k) == (1, 1)


# ------------------------------------------------------------------------------------------------
# Sec. 3 closed forms against exact enumeration
# ------------------------------------------------------------------------------------------------
def _round_tokens_dist(a: Fraction, k: int) -> dict[int, Fraction]:
    """Distribution of the tokens one round yields: i accepted drafts then the bonus/correction."""
    d = {}
    for outcome in itertools.product([0, 1], repeat=k):
        p = Fraction(1)
        for o in outcome:
            p *= a if o else 1 - a
        acc = 0
        for o in outcome:
            if not o:
                break
            acc += 1
        d[acc + 1] = d.get(acc + 1, Fraction(0)) + p
    return d


@pytest.mark.parametrize("a,c,k", [(Fraction(4, 5), Fraction(3, 10), 3), (Fraction(1, 3), Fraction(1, 20), 5),
                                   (Fraction(9, 10), Fraction(2, 5), 1)])
def test_sd_ewif_equals_enumerated_expectation(a, c, k):
    dist = _round_tokens_dist(a, k)
    expect = sum(i * p for i, p in dist.items()) / (c * k + 1)
    assert D.ewif_sd(float(a), float(c), k) == pytest.approx(float(expect), rel=1e-12)
    # and the derivative at 1 of the generating function
    h = 1e-6
    dphi = (D.pgf_sd(float(a), k, 1 + h) - D.pgf_sd(float(a), k, 1 - h)) / (2 * h)
    assert dphi / float(c * k + 1) == pytest.approx(float(expect), rel=1e-7)


@pytest.mark.parametrize("a1,c1,k1,a2,c2,k2", [(Fraction(9, 10), Fraction(2, 5), 2, Fraction(4, 5), Fraction(3, 10), 2),
                                               (Fraction(1, 2), Fraction(1, 10), 3, Fraction(2, 3), Fraction(1, 50), 4)])
def test_hc_ewif_equals_enumerated_expectation(a1, c1, k1, a2, c2, k2):
    # d1 drafts k1 tokens, then d2 drafts k2 more; acceptance stops at the first rejection; one bonus
    exp_tokens = Fraction(0)
    for outcome in itertools.product([0, 1], repeat=k1 + k2):
        p = Fraction(1)
        for i, o in enumerate(outcome):
            ai = a1 if i < k1 else a2
            p *= ai if o else 1 - ai
        acc = 0
        for o in outcome:
            if not o:
                break
            acc += 1
        exp_tokens += p * (acc + 1)
    expect = exp_tokens / (1 + k1 * c1 + k2 * c2)
    assert D.ewif_hc(float(a1), float(c1), k1, float(a2), float(c2), k2) == pytest.approx(float(expect), rel=1e-12)


@pytest.mark.parametrize("a,a12,c1,c2,n,k", [(Fraction(4, 5), Fraction(3, 5), Fraction(2, 5), Fraction(1, 20), 2, 2),
                                             (Fraction(2, 3), Fraction(9, 10), Fraction(1, 4), Fraction(1, 100), 3, 3)])
def test_vc_ewif_equals_enumerated_expectation(a, a12, c1, c2, n, k):
    # n rounds of d2 drafting k tokens checked by d1 give K d1-level tokens (sum of n independent
    # round yields); the target then accepts a prefix of them plus one token
    one = _round_tokens_dist(a12, k)
    dist = {0: Fraction(1)}
    for _ in range(n):
        nxt = {}
        for s, p in dist.items():
            for j, q in one.items():
                nxt[s + j] = nxt.get(s + j, Fraction(0)) + p * q
        dist = nxt
    exp_tokens = sum(p * (1 - a ** (K + 1)) / (1 - a) for K, p in dist.items())
    expect = exp_tokens / (1 + n * c1 + n * k * c2)
    assert D.ewif_vc(float(a), float(a12), float(c1), float(c2), n, k) == pytest.approx(float(expect), rel=1e-12)


def test_step_objective_is_the_marginal_hc_gain():
    # Eq. 5 drops the target's own round from T_HC(S for k tokens, bottom draft for one token):
    # T_s = (T_HC (1 + c k + c_dn) - 1) / (c k + c_dn)
    for a, c, k, a_dn, c_dn in [(0.9, 0.4, 2, 0.5, 0.01), (0.6, 0.2, 5, 0.3, 0.05), (0.75, 0.5, 1, 0.7, 0.1)]:
        t_hc = D.ewif_hc(a, c, k, a_dn, c_dn, 1)
        assert D.step_objective(a, c, k, a_dn, c_dn) == pytest.approx((t_hc * (1 + c * k + c_dn) - 1) / (c * k + c_dn),
                                                                      rel=1e-12)
    # the a = 1 branch agrees with the limit of the general branch
    assert D.step_objective(1.0, 0.3, 4, 0.5, 0.02) == pytest.approx(D.step_objective(1 - 1e-10, 0.3, 4, 0.5, 0.02),
                                                                      rel=1e-6)


def test_single_config_without_future_term_prefers_the_shortest_draft():
    # the local speedup a (1 - a^k) / ((1 - a) c k) is a mean of decreasing terms: k = 1 is best
    for a in (0.3, 0.6, 0.95):
        s, k, v = D.find_best_config([a], [0.25], 0.0, 0.0, 8)
        assert (s, k) == (0, 1) and v == pytest.approx(a / 0.25)


def test_no_positive_objective_returns_no_configuration():
    s, k, _ = D.find_best_config([0.0], [0.5], 0.0, 0.01, 4)
    assert s is None and k == 0


# ------------------------------------------------------------------------------------------------
# Sec. 4.2 EMA and App. D (unused configurations keep their estimate)
# ------------------------------------------------------------------------------------------------
def test_ema_closed_form_and_window():
    est = D.AlphaEstimates([0.2, 0.5], lam=0.7, window=20)
    for t in range(1, 11):
        est.record(0, True)
        est.step([0])
        assert est.alpha[0] == pytest.approx(1 - 0.8 * 0.7 ** t, rel=1e-12)
    assert est.alpha[1] == 0.5  # never used: unchanged
    # only the last H outcomes count
    est2 = D.AlphaEstimates([0.0], lam=0.0, window=4)
    for o in [1, 1, 1, 1, 0, 0]:
        est2.record(0, bool(o))
    est2.step([0])
    assert est2.alpha[0] == pytest.approx(0.5)


# ------------------------------------------------------------------------------------------------
# Algorithm 1 invariants (K = 1)
# ------------------------------------------------------------------------------------------------
def _fake_draft(cfg, path, k):
    base = 7 * len(path) + 13 * cfg
    return [(base + 3 * i) % 101 for i in range(k)]


@pytest.mark.parametrize("alphas,costs,a_dn,c_dn,k_max,t_min,m_max", [
    ([0.9, 0.8], [0.4, 0.3], 0.5, 0.05, 4, 1.0, 16),
    ([0.7, 0.6, 0.95], [0.3, 0.1, 0.6], 0.4, 0.02, 3, 0.5, 64),
    ([0.5], [0.2], 0.3, 0.05, 5, 4.0, 32),
])
def test_draft_tree_invariants(alphas, costs, a_dn, c_dn, k_max, t_min, m_max):
    tr = D.draft_tree(alphas, costs, a_dn, c_dn, k_max, t_min, m_max, _fake_draft)
    par, pacc, cfg = tr["parent"], tr["p_acc"], tr["cfg"]
    n = len(par)
    assert n <= m_max and par[0] == -1 and pacc[0] == 1.0
    kids = [0] * n
    for i in range(1, n):
        assert 0 <= par[i] < i
        kids[par[i]] += 1
        assert pacc[i] == pytest.approx(pacc[par[i]] * alphas[cfg[i]])
    assert max(kids) <= 1  # K = 1 from a single root: each expansion extends the one leaf
    s_best, k_best, _ = D.find_best_config(alphas, costs, a_dn, c_dn, k_max)
    for leaf, s, k in tr["steps"]:
        assert (s, k) == (s_best, k_best)  # estimates fixed during one tree
        assert a_dn / c_dn * pacc[leaf] >= t_min
    if n < m_max:  # stopped by the threshold: the last leaf fails it
        assert a_dn / c_dn * pacc[n - 1] < t_min
    # the number of drafted tokens before stopping follows from the geometric decay of P_acc
    a = alphas[s_best]
    depth_ok = 0
    while a_dn / c_dn * a ** depth_ok >= t_min:
        depth_ok += 1
    expected_nodes = min(m_max, 1 + math.ceil(depth_ok / k_best) * k_best) if depth_ok > 0 else 1
    assert n == expected_nodes


# ------------------------------------------------------------------------------------------------
# Sec. 4.2 latency model (Bayesian linear regression)
# ------------------------------------------------------------------------------------------------
def test_blr_limits_and_sequential_updates():
    import numpy as np

    rng = np.random.default_rng(7)
    x = rng.uniform(1.0, 15.0, 12)  # GB moved per step
    y = 25.0 + x * 153.8 + rng.normal(0, 30.0, 12)  # microseconds: overhead + bytes at 6.5 TB/s
    # a flat prior gives ordinary least squares
    mean, _ = D.blr_posterior(x, y, [0.0, 0.0], [1e12, 1e12], 30.0)
    ols = np.linalg.lstsq(np.stack([np.ones(12), x], 1), y, rcond=None)[0]
    assert mean == pytest.approx(ols, rel=1e-6)
    # no data gives the prior
    mean0, cov0 = D.blr_posterior([], [], [5.0, 150.0], [2.0, 10.0], 30.0)
    assert mean0 == pytest.approx([5.0, 150.0]) and cov0 == pytest.approx(np.diag([4.0, 100.0]))
    # conjugacy: one point at a time (each posterior the next prior, through its full covariance)
    # equals the batch posterior
    mu, cov = np.array([10.0, 140.0]), np.diag([50.0 ** 2, 40.0 ** 2])
    for xi, yi in zip(x, y):
        h = np.array([1.0, xi])
        s = h @ cov @ h + 30.0 ** 2
        gain = cov @ h / s
        mu = mu + gain * (yi - h @ mu)
        cov = cov - np.outer(gain, h @ cov)
    mean_b, cov_b = D.blr_posterior(x, y, [10.0, 140.0], [50.0, 40.0], 30.0)
    assert mean_b == pytest.approx(mu, rel=1e-6)
    assert cov_b == pytest.approx(cov, rel=1e-5, abs=1e-30)



# ------------------------------------------------------------------------------------------------
# Algorithm 1 with K candidates per drafted position (top-K / top-P) and sibling-parallel drafting
# ------------------------------------------------------------------------------------------------
def test_topp_keep_hand_cases():
    assert D.topp_keep([0.5, 0.25, 0.25], 0.75) == [0.5, 0.25]  # mass 0.75 reached: the third is dropped
    assert D.topp_keep([0.5, 0.25, 0.25], 0.76) == [0.5, 0.25, 0.25]
    assert D.topp_keep([0.5, 0.25, 0.25], 0.5) == [0.5]
    assert D.topp_keep([0.5, 0.25, 0.25], 0.25) == [0.5]  # the first is always kept
    assert D.topp_keep([2.0, 1.0, 1.0], 1.0) == [0.5, 0.25, 0.25]  # normalised over the K
    assert D.topp_keep([0.3], 0.1) == [1.0]


def test_topk_tree_worked_example():
    """Hand-traced: one configuration (a = 0.8, k = 2), candidates (token 1, p 0.6), (token 2, p 0.4)
    after every path, P_tree = 0.9 (both kept), m_max = 12.
      expansion 1: root -> n1 (1, 0.48), n2 (2, 0.32); n1 -> n3 (1, 0.2304), n4 (2, 0.1536);
      expansion 2: leaf n2 (0.32 is the highest active P_acc; its sibling n1 is expanded already):
                   n2 -> n5 (1, 0.1536), n6 (2, 0.1024); n5 -> n7 (1, 0.073728), n8 (2, 0.049152);
      expansion 3: leaf n3 (0.2304) with its active sibling n4 as a second branch:
                   n3 -> n9 (1, 0.110592), n10 (2, 0.073728); n4 -> n11 (1, 0.073728): 12 nodes, full."""
    s, k, _ = D.find_best_config([0.8], [0.05], 0.5, 0.2, 2)  # Eq. 5: 5.87 at k = 2 against 4.8 at k = 1
    assert (s, k) == (0, 2)
    tr = D.draft_tree_topk([0.8], [0.05], 0.5, 0.2, 2, 0.0, 12, 0.9, lambda cfg, path: [(1, 0.6), (2, 0.4)])
    assert tr["parent"] == [-1, 0, 0, 1, 1, 2, 2, 5, 5, 3, 3, 4]
    assert tr["token"] == [None, 1, 2, 1, 2, 1, 2, 1, 2, 1, 2, 1]
    assert tr["p_acc"] == pytest.approx([1.0, 0.48, 0.32, 0.2304, 0.1536, 0.1536, 0.1024, 0.073728, 0.049152,
                                         0.110592, 0.073728, 0.073728], rel=1e-12)
    assert tr["steps"] == [(0, 0, 2, [0]), (2, 0, 2, [2]), (3, 0, 2, [3, 4])]


def _fake_cands(K):
    def cands(cfg, path):
        base = (7 * len(path) + 13 * cfg + 5 * path[-1]) % 97
        w = [1.0 / (j + 1 + (base % 3)) for j in range(K)]
        return [((base + 11 * j) % 101, w[j]) for j in range(K)]
    return cands


def _depth_token(cfg, depth):
    return (7 * depth + 13 * cfg) % 101


@pytest.mark.parametrize("alphas,costs,a_dn,c_dn,k_max,t_min,m_max", [
    ([0.9, 0.8], [0.4, 0.3], 0.5, 0.05, 4, 1.0, 16),
    ([0.7, 0.6, 0.95], [0.3, 0.1, 0.6], 0.4, 0.02, 3, 0.5, 64),
    ([0.5], [0.2], 0.3, 0.05, 5, 4.0, 32),
])
def test_topk_tree_with_one_candidate_is_algorithm_1(alphas, costs, a_dn, c_dn, k_max, t_min, m_max):
    """K = 1: the top-K expansion is the chain expansion of draft_tree, node for node (a draft
    whose token depends on the configuration and the depth, given in both forms)."""
    want = D.draft_tree(alphas, costs, a_dn, c_dn, k_max, t_min, m_max,
                        lambda cfg, path, k: [_depth_token(cfg, len(path) + i) for i in range(k)])
    got = D.draft_tree_topk(alphas, costs, a_dn, c_dn, k_max, t_min, m_max, 0.5,
                            lambda cfg, path: [(_depth_token(cfg, len(path)), 0.37)])
    assert got["parent"] == want["parent"] and got["token"] == want["token"] and got["cfg"] == want["cfg"]
    assert got["p_acc"] == pytest.approx(want["p_acc"], rel=1e-12)
    assert [st[:3] for st in got["steps"]] == want["steps"]
    assert all(st[3] == [st[0]] for st in got["steps"])  # one branch: no siblings exist at K = 1


@pytest.mark.parametrize("K,p_tree,m_max", [(2, 0.9, 24), (3, 0.6, 64), (4, 1.0, 40), (3, 0.2, 64)])
def test_topk_tree_invariants(K, p_tree, m_max):
    alphas, costs = [0.85, 0.7], [0.35, 0.15]
    cands = _fake_cands(K)
    tr = D.draft_tree_topk(alphas, costs, 0.5, 0.02, 3, 0.2, m_max, p_tree, cands)
    par, tok, pacc, cfg = tr["parent"], tr["token"], tr["p_acc"], tr["cfg"]
    n = len(par)
    assert n <= m_max and par[0] == -1 and pacc[0] == 1.0

    def path_to(v):
        p = []
        while v >= 0:
            p.append(v)
            v = par[v]
        return p[::-1]

    kids = {}
    for i in range(1, n):
        assert 0 <= par[i] < i
        kids.setdefault(par[i], []).append(i)
    for v, ch in kids.items():
        # the children of a node are the kept prefix of its candidates, in rank order (each node
        # receives candidates from one drafted position only)
        pairs = cands(cfg[ch[0]], path_to(v))
        kept = D.topp_keep([p for _, p in pairs], p_tree)
        assert len(ch) <= len(kept)
        if ch[-1] != n - 1:  # not cut by the size limit
            assert len(ch) == len(kept)
        for j, c in enumerate(ch):
            assert tok[c] == pairs[j][0]
            assert pacc[c] == pytest.approx(pacc[v] * alphas[cfg[c]] * kept[j], rel=1e-12)
    for leaf, s, k, branches in tr["steps"]:
        assert branches[0] == leaf
        assert all(par[b] == par[leaf] for b in branches)  # the leaf and its siblings
    if p_tree <= 1.0 / K:  # the top-1 alone reaches the mass: a chain per expansion, no siblings
        assert all(len(ch) == 1 for ch in kids.values())


# ------------------------------------------------------------------------------------------------
# Sec. 4.2 vertical cascade VC(d_i, d_n) as one holistic round
# ------------------------------------------------------------------------------------------------
def test_vc_accept_hand_cases():
    assert D.vc_accept([], [7]) == [7]  # nothing proposed: d_i drafts one token
    assert D.vc_accept([5, 6, 9], [5, 6, 8, 1]) == [5, 6, 8]  # two accepted, then d_i's correction
    assert D.vc_accept([5, 6, 9], [5, 6, 9, 4]) == [5, 6, 9, 4]  # all accepted plus d_i's next token
    assert D.vc_accept([3, 6], [5, 6, 2]) == [5]  # the first rejected: later matches do not count


def test_vc_accept_equals_greedy_chain_prefix():
    """Whatever d_n proposes, the round's tokens are a prefix of d_i's own greedy chain: brute force
    over proposals against a fixed greedy continuation g (d_i's argmax after g[:r] is g[r])."""
    import itertools

    g = [4, 1, 3, 3, 0]
    for j in range(4):
        for prop in itertools.product(range(5), repeat=j):
            # d_i's argmax after each proposal prefix: g continues only while the proposals follow g
            am, ok = [], True
            for r in range(j + 1):
                am.append(g[r] if ok else (r * 7 + 2) % 5)
                ok = ok and r < j and prop[r] == g[r]
            got = D.vc_accept(list(prop), am)
            a = 0
            while a < j and prop[a] == g[a]:
                a += 1
            assert got == g[:a + 1]
