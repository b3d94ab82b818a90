"""CPU oracle of the Dynamic Tree Cascade (DyTC) scheduler and the cascade EWIF closed forms.

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle/``: only ``tests/`` (and ``bench.py``'s CPU
arms) may import it.  The native scheduler in the CUDA library shares no code with it.

What it computes (CAS-Spec, arXiv 2510.26843):
  * Sec. 3, expected walltime improvement factors (EWIF) under i.i.d. Bernoulli acceptance:
      - standard speculative decoding, T_SD = (1 - a^(k+1)) / ((1 - a)(c k + 1)), the derivative at
        1 of the probability generating function phi_(a,k)(x) of the tokens one round yields,
        divided by the round's cost;
      - the vertical cascade VC(d1, d2), T_VC = (1 - a phi(a)^n) / ((1 - a)(1 + n c1 + n k c2)),
        phi = phi_(a12, k), a = alpha(t, d1), a12 = alpha(d1, d2);
      - the horizontal cascade HC(d1, d2),
        T_HC = [(1 - a1^(k1+1)) / (1 - a1) + a1^k1 a2 (1 - a2^k2) / (1 - a2)] / (1 + k1 c1 + k2 c2);
  * Sec. 4.2, the online estimates: alpha_new = lambda alpha_prev + (1 - lambda) alpha_recent, where
    alpha_recent is the mean of the last H first-draft-token outcomes of the configuration, and
    configurations not used in a step keep their estimate (App. D);
  * Sec. 4.2 Eq. 5 and App. D Algorithm 2 (FindBestConfigurationForStep): maximise over the
    candidate configurations S and k in [1, k_max]
      T_s(S, k) = (E_acc + a_S^k a_dn) / (c_S k + c_dn),  E_acc = a_S (1 - a_S^k) / (1 - a_S)
    (E_acc = k when a_S is 1), the local speedup of the step plus the least future speedup of the
    bottom draft d_n;
  * Sec. 4.2 Algorithm 1 (draft tree generation): expand the active leaf with the highest
    accumulated acceptance P_acc, stop when a_dn / c_dn * P_acc < t_min or the tree holds m_max
    nodes, choose (S, k) by Algorithm 2; with one token per drafted position (K = 1, `draft_tree`)
    append the k drafted tokens below the leaf with P_acc(child) = P_acc(parent) * a_S; with K
    candidates per position and sibling-parallel drafting, `draft_tree_topk` (readings below);
  * Sec. 4.2 vertical cascade VC(d_i, d_n) as one holistic round (`vc_accept`): d_i's drafted tokens
    are the low-level proposals it accepts in order, then its own next token.

  * Sec. 4.2, the hardware-aware latency prediction behind the cost coefficients: a Bayesian linear
    regression of step latency on the bytes the step moves (a roofline: latency = w0 + w1 * bytes),
    Gaussian prior N(mu0, diag(sd0^2)) on w and Gaussian noise; c(S) = predicted latency of draft S /
    predicted latency of the target.

Readings (the paper is silent or inconsistent; each is also listed in the design notes):
  * the latency model's regressor is the bytes a step moves (weights of its active layers, K/V,
    activations), the quantity the roofline of a memory-bound step is linear in; the paper names
    only "roofline latency" and "Bayesian linear regression";
  * phi^n in T_VC is the n-th power of the generating function (n independent rounds of d2);
  * only leaves are expanded: Algorithm 1 marks every new node active and never clears the expanded
    node, which would let a node be drafted twice from the same sequence; a node that receives a
    child is no longer an active leaf;
  * ties: Algorithm 2 keeps the first (S, k) reaching the maximum (strict >); among active leaves of
    equal P_acc the lowest node index is expanded;
  * Algorithm 1 with K > 1 (`draft_tree_topk`; the printed loop, its function names and the shape
    of y disagree with one another): at every drafted position the draft's K best tokens, their
    probabilities normalised over the K, are candidate children of the branch's current node; the
    first candidate is always kept and each further one while the normalised mass kept before it
    is below P_tree (top-P); the top-1 child continues the branch.  The token-level refinement of
    P_acc (Sec. 4.2, "normalized probability" of a drafted token) is
    P_acc(child) = P_acc(parent) * a_S * p_norm(child), which is Algorithm 1's a_S product at K = 1.
    Sibling-parallel drafting: expanding a leaf with a neural draft extends, in the same draft
    steps and by the same k, every active sibling of that leaf (same parent), each as a branch of
    its own; branches are processed in node order, and within a branch candidates in rank order,
    until the tree holds m_max nodes;
  * "a ~ 1" and "c k + c_dn ~ 0" in Algorithm 2 are |1 - a| < 1e-9 and |c k + c_dn| < 1e-12.
"""
from __future__ import annotations

import math


# ------------------------------------------------------------------------------------------------
# Sec. 3: EWIF closed forms
# ------------------------------------------------------------------------------------------------
def pgf_sd(a: float, k: int, x: float) -> float:
    """phi_(a,k)(x) = 1 + (x - 1)(1 - a^(k+1) x^(k+1)) / (1 - a x): generating function of the number of
    tokens one speculative round with draft length k yields (Sec. 3)."""
    if abs(1.0 - a * x) < 1e-15:
        return 1.0 + (x - 1.0) * (k + 1)
    return 1.0 + (x - 1.0) * (1.0 - (a * x) ** (k + 1)) / (1.0 - a * x)


def ewif_sd(a: float, c: float, k: int) -> float:
    """T_SD = (1 - a^(k+1)) / ((1 - a)(c k + 1)) (Sec. 3)."""
    num = (k + 1) if abs(1.0 - a) < 1e-12 else (1.0 - a ** (k + 1)) / (1.0 - a)
    return num / (c * k + 1.0)


def ewif_vc(a: float, a12: float, c1: float, c2: float, n: int, k: int) -> float:
    """T_VC(d1, d2) = (1 - a phi(a)^n) / ((1 - a)(1 + n c1 + n k c2)), phi = phi_(a12, k) (Sec. 3)."""
    phi = pgf_sd(a12, k, a)
    return (1.0 - a * phi ** n) / ((1.0 - a) * (1.0 + n * c1 + n * k * c2))


def ewif_hc(a1: float, c1: float, k1: int, a2: float, c2: float, k2: int) -> float:
    """T_HC(d1, d2) (Sec. 3, after CS-Drafting Thm. 4.5)."""
    first = (1.0 - a1 ** (k1 + 1)) / (1.0 - a1)
    second = a1 ** k1 * a2 * (1.0 - a2 ** k2) / (1.0 - a2)
    return (first + second) / (1.0 + k1 * c1 + k2 * c2)


def best_sd(a: float, c: float, k_max: int) -> tuple[float, int]:
    """max over k in [1, k_max] of T_SD, with the first maximising k."""
    best, arg = -math.inf, 0
    for k in range(1, k_max + 1):
        v = ewif_sd(a, c, k)
        if v > best:
            best, arg = v, k
    return best, arg


def best_hc(a1: float, c1: float, a2: float, c2: float, k_max: int) -> tuple[float, int, int]:
    """max over k1, k2 in [1, k_max] of T_HC."""
    best, arg = -math.inf, (0, 0)
    for k1 in range(1, k_max + 1):
        for k2 in range(1, k_max + 1):
            v = ewif_hc(a1, c1, k1, a2, c2, k2)
            if v > best:
                best, arg = v, (k1, k2)
    return best, arg[0], arg[1]


# ------------------------------------------------------------------------------------------------
# Sec. 4.2: acceptance-rate estimates (EMA over a window of first-token outcomes)
# ------------------------------------------------------------------------------------------------
class AlphaEstimates:
    """Per configuration: the estimate alpha and the last H first-draft-token outcomes (0/1)."""

    def __init__(self, alpha_init: list[float], lam: float = 0.7, window: int = 20):
        self.alpha = list(alpha_init)
        self.lam = lam
        self.window = window
        self.hist: list[list[int]] = [[] for _ in alpha_init]

    def record(self, cfg: int, accepted: bool) -> None:
        h = self.hist[cfg]
        h.append(1 if accepted else 0)
        if len(h) > self.window:
            del h[0]

    def step(self, used: list[int]) -> None:
        """End of a generation step: alpha_new = lam alpha_prev + (1 - lam) alpha_recent for every
        configuration used in the step; the others keep their estimate (App. D)."""
        for cfg in sorted(set(used)):
            h = self.hist[cfg]
            if h:
                recent = sum(h) / len(h)
                self.alpha[cfg] = self.lam * self.alpha[cfg] + (1.0 - self.lam) * recent


# ------------------------------------------------------------------------------------------------
# Eq. 5 / Algorithm 2
# ------------------------------------------------------------------------------------------------
def step_objective(a: float, c: float, k: int, a_dn: float, c_dn: float) -> float | None:
    """T_s(S, k) of Eq. 5; None where Algorithm 2 skips the pair (c k + c_dn ~ 0)."""
    if abs(c * k + c_dn) < 1e-12:
        return None
    e_acc = float(k) if abs(1.0 - a) < 1e-9 else a * (1.0 - a ** k) / (1.0 - a)
    return (e_acc + a ** k * a_dn) / (c * k + c_dn)


def find_best_config(alphas: list[float], costs: list[float], a_dn: float, c_dn: float,
                     k_max: int) -> tuple[int | None, int, float]:
    """Algorithm 2: (configuration, k, objective) maximising Eq. 5; (None, 0, obj) if no positive
    objective exists."""
    best, s_best, k_best = -math.inf, None, 0
    for s, (a, c) in enumerate(zip(alphas, costs)):
        for k in range(1, k_max + 1):
            v = step_objective(a, c, k, a_dn, c_dn)
            if v is None:
                continue
            if v > best:
                best, s_best, k_best = v, s, k
    if best <= 0.0:
        return None, 0, best
    return s_best, k_best, best


# ------------------------------------------------------------------------------------------------
# Algorithm 1 (K = 1)
# ------------------------------------------------------------------------------------------------
def draft_tree(alphas: list[float], costs: list[float], a_dn: float, c_dn: float, k_max: int,
               t_min: float, m_max: int, draft) -> dict:
    """Build one draft tree.  ``draft(cfg, path, k)`` returns the k tokens configuration ``cfg`` drafts
    greedily after the node sequence ``path`` (root first).  Returns the tree as lists indexed by
    node: parent (-1 for the root), token (None for the root), cfg (-1 for the root), p_acc, and the
    expansions made, each (leaf, cfg, k)."""
    parent, token, cfg_of, p_acc, active = [-1], [None], [-1], [1.0], [True]
    steps = []
    while len(parent) < m_max:
        cands = [i for i in range(len(parent)) if active[i]]
        if not cands:
            break
        leaf = max(cands, key=lambda i: (p_acc[i], -i))
        if c_dn > 0.0 and a_dn / c_dn * p_acc[leaf] < t_min:  # a free bottom draft never stops it
            break
        s, k, _ = find_best_config(alphas, costs, a_dn, c_dn, k_max)
        if s is None:
            active[leaf] = False
            break
        path = []
        v = leaf
        while v >= 0:
            path.append(v)
            v = parent[v]
        path.reverse()
        toks = draft(s, path, k)
        steps.append((leaf, s, k))
        active[leaf] = False
        node = leaf
        for i in range(k):
            parent.append(node)
            token.append(toks[i])
            cfg_of.append(s)
            p_acc.append(p_acc[node] * alphas[s])
            active.append(True)
            if node != leaf:
                active[node] = False
            node = len(parent) - 1
            if len(parent) >= m_max:
                return {"parent": parent, "token": token, "cfg": cfg_of, "p_acc": p_acc, "steps": steps}
    return {"parent": parent, "token": token, "cfg": cfg_of, "p_acc": p_acc, "steps": steps}


def topp_keep(probs: list[float], p_tree: float) -> list[float]:
    """Normalised probabilities of the candidates kept from one position's K best (rank order):
    the first always, each further one while the normalised mass before it is below p_tree."""
    total = sum(probs)
    kept, mass = [], 0.0
    for j, p in enumerate(probs):
        if j > 0 and mass >= p_tree:
            break
        q = p / total
        kept.append(q)
        mass += q
    return kept


def draft_tree_topk(alphas: list[float], costs: list[float], a_dn: float, c_dn: float, k_max: int,
                    t_min: float, m_max: int, p_tree: float, cands, chain_cfgs=()) -> dict:
    """Algorithm 1 with K candidates per drafted position and sibling-parallel drafting.

    ``cands(cfg, path)`` returns configuration ``cfg``'s K best next tokens after the node sequence
    ``path`` (root first), as (token, probability) pairs in rank order.  Configurations in
    ``chain_cfgs`` (a retrieval bottom draft) give one candidate per position and draft no
    siblings; an empty candidate list ends that branch, and at an expansion's first position it
    ends the drafting (nothing to propose).  Returns the tree like ``draft_tree``; ``steps`` holds
    (leaf, cfg, k, branches)."""
    parent, token, cfg_of, p_acc, active = [-1], [None], [-1], [1.0], [True]
    steps = []

    def out():
        return {"parent": parent, "token": token, "cfg": cfg_of, "p_acc": p_acc, "steps": steps}

    def path_to(v):
        path = []
        while v >= 0:
            path.append(v)
            v = parent[v]
        return path[::-1]

    while len(parent) < m_max:
        open_leaves = [i for i in range(len(parent)) if active[i]]
        if not open_leaves:
            break
        leaf = max(open_leaves, key=lambda i: (p_acc[i], -i))
        if c_dn > 0.0 and a_dn / c_dn * p_acc[leaf] < t_min:
            break
        s, k, _ = find_best_config(alphas, costs, a_dn, c_dn, k_max)
        if s is None:
            active[leaf] = False
            break
        branches = [leaf]
        if s not in chain_cfgs and leaf != 0:
            branches += [j for j in range(len(parent)) if j != leaf and active[j] and parent[j] == parent[leaf]]
        steps.append((leaf, s, k, list(branches)))
        cur = list(branches)
        for pos in range(k):
            nxt = []
            for c in cur:
                pairs = cands(s, path_to(c))
                if s in chain_cfgs:
                    pairs = pairs[:1]
                if not pairs:
                    if pos == 0 and c == leaf:
                        return out()
                    continue
                kept = topp_keep([p for _, p in pairs], 1.0 if s in chain_cfgs else p_tree)
                active[c] = False  # c receives children: no longer a leaf
                first = None
                for (tok, _), q in zip(pairs, kept):
                    parent.append(c)
                    token.append(tok)
                    cfg_of.append(s)
                    p_acc.append(p_acc[c] * alphas[s] * q)
                    active.append(True)
                    if first is None:
                        first = len(parent) - 1
                    if len(parent) >= m_max:
                        return out()
                nxt.append(first)
            cur = nxt
    return out()


def vc_accept(proposals: list[int], argmax: list[int]) -> list[int]:
    """One holistic round of the vertical cascade VC(d_i, d_n) (Sec. 4.2: its draft length follows
    from how many low-level tokens d_i accepts): d_n proposed `proposals` below the leaf; d_i's
    greedy choices are argmax[0] at the leaf and argmax[r] after the r-th proposal.  Returns d_i's
    drafted tokens: the proposals it accepts in order, then its own next token."""
    out = []
    for r, q in enumerate(proposals):
        if q != argmax[r]:
            break
        out.append(q)
    out.append(argmax[len(out)])
    return out


# ------------------------------------------------------------------------------------------------
# Sec. 4.2: latency model (Bayesian linear regression)
# ------------------------------------------------------------------------------------------------
def blr_posterior(x, y, mu0, sd0, noise_sd):
    """Posterior mean and covariance of w in y = w0 + w1 x + e, e ~ N(0, noise_sd^2), with prior
    w ~ N(mu0, diag(sd0^2)): cov = (S0^-1 + X^T X / s^2)^-1, mean = cov (S0^-1 mu0 + X^T y / s^2)."""
    import numpy as np

    X = np.stack([np.ones(len(x)), np.asarray(x, dtype=np.float64)], axis=1) if len(x) else np.zeros((0, 2))
    y = np.asarray(y, dtype=np.float64)
    prec0 = np.diag(1.0 / np.asarray(sd0, dtype=np.float64) ** 2)
    prec = prec0 + X.T @ X / noise_sd ** 2
    cov = np.linalg.inv(prec)
    mean = cov @ (prec0 @ np.asarray(mu0, dtype=np.float64) + X.T @ y / noise_sd ** 2)
    return mean, cov

