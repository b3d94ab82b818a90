"""The native DyTC scheduler (casspec_ewif_*, casspec_dytc_*: host code in the C-ABI library) against
the DyTC oracle, on seeded random inputs.  No GPU: these entry points do no device work."""
from __future__ import annotations

import random

import pytest

from oracle import dytc_oracle as D


@pytest.fixture(scope="module")
def cs():
    from paper_2510_26843_gb300 import build as b

    b.build()
    import paper_2510_26843_gb300 as m

    m.load_library()
    return m


def _rng(seed):
    return random.Random(seed)


def test_ewif_closed_forms_match_oracle(cs):
    r = _rng(1)
    for _ in range(300):
        a, a2, a12 = r.uniform(0.01, 0.99), r.uniform(0.01, 0.99), r.uniform(0.01, 0.99)
        c, c2 = r.uniform(0.0, 1.0), r.uniform(0.0, 0.2)
        k, k2, n = r.randint(0, 10), r.randint(0, 10), r.randint(1, 6)
        assert cs.ewif_sd(a, c, k) == pytest.approx(D.ewif_sd(a, c, k), rel=1e-12)
        assert cs.ewif_hc(a, c, k, a2, c2, k2) == pytest.approx(D.ewif_hc(a, c, k, a2, c2, k2), rel=1e-12)
        assert cs.ewif_vc(a, a12, c, c2, n, k) == pytest.approx(D.ewif_vc(a, a12, c, c2, n, k), rel=1e-12)
    assert cs.ewif_sd(1.0, 0.2, 3) == pytest.approx(4 / 1.6)  # a = 1: every draft accepted


def test_objective_and_best_config_match_oracle(cs):
    r = _rng(2)
    for _ in range(200):
        n_cfg = r.randint(1, 6)
        alphas = [r.choice([r.uniform(0, 1), 1.0, 0.0]) if r.random() < 0.1 else r.uniform(0, 1) for _ in range(n_cfg)]
        costs = [r.uniform(0.01, 1.0) for _ in range(n_cfg)]
        a_dn, c_dn, k_max = r.uniform(0, 1), r.choice([0.0, r.uniform(0.0, 0.1)]), r.randint(1, 8)
        for s in range(n_cfg):
            for k in range(1, k_max + 1):
                want = D.step_objective(alphas[s], costs[s], k, a_dn, c_dn)
                got = cs.dytc_objective(alphas[s], costs[s], k, a_dn, c_dn)
                assert (want is None and got != got) or got == pytest.approx(want, rel=1e-12)
        sch = cs.Dytc(alphas, costs, a_dn, c_dn, k_max, 0.0, 16)
        s_o, k_o, v_o = D.find_best_config(alphas, costs, a_dn, c_dn, k_max)
        s_n, k_n, v_n = sch.best_config()
        assert (s_n, k_n) == (s_o, k_o)
        if s_o is not None:
            assert v_n == pytest.approx(v_o, rel=1e-12)
        sch.close()


def test_ema_matches_oracle(cs):
    r = _rng(3)
    n_cfg = 4
    init = [r.uniform(0, 1) for _ in range(n_cfg)]
    sch = cs.Dytc(init, [0.3] * n_cfg, 0.5, 0.01, 4, 0.0, 16, lam=0.7, window=5)
    ora = D.AlphaEstimates(init, lam=0.7, window=5)
    for _ in range(60):
        used = [c for c in range(n_cfg) if r.random() < 0.5]
        for c in used:
            for _ in range(r.randint(1, 3)):
                acc = r.random() < 0.6
                sch.record(c, acc)
                ora.record(c, acc)
        sch.end_step()
        ora.step(used)
        for c in range(n_cfg):
            assert sch.alpha(c) == pytest.approx(ora.alpha[c], rel=1e-12, abs=1e-15)
    sch.close()


def _fake_draft(cfg, path, k):
    base = 7 * len(path) + 13 * cfg
    return [(base + 3 * i) % 101 for i in range(k)]


@pytest.mark.parametrize("seed", range(8))
def test_draft_tree_matches_oracle(cs, seed):
    r = _rng(100 + seed)
    n_cfg = r.randint(1, 4)
    alphas = [r.uniform(0.3, 0.99) for _ in range(n_cfg)]
    costs = [r.uniform(0.05, 0.8) for _ in range(n_cfg)]
    a_dn, c_dn = r.uniform(0.1, 0.8), r.choice([0.0, r.uniform(0.01, 0.1)])
    k_max, t_min, m_max = r.randint(1, 6), r.uniform(0.1, 10.0), r.randint(2, 64)
    want = D.draft_tree(alphas, costs, a_dn, c_dn, k_max, t_min, m_max, _fake_draft)
    sch = cs.Dytc(alphas, costs, a_dn, c_dn, k_max, t_min, m_max)
    sch.tree_reset()
    steps = []
    while True:
        plan = sch.tree_plan()
        if plan is None:
            break
        leaf, s, k = plan
        tr = sch.tree_get()
        path, v = [], leaf
        while v >= 0:
            path.append(v)
            v = tr["parent"][v]
        path.reverse()
        steps.append((leaf, s, k))
        sch.tree_extend(leaf, s, _fake_draft(s, path, k))
    got = sch.tree_get()
    assert steps == want["steps"]
    assert got["parent"] == want["parent"]
    assert got["token"][1:] == want["token"][1:] and got["token"][0] == -1
    assert got["cfg"] == want["cfg"]
    assert got["p_acc"] == pytest.approx(want["p_acc"], rel=1e-12)
    sch.close()


def test_argument_errors(cs):
    with pytest.raises(cs.CasspecError):
        cs.Dytc([1.5], [0.1], 0.5, 0.01, 4, 1.0, 16)  # acceptance outside [0, 1]
    with pytest.raises(cs.CasspecError):
        cs.Dytc([0.5], [0.1], 0.5, 0.01, 4, 1.0, 65)  # tree larger than CASSPEC_MAX_TREE
    with pytest.raises(cs.CasspecError):
        cs.Dytc([0.5], [0.1], 0.5, 0.01, 65, 1.0, 16)  # draft longer than any tree
    sch = cs.Dytc([0.5], [0.1], 0.5, 0.01, 4, 1.0, 16)
    with pytest.raises(cs.CasspecError):
        sch.record(3, True)  # no such configuration
    with pytest.raises(cs.CasspecError):
        sch.tree_extend(5, 0, [1])  # no such leaf
    sch.close()


def test_latency_fit_matches_oracle(cs):
    import numpy as np

    rng = np.random.default_rng(11)
    for m in (0, 1, 5, 40):
        x = rng.uniform(1.0, 30.0, m)  # GB moved per step
        y = 20.0 + x * 151.5 + rng.normal(0, 50.0, m)  # microseconds (6.6 TB/s)
        mu0, sd0, noise = [0.0, 150.0], [100.0, 100.0], 40.0
        w, cov = cs.latency_fit(x, y, mu0, sd0, noise)
        mean_o, cov_o = D.blr_posterior(x, y, mu0, sd0, noise)
        assert w == pytest.approx(list(mean_o), rel=1e-9)
        assert cov == pytest.approx(list(cov_o.reshape(-1)), rel=1e-9, abs=1e-30)
    with pytest.raises(cs.CasspecError):
        cs.latency_fit([1.0], [2.0], [0.0, 0.0], [0.0, 1.0], 1.0)  # zero prior spread



@pytest.mark.parametrize("alphas,costs,a_dn,c_dn,k_max,t_min,m_max", [
    ([0.8], [0.3], 0.5, 0.05, 4, 1.0, 1),       # a one-node tree: nothing to expand
    ([0.8, 0.6], [0.3, 0.2], 0.5, 0.0, 3, 1e9, 20),  # a free bottom draft: only the size limit stops
    ([1.0, 0.5], [0.4, 0.1], 0.5, 0.05, 5, 1.0, 64),  # a draft that is always accepted (E_acc = k)
    ([0.9], [0.3], 0.5, 0.05, 1, 0.0, 64),      # k_max = 1: one token per expansion
    ([0.0, 0.0], [0.3, 0.3], 0.0, 0.05, 4, 0.0, 16),  # no positive objective: the root is closed
])
def test_draft_tree_edge_cases_match_oracle(cs, alphas, costs, a_dn, c_dn, k_max, t_min, m_max):
    want = D.draft_tree(alphas, costs, a_dn, c_dn, k_max, t_min, m_max, _fake_draft)
    sch = cs.Dytc(alphas, costs, a_dn, c_dn, k_max, t_min, m_max)
    sch.tree_reset()
    while True:
        plan = sch.tree_plan()
        if plan is None:
            break
        leaf, s, k = plan
        tr = sch.tree_get()
        path, v = [], leaf
        while v >= 0:
            path.append(v)
            v = tr["parent"][v]
        sch.tree_extend(leaf, s, _fake_draft(s, path[::-1], k))
    got = sch.tree_get()
    assert got["parent"] == want["parent"] and got["cfg"] == want["cfg"]
    assert got["p_acc"] == pytest.approx(want["p_acc"], rel=1e-12)
    sch.close()


def _cands_f32(K):
    """Seeded fake candidates: K distinct tokens with float32-exact decreasing probabilities."""
    import numpy as np

    def cands(cfg, path):
        h = (7 * len(path) + 13 * cfg + 5 * path[-1] + 3) % 89
        w = np.sort(np.random.default_rng(h).uniform(0.01, 1.0, K).astype(np.float32))[::-1]
        return [((h + 17 * j) % 211, float(w[j])) for j in range(K)]
    return cands


def _native_topk_tree(cs, sch, cands, chain_cfgs=()):
    """Algorithm 1 with K candidates, driven through tree_plan / tree_begin / tree_add as the GPU
    round drives it; returns the steps (leaf, cfg, k, branches)."""
    sch.tree_reset()
    steps = []
    while True:
        plan = sch.tree_plan()
        if plan is None:
            break
        leaf, s, k = plan
        branches = sch.tree_begin(leaf, siblings=s not in chain_cfgs)
        steps.append((leaf, s, k, list(branches)))
        cur, full = list(branches), False
        for _ in range(k):
            tr = sch.tree_get()
            nxt = []
            for c in cur:
                path, v = [], c
                while v >= 0:
                    path.append(v)
                    v = tr["parent"][v]
                pairs = cands(s, path[::-1])
                if s in chain_cfgs:
                    pairs = pairs[:1]
                child = sch.tree_add(c, s, [t for t, _ in pairs], [p for _, p in pairs])
                if child == 0:
                    full = True
                    break
                nxt.append(child)
            if full:
                break
            cur = nxt
            if len(sch.tree_get()["parent"]) >= sch.m_max:
                break
        if full:
            break
    return steps


@pytest.mark.parametrize("seed", range(10))
def test_topk_tree_matches_oracle(cs, seed):
    r = _rng(500 + seed)
    n_cfg = r.randint(1, 4)
    alphas = [r.uniform(0.3, 0.99) for _ in range(n_cfg)]
    costs = [r.uniform(0.05, 0.8) for _ in range(n_cfg)]
    a_dn, c_dn = r.uniform(0.1, 0.8), r.choice([0.0, r.uniform(0.01, 0.1)])
    k_max, t_min, m_max = r.randint(1, 5), r.uniform(0.05, 3.0), r.randint(2, 64)
    K, p_tree = r.randint(1, 8), r.choice([1.0, r.uniform(0.3, 0.99)])
    chain = (n_cfg - 1,) if n_cfg > 1 and r.random() < 0.5 else ()
    cands = _cands_f32(K)
    want = D.draft_tree_topk(alphas, costs, a_dn, c_dn, k_max, t_min, m_max, p_tree, cands, chain_cfgs=chain)
    sch = cs.Dytc(alphas, costs, a_dn, c_dn, k_max, t_min, m_max, topk=K, p_tree=p_tree)
    steps = _native_topk_tree(cs, sch, cands, chain)
    got = sch.tree_get()
    assert steps == want["steps"]
    assert got["parent"] == want["parent"] and got["cfg"] == want["cfg"]
    assert got["token"][1:] == want["token"][1:]
    assert got["p_acc"] == pytest.approx(want["p_acc"], rel=1e-12)
    sch.close()


def test_topk_tree_argument_errors(cs):
    for kw in ({"topk": 0}, {"topk": 9}, {"p_tree": 0.0}, {"p_tree": 1.5}):
        with pytest.raises(cs.CasspecError):
            cs.Dytc([0.5], [0.1], 0.5, 0.01, 4, 1.0, 16, **kw)
    sch = cs.Dytc([0.5], [0.1], 0.5, 0.01, 4, 1.0, 16, topk=3, p_tree=0.9)
    with pytest.raises(cs.CasspecError):
        sch.tree_begin(4)  # no such node
    with pytest.raises(cs.CasspecError):
        sch.tree_add(0, 0, [], [])  # no candidate
    with pytest.raises(cs.CasspecError):
        sch.tree_add(0, 0, [1, 2], [0.0, 0.0])  # no probability mass
    with pytest.raises(cs.CasspecError):
        sch.tree_add(0, 1, [1], [1.0])  # no such configuration
    assert sch.tree_add(0, 0, [5, 6, 7], [0.5, 0.3, 0.2]) == 1
    assert sch.tree_get()["parent"] == [-1, 0, 0, 0]  # mass 0.5, then 0.8, both below 0.9: all three kept
    assert sch.tree_add(1, 0, [8, 9], [0.95, 0.05]) == 4
    assert sch.tree_get()["parent"] == [-1, 0, 0, 0, 1]  # 0.95 reaches 0.9: the second is dropped
    sch.close()


def test_vc_accept_matches_oracle(cs):
    r = _rng(900)
    for _ in range(500):
        j = r.randint(0, 6)
        g = [r.randint(0, 4) for _ in range(j + 1)]
        prop = [g[i] if r.random() < 0.7 else r.randint(0, 4) for i in range(j)]
        assert cs.vc_accept(prop, g) == D.vc_accept(prop, g)
    assert cs.load_library().casspec_vc_accept(None, -1, None, None) == cs.E_INVAL


def test_draft_cfg_marshalling(cs):
    import numpy as np

    mask = np.array([1, 0, 1], dtype=np.uint8)
    arr, keep = cs.draft_cfgs([(mask, 0), (None, 1), ("pld", 4), ("vc", mask, 1, 3), ("vc", None, 0, 2)])
    got = [(a.skip_mask is not None, a.quant_mode, a.pld_n_max, a.vc) for a in arr]
    assert got == [(True, 0, 0, 0), (False, 1, 0, 0), (False, 0, 4, 0), (True, 1, 3, 1), (False, 0, 2, 1)]
    assert arr[0].skip_mask == keep[0].ctypes.data and list(keep[3]) == [1, 0, 1]


def _cfg7b(cs):
    import synth

    s = synth.LLAMA7B
    return cs.config(s.n_layers, s.d_model, s.n_heads, s.head_dim, s.ffn, s.vocab)


def test_step_bytes_match_the_bench_byte_model(cs):
    """casspec_step_bytes (the latency model's regressor) equals the benchmark's algorithmic bytes for
    the 7B verify, a 50% layer-skip draft and a W8A8 draft; sub-block masks drop exactly their block."""
    import numpy as np

    import bench
    import synth

    sh = bench._shape()
    cfg = _cfg7b(cs)
    assert cs.step_bytes(cfg, None, 0, 64, 2048) == bench.algorithmic_bytes(sh, 64, 2048)["total"]
    mask = synth.skip_masks(7, sh.n_layers, [0.5])[0]
    assert cs.step_bytes(cfg, mask, 0, 8, 2048) == bench.algorithmic_bytes(sh, 8, 2048, 16)["total"]
    assert cs.step_bytes(cfg, None, 1, 8, 2048) == bench.algorithmic_bytes(sh, 8, 2048, None, 1)["total"]
    d, F, V, L = sh.d_model, sh.ffn, sh.vocab, sh.n_layers
    head = V * d * 2 + 8 * V * 4
    assert cs.step_bytes(cfg, np.zeros(L, np.uint8), 0, 8, 2048) == head
    no_attn = np.full(L, 1 | cs.SKIP_ATTN, np.uint8)
    assert cs.step_bytes(cfg, no_attn, 0, 8, 2048) == head + L * 3 * d * F * 2  # no K/V either
    no_ffn = np.full(L, 1 | cs.SKIP_FFN, np.uint8)
    assert cs.step_bytes(cfg, no_ffn, 0, 8, 2048) == head + L * (4 * d * d * 2 + 2 * 2048 * d * 2 + 2 * 8 * d * 2)
    assert cs.step_bytes(cfg, None, 2, 8, 2048) == bench.algorithmic_bytes(sh, 8, 2048, None, 2)["total"]
    with pytest.raises(cs.CasspecError):
        cs.step_bytes(cfg, None, 3, 8, 2048)


def test_costs_fitted_from_measured_steps(cs):
    """Steps measured on a roofline (20 us + bytes at 6.5 TB/s, noise 20 us) give the cost coefficients
    of the fitted model, the same as the oracle's posterior mean predicts, and near the true ratios."""
    import numpy as np

    rng = np.random.default_rng(5)
    x = rng.uniform(1e9, 1.5e10, 60)
    y = 20.0 + x / 6.5e6 + rng.normal(0, 20.0, 60)
    mu0, sd0, noise = [0.0, 1.0 / 6e6], [100.0, 1e-6], 20.0
    sch = cs.Dytc([0.6, 0.7, 0.3], [0.5, 0.5, 0.5], 0.3, 0.02, 4, 1.0, 16)
    for a, b in zip(x, y):
        sch.observe(0, a, b)
    cfg_bytes, target = [7.3e9, 7.8e9, 4.0e9], 1.433e10
    w = sch.fit_costs([0, 0, 0], cfg_bytes, target, mu0, sd0, noise)
    mean, _ = D.blr_posterior(x, y, mu0, sd0, noise)
    assert w[0] == pytest.approx(list(mean), rel=1e-9)
    prior, _ = D.blr_posterior([], [], mu0, sd0, noise)  # classes without steps keep the prior
    assert w[1] == pytest.approx(list(prior), rel=1e-12)
    costs = [sch.cost(c) for c in range(3)]
    pred = [(mean[0] + mean[1] * b) / (mean[0] + mean[1] * target) for b in cfg_bytes]
    assert costs == pytest.approx(pred, rel=1e-9)
    true = [(20.0 + b / 6.5e6) / (20.0 + target / 6.5e6) for b in cfg_bytes]
    assert costs == pytest.approx(true, rel=0.02)
    # Algorithm 2 now runs on the fitted costs
    s_o, k_o, _ = D.find_best_config([0.6, 0.7, 0.3], pred, 0.3, 0.02, 4)
    assert sch.best_config()[:2] == (s_o, k_o)
    with pytest.raises(cs.CasspecError):
        sch.fit_costs([0, 0, 0], cfg_bytes, 0.0, mu0, sd0, noise)
    with pytest.raises(cs.CasspecError):
        sch.fit_costs([0, 0, cs.DYTC_MAX_CLASS], cfg_bytes, target, mu0, sd0, noise)
    with pytest.raises(cs.CasspecError):
        sch.observe(0, 1e9, 0.0)
    with pytest.raises(cs.CasspecError):
        sch.observe(-1, 1e9, 10.0)
    sch.close()


def test_costs_fitted_per_arithmetic_class(cs):
    """A W8A8 step moves half the bytes of a bf16 step but is slower per byte (its integer MMA work,
    not its bytes, sets its time).  One line over the mixed observations predicts neither draft's
    cost; fitted per class, each class follows its own line (the oracle's posterior on that class's
    steps alone) and the costs come out near their true values and in their true order."""
    import numpy as np

    rng = np.random.default_rng(9)
    xb = rng.uniform(4e9, 1.5e10, 40)            # bf16 steps: 20 us + bytes at 6.5 TB/s
    yb = 20.0 + xb / 6.5e6 + rng.normal(0, 10.0, 40)
    xq = rng.uniform(2e9, 8e9, 40)               # W8A8 steps: 30 us + bytes at 1.8 TB/s
    yq = 30.0 + xq / 1.8e6 + rng.normal(0, 10.0, 40)
    mu0, sd0, noise = [0.0, 1.0 / 6e6], [100.0, 1e-5], 10.0
    sch = cs.Dytc([0.6, 0.8], [0.5, 0.5], 0.3, 0.02, 4, 1.0, 16)
    for a, b in zip(xb, yb):
        sch.observe(0, a, b)
    for a, b in zip(xq, yq):
        sch.observe(1, a, b)
    skip_bytes, int8_bytes, target = 7.3e9, 7.8e9, 1.433e10
    w = sch.fit_costs([0, 1], [skip_bytes, int8_bytes], target, mu0, sd0, noise)
    mb, _ = D.blr_posterior(xb, yb, mu0, sd0, noise)
    mq, _ = D.blr_posterior(xq, yq, mu0, sd0, noise)
    assert w[0] == pytest.approx(list(mb), rel=1e-9) and w[1] == pytest.approx(list(mq), rel=1e-9)
    t_target = mb[0] + mb[1] * target
    c_skip, c_int8 = sch.cost(0), sch.cost(1)
    assert c_skip == pytest.approx((mb[0] + mb[1] * skip_bytes) / t_target, rel=1e-9)
    assert c_int8 == pytest.approx((mq[0] + mq[1] * int8_bytes) / t_target, rel=1e-9)
    true_skip = (20.0 + skip_bytes / 6.5e6) / (20.0 + target / 6.5e6)
    true_int8 = (30.0 + int8_bytes / 1.8e6) / (20.0 + target / 6.5e6)
    assert c_skip == pytest.approx(true_skip, rel=0.03) and c_int8 == pytest.approx(true_int8, rel=0.03)
    assert c_int8 > 1.0 > c_skip  # the W8A8 draft costs more than the verify it serves
    # one line over both classes predicts neither draft's cost
    m1, _ = D.blr_posterior(np.r_[xb, xq], np.r_[yb, yq], mu0, sd0, noise)
    one = [(m1[0] + m1[1] * b) / (m1[0] + m1[1] * target) for b in (skip_bytes, int8_bytes)]
    assert abs(one[0] / true_skip - 1) > 0.2 and abs(one[1] / true_int8 - 1) > 0.2
    sch.close()
