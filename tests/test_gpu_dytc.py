"""DyTC speculative decoding on the GPU (Sec. 4.2 Algorithm 1 with the native scheduler, drafts and
verification as tree steps): on the tiny decoder, rounds of casspec_dytc_round must reproduce the
oracle's greedy autoregressive output (losslessness, Sec. 5.1), except after a near-tie of greedy
decoding itself (top-2 logit margin below 1e-3), and the acceptance estimates must follow what the
target accepted."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

SH = synth.TINY
SEED = 1234
MARGIN = 1e-3


@pytest.fixture(scope="module")
def cs():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2510_26843_gb300 as m

    m.load_library()
    return m


def _truth(prefix, steps):
    ow = oracle.Weights.from_seed(SEED, SH, keep_layers=SH.n_layers)
    okv = oracle.KVCache(SH.n_layers, SH.n_heads, SH.head_dim, 256)
    lg = oracle.tree_step(ow, okv, prefix, synth.chain(len(prefix)))
    oracle.kv_compact(okv, list(range(len(prefix))))
    truth, margins = [int(oracle.argmax_lowest(lg[-1:])[0])], [oracle.top2_margin(lg[-1:])[0]]
    while len(truth) < steps + 1:
        lg = oracle.tree_step(ow, okv, [truth[-1]], [-1])
        oracle.kv_compact(okv, [0])
        truth.append(int(oracle.argmax_lowest(lg)[0]))
        margins.append(oracle.top2_margin(lg)[0])
    return truth, margins


def test_dytc_rounds_are_lossless_and_learn_acceptance(cs):
    from paper_2510_26843_gb300.workload import DeviceKV, DeviceModel

    steps = 40
    prefix = synth.prefix_tokens(SEED, 64, SH.vocab)
    truth, margins = _truth(prefix, steps)

    dm = DeviceModel(SH, SEED, with_int8=True)
    kv = DeviceKV(dm, 256)
    n0 = len(prefix)
    t = torch.tensor(np.asarray(prefix, dtype=np.int32), device="cuda")
    p = torch.tensor(np.asarray(synth.chain(n0), dtype=np.int32), device="cuda")
    logits = torch.empty(n0, SH.vocab, device="cuda")
    cs.tree_step(dm.h, kv.h, t, p, n0, None, 0, logits)
    cs.kv_compact(kv.h, torch.tensor([n0, *range(n0), 0], dtype=torch.int32, device="cuda"))
    out = [int(torch.argmax(logits[-1]).item())]

    # two draft configurations of the 2-layer model: the first layer alone (bf16), and every layer
    # in W8A8; a notional bottom draft (alpha 0.3, cost 0.05)
    cfgs = [(np.array([1, 0], dtype=np.uint8), 0), (None, 1)]
    sch = cs.Dytc([0.5, 0.5], [0.5, 0.6], alpha_dn=0.3, c_dn=0.05, k_max=4, t_min=0.5, m_max=16)
    work = torch.zeros(cs.DYTC_WORK, dtype=torch.int32, device="cuda")
    rounds = drafted = 0
    while len(out) < steps:
        toks, nd = sch.round(dm.h, kv.h, cfgs, out[-1], work)
        assert 1 <= len(toks) <= nd + 1
        out.extend(toks)
        drafted += nd
        rounds += 1
    assert cs.get_status(dm.h) == 0
    first_diff = next((i for i in range(steps) if out[i] != truth[i]), None)
    if first_diff is not None:
        assert min(margins[: first_diff + 1]) < MARGIN, (first_diff, out[:steps], truth[:steps])
    assert drafted > 0 and rounds < steps  # drafts were made and some were accepted
    # the W8A8 draft of every layer agrees with the target far more often than the half-depth one
    assert sch.alpha(1) > sch.alpha(0)
    P, T = cs.kv_length(kv.h)
    assert T == 0 and P == n0 + len(out) - 1  # every committed token but the last root is cached
    sch.close()
    kv.close()
    dm.close()


def test_dytc_rounds_with_prompt_lookup_bottom_draft_are_lossless(cs):
    """The same with the prompt-lookup draft (casspec_pld_draft over the committed history) as a third
    configuration: whatever it proposes, verification keeps the output equal to greedy decoding."""
    from paper_2510_26843_gb300.workload import DeviceKV, DeviceModel

    steps = 48
    prefix = synth.prefix_tokens(SEED + 1, 64, SH.vocab)
    truth, margins = _truth(prefix, steps)
    dm = DeviceModel(SH, SEED, with_int8=True)
    kv = DeviceKV(dm, 256)
    n0 = len(prefix)
    t = torch.tensor(np.asarray(prefix, dtype=np.int32), device="cuda")
    p = torch.tensor(np.asarray(synth.chain(n0), dtype=np.int32), device="cuda")
    logits = torch.empty(n0, SH.vocab, device="cuda")
    cs.tree_step(dm.h, kv.h, t, p, n0, None, 0, logits)
    cs.kv_compact(kv.h, torch.tensor([n0, *range(n0), 0], dtype=torch.int32, device="cuda"))
    out = [int(torch.argmax(logits[-1]).item())]
    history = torch.zeros(n0 + steps + 4 * cs.MAX_TREE, dtype=torch.int32, device="cuda")
    history[:n0] = t
    history[n0] = out[0]
    hist_len = n0 + 1

    cfgs = [(np.array([1, 0], dtype=np.uint8), 0), (None, 1), ("pld", 4)]
    sch = cs.Dytc([0.5, 0.5, 0.3], [0.5, 0.6, 0.02], alpha_dn=0.3, c_dn=0.02, k_max=4, t_min=0.5, m_max=16)
    work = torch.zeros(cs.DYTC_WORK, dtype=torch.int32, device="cuda")
    rounds = 0
    while len(out) < steps:
        toks, nd = sch.round(dm.h, kv.h, cfgs, out[-1], work, history, hist_len)
        assert 1 <= len(toks) <= nd + 1
        history[hist_len:hist_len + len(toks)] = torch.tensor(toks, dtype=torch.int32, device="cuda")
        hist_len += len(toks)
        out.extend(toks)
        rounds += 1
    assert cs.get_status(dm.h) == 0
    first_diff = next((i for i in range(steps) if out[i] != truth[i]), None)
    if first_diff is not None:
        assert min(margins[: first_diff + 1]) < MARGIN, (first_diff, out[:steps], truth[:steps])
    assert rounds < steps
    P, T = cs.kv_length(kv.h)
    assert T == 0 and P == n0 + len(out) - 1
    sch.close()
    kv.close()
    dm.close()



def test_dytc_rounds_with_top_k_siblings_are_lossless(cs):
    """K = 3 candidates per drafted position with top-P 0.9 (Algorithm 1's tree expansion) and
    sibling-parallel drafting, with the two model drafts and the prompt-lookup draft: the output
    stays greedy decoding, and the trees branch."""
    from paper_2510_26843_gb300.workload import DeviceKV, DeviceModel

    steps = 48
    prefix = synth.prefix_tokens(SEED + 2, 64, SH.vocab)
    truth, margins = _truth(prefix, steps)
    dm = DeviceModel(SH, SEED, with_int8=True)
    kv = DeviceKV(dm, 256)
    n0 = len(prefix)
    t = torch.tensor(np.asarray(prefix, dtype=np.int32), device="cuda")
    p = torch.tensor(np.asarray(synth.chain(n0), dtype=np.int32), device="cuda")
    logits = torch.empty(n0, SH.vocab, device="cuda")
    cs.tree_step(dm.h, kv.h, t, p, n0, None, 0, logits)
    cs.kv_compact(kv.h, torch.tensor([n0, *range(n0), 0], dtype=torch.int32, device="cuda"))
    out = [int(torch.argmax(logits[-1]).item())]
    history = torch.zeros(n0 + steps + 4 * cs.MAX_TREE, dtype=torch.int32, device="cuda")
    history[:n0] = t
    history[n0] = out[0]
    hist_len = n0 + 1

    # the W8A8 draft starts as Algorithm 2's choice (Eq. 5: 10.3 against 9.75 for the prompt lookup);
    # the tiny drafts' distributions are flat (normalised top-1 of three about 0.35), so its
    # expansions keep all three candidates and the tree branches from the first position
    cfgs = [(np.array([1, 0], dtype=np.uint8), 0), (None, 1), ("pld", 4)]
    sch = cs.Dytc([0.6, 0.95, 0.3], [0.5, 0.1, 0.02], alpha_dn=0.3, c_dn=0.02, k_max=3, t_min=0.3, m_max=32,
                  topk=3, p_tree=0.9)
    work = torch.zeros(cs.DYTC_WORK, dtype=torch.int32, device="cuda")
    dlog = torch.empty(cs.MAX_TREE, SH.vocab, device="cuda")
    rounds = branched = 0
    while len(out) < steps:
        toks, nd = sch.round(dm.h, kv.h, cfgs, out[-1], work, history, hist_len, dev_logits=dlog)
        assert 1 <= len(toks) <= nd + 1
        tr = sch.tree_get()
        kids = np.bincount(np.asarray(tr["parent"][1:], dtype=np.int64), minlength=len(tr["parent"]))
        branched += int(kids.max(initial=0) > 1)
        history[hist_len:hist_len + len(toks)] = torch.tensor(toks, dtype=torch.int32, device="cuda")
        hist_len += len(toks)
        out.extend(toks)
        rounds += 1
    assert cs.get_status(dm.h) == 0
    first_diff = next((i for i in range(steps) if out[i] != truth[i]), None)
    if first_diff is not None:
        assert min(margins[: first_diff + 1]) < MARGIN, (first_diff, out[:steps], truth[:steps])
    assert branched > 0 and rounds < steps
    P, T = cs.kv_length(kv.h)
    assert T == 0 and P == n0 + len(out) - 1
    # a round with K > 1 needs the logits buffer
    with pytest.raises(cs.CasspecError):
        sch.round(dm.h, kv.h, cfgs, out[-1], work, history, hist_len)
    sch.close()
    kv.close()
    dm.close()


def test_dytc_rounds_with_vertical_cascade(cs):
    """VC(first-layer draft, prompt lookup) as a configuration (Sec. 4.2: one holistic round per
    expansion): every node it drafts is the first-layer draft's own greedy token at its parent
    (checked against the oracle's draft, except at near-ties), and the output stays greedy decoding.
    The prefix repeats a 16-token segment so that the lookup has matches to propose."""
    from paper_2510_26843_gb300.workload import DeviceKV, DeviceModel

    steps = 40
    seg = synth.prefix_tokens(SEED + 3, 16, SH.vocab)
    prefix = np.concatenate([seg] * 4)
    truth, margins = _truth(prefix, steps)
    ow = oracle.Weights.from_seed(SEED, SH, keep_layers=SH.n_layers)
    dm = DeviceModel(SH, SEED, with_int8=True)
    kv = DeviceKV(dm, 256)
    n0 = len(prefix)
    t = torch.tensor(np.asarray(prefix, dtype=np.int32), device="cuda")
    p = torch.tensor(np.asarray(synth.chain(n0), dtype=np.int32), device="cuda")
    logits = torch.empty(n0, SH.vocab, device="cuda")
    cs.tree_step(dm.h, kv.h, t, p, n0, None, 0, logits)
    cs.kv_compact(kv.h, torch.tensor([n0, *range(n0), 0], dtype=torch.int32, device="cuda"))
    out = [int(torch.argmax(logits[-1]).item())]
    history = torch.zeros(n0 + steps + 4 * cs.MAX_TREE, dtype=torch.int32, device="cuda")
    history[:n0] = t
    history[n0] = out[0]
    hist_len = n0 + 1

    d1 = np.array([1, 0], dtype=np.uint8)
    cfgs = [("vc", d1, 0, 4), (None, 1)]
    # Eq. 5 picks the cascade with k = 3 at these estimates
    sch = cs.Dytc([0.8, 0.9], [0.2, 0.6], alpha_dn=0.3, c_dn=0.3, k_max=4, t_min=0.3, m_max=24)
    assert sch.best_config()[:2] == (0, 3)
    work = torch.zeros(cs.DYTC_WORK, dtype=torch.int32, device="cuda")
    rounds = checked = 0
    while len(out) < steps:
        committed, root = list(prefix) + out[:-1], out[-1]
        toks, nd = sch.round(dm.h, kv.h, cfgs, root, work, history, hist_len)
        tr = sch.tree_get()
        vc_nodes = [v for v in range(1, len(tr["parent"])) if tr["cfg"][v] == 0]
        if vc_nodes:
            okv = oracle.KVCache(SH.n_layers, SH.n_heads, SH.head_dim, 256)
            oracle.tree_step(ow, okv, committed, synth.chain(len(committed)), skip_mask=d1)
            oracle.kv_compact(okv, list(range(len(committed))))
            ttoks = [root] + tr["token"][1:]
            lg = oracle.tree_step(ow, okv, ttoks, tr["parent"], skip_mask=d1)
            am, mg = oracle.argmax_lowest(lg), oracle.top2_margin(lg)
            for v in vc_nodes:
                if mg[tr["parent"][v]] >= MARGIN:
                    assert tr["token"][v] == am[tr["parent"][v]], (rounds, v)
                    checked += 1
        history[hist_len:hist_len + len(toks)] = torch.tensor(toks, dtype=torch.int32, device="cuda")
        hist_len += len(toks)
        out.extend(toks)
        rounds += 1
    assert cs.get_status(dm.h) == 0
    first_diff = next((i for i in range(steps) if out[i] != truth[i]), None)
    if first_diff is not None:
        assert min(margins[: first_diff + 1]) < MARGIN, (first_diff, out[:steps], truth[:steps])
    assert checked > 0 and rounds < steps
    P, T = cs.kv_length(kv.h)
    assert T == 0 and P == n0 + len(out) - 1
    sch.close()
    kv.close()
    dm.close()
