"""GPU parity on a model whose residual projections do not split K over CTA pairs: with F = 64 the
down projection has a single 64-column k-block, so the residual projections stay unpaired, every
CTA runs the whole K of its Wo / Wdown rows, and the projection chain finishes them with its
unpaired residual epilogue (the path models wider than d = 6080 take; the 7B, 13B and tiny models
all pair).  d = 128 (two heads of 64), V = 512, 2 layers; prefix, tree verify, greedy acceptance and
compaction against the fp64 oracle (Sec. 4.2), logits within 2e-2 of the oracle's range."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

SH = synth.ModelShape(2, 128, 2, 64, 64, 512)
SEED = 4242
TOL_BF16, MARGIN = 2e-2, 1e-3


@pytest.fixture(scope="module")
def cs():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2510_26843_gb300 as m

    m.load_library()
    return m


def _i32(a):
    return torch.tensor(np.asarray(a, dtype=np.int32), device="cuda")


def test_unpaired_residual_projections(cs):
    from paper_2510_26843_gb300.workload import DeviceKV, DeviceModel

    dm = DeviceModel(SH, SEED)
    ow = oracle.Weights.from_seed(SEED, SH, keep_layers=SH.n_layers)
    kv = DeviceKV(dm, 256)
    okv = oracle.KVCache(SH.n_layers, SH.n_heads, SH.head_dim, 256)

    def step(toks, parent):
        n = len(toks)
        logits = torch.full((n, SH.vocab), float("nan"), device="cuda")
        cs.tree_step(dm.h, kv.h, _i32(toks), _i32(parent), n, None, 0, logits)
        torch.cuda.synchronize()
        return logits.cpu().numpy().astype(np.float64)

    def rel_err(got, ref):
        return np.max(np.abs(got - ref) / np.ptp(ref, axis=1, keepdims=True), axis=1)

    # a 40-token prefix committed through one chain step on both sides
    prefix = synth.tokens(SEED, 40, SH.vocab)
    got = step(prefix, synth.chain(40))
    ref = oracle.tree_step(ow, okv, prefix, synth.chain(40))
    assert np.all(rel_err(got, ref) < TOL_BF16), rel_err(got, ref).max()
    acc = _i32([40, *range(40), 0])
    cs.kv_compact(kv.h, acc)
    oracle.kv_compact(okv, list(range(40)))
    # a 33-node tree (a ragged tail past 32 tokens)
    parent = synth.tree(SEED + 1, 33, 4)
    toks = synth.tokens(SEED + 1, 33, SH.vocab)
    got = step(toks, parent)
    ref = oracle.tree_step(ow, okv, toks, parent)
    assert np.all(rel_err(got, ref) < TOL_BF16), rel_err(got, ref).max()
    out = torch.zeros(35, dtype=torch.int32, device="cuda")
    cs.accept_greedy(dm.h, None, _i32(toks), _i32(parent), 33, out)
    torch.cuda.synchronize()
    L = int(out[0])
    gpu_path = out[1:1 + L].cpu().tolist()
    path, bonus = oracle.accept_greedy(oracle.argmax_lowest(ref), toks, parent)
    if np.all(oracle.top2_margin(ref)[path] >= MARGIN):
        assert gpu_path == path and int(out[L + 1]) == bonus
    cs.kv_compact(kv.h, out)
    assert cs.kv_length(kv.h) == (40 + L, 0)
    assert cs.get_status(dm.h) == 0
    kv.close()
    dm.close()
