"""Bounds checks of the step's outputs on the GPU (in place of a memory checker): guard words around
every buffer a tree step, the greedy acceptance and the compaction write, and around the cache slots
they must not touch, keep their exact bit patterns (Sec. 4.2's verify / accept / compact, tiny model,
bf16 and W8A8 modes, full and ragged trees)."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

SH = synth.TINY
SEED = 777
F32_GUARD = np.int32(0x7FC0_0BAD)  # a NaN with a payload: no kernel writes it
I16_GUARD = 0x7BAD
I32_GUARD = -123456789


@pytest.fixture(scope="module")
def cs():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2510_26843_gb300 as m

    m.load_library()
    return m


@pytest.fixture(scope="module")
def dm(cs):
    from paper_2510_26843_gb300.workload import DeviceModel

    d = DeviceModel(SH, SEED, with_int8=True)
    yield d
    d.close()


def _i32(a):
    return torch.tensor(np.asarray(a, dtype=np.int32), device="cuda")


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("n", [1, 17, 64])
def test_outputs_stay_in_bounds(cs, dm, mode, n):
    from paper_2510_26843_gb300.workload import DeviceKV

    P, cap = 100, 256
    kv = DeviceKV(dm, cap)
    kv.load_random_prefix(SEED, P)
    # guard the cache slots beyond the tree on every layer; remember the prefix
    before = []
    for l in range(SH.n_layers):
        K, V = kv.layer(l)
        for t in (K, V):
            t[:, P + n:, :] = I16_GUARD
            before.append(t[:, :P, :].clone())
    torch.cuda.synchronize()
    parent = synth.tree(SEED + n, n, 8) if n > 1 else np.array([-1])
    toks = synth.tokens(SEED + n, n, SH.vocab)
    # logits with one guard row before and after
    lg = torch.empty((n + 2, SH.vocab), dtype=torch.float32, device="cuda")
    lg.view(torch.int32).fill_(int(F32_GUARD))
    cs.tree_step(dm.h, kv.h, _i32(toks), _i32(parent), n, None, mode, lg[1:n + 1])
    # acceptance output [L, path..., bonus] (<= n + 2 words) between guard words
    acc = torch.full((n + 4,), I32_GUARD, dtype=torch.int32, device="cuda")
    cs.accept_greedy(dm.h, None, _i32(toks), _i32(parent), n, acc[1:n + 3])
    torch.cuda.synchronize()
    g = lg.view(torch.int32).cpu().numpy()
    assert np.all(g[0] == F32_GUARD) and np.all(g[n + 1] == F32_GUARD)
    assert np.all(np.isfinite(lg[1:n + 1].cpu().numpy()))
    a = acc.cpu().numpy()
    assert a[0] == I32_GUARD and a[n + 3] == I32_GUARD
    L = int(a[1])
    assert 1 <= L <= n
    assert np.all(a[L + 3:n + 3] == I32_GUARD)  # words past [L, path, bonus] untouched
    cs.kv_compact(kv.h, acc[1:n + 3])
    torch.cuda.synchronize()
    assert cs.kv_length(kv.h) == (P + L, 0)
    assert cs.get_status(dm.h) == 0
    i = 0
    for l in range(SH.n_layers):
        K, V = kv.layer(l)
        for t in (K, V):
            assert torch.equal(t[:, :P, :], before[i])  # the committed prefix is never written
            assert bool((t[:, P + n:, :] == I16_GUARD).all())  # nor any slot past the tree
            i += 1
    kv.close()
