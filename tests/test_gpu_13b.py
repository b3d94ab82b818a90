"""GPU parity at the Llama-13B shapes (d=5120, 40 heads x 128, F=13824, V=32000) against the CPU oracle,
in the launch configuration the benchmark times (CUDA graphs + programmatic dependent launch).

The model is the first two layers of the seeded 13B-shaped model, so the oracle stays fast while every
projection, tile count and the attention run at 13B sizes:

  * verify step, prefix 4096, 64-node tree (depth <= 8): logits, acceptance, compaction byte-exact;
  * the cascade's sparse draft on the same model (W8A8 with one of the two layers on), two tree levels
    appended one after the other under the nesting rule.

Tolerances as elsewhere: 2e-2 (bf16) / 5e-2 (int8) of the oracle's logit range; indices bit-exact
unless the oracle's top-2 margin is below 1e-3.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

SEED = 1313
SH13 = synth.ModelShape(2, 5120, 40, 128, 13824, 32000)
TOL_BF16, TOL_INT8, MARGIN = 2e-2, 5e-2, 1e-3
P = 4096


@pytest.fixture(scope="module")
def cs():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2510_26843_gb300 as m

    m.load_library()
    return m


@pytest.fixture(scope="module")
def dm13(cs):
    from paper_2510_26843_gb300.workload import DeviceModel

    dm = DeviceModel(SH13, SEED, with_int8=True)
    cs.set_options(dm.h, cs.OPT_PDL | cs.OPT_GRAPHS)
    yield dm
    dm.close()


@pytest.fixture(scope="module")
def ow13():
    return oracle.Weights.from_seed(SEED, SH13, keep_layers=2)


def _i32(a):
    return torch.tensor(np.asarray(a, dtype=np.int32), device="cuda")


def rel_err(got, ref):
    return np.max(np.abs(got - ref) / np.ptp(ref, axis=1, keepdims=True), axis=1)


def oracle_cache(extra):
    okv = oracle.KVCache(SH13.n_layers, SH13.n_heads, SH13.head_dim, P + extra)
    for l in range(SH13.n_layers):
        k = synth.bf16_to_f32(synth.prefix_kv_bf16(SEED, SH13, l, "k", P)).astype(np.float64)
        v = synth.bf16_to_f32(synth.prefix_kv_bf16(SEED, SH13, l, "v", P)).astype(np.float64)
        okv.load_prefix(l, k, v)
    return okv


def gpu_step(cs, dm, kv, toks, parent, mask=None, mode=0):
    n = len(toks)
    t, p = _i32(toks), _i32(parent)
    logits = torch.full((n, SH13.vocab), float("nan"), device="cuda")
    cs.tree_step(dm.h, kv.h, t, p, n, mask, mode, logits)
    torch.cuda.synchronize()
    return logits.cpu().numpy().astype(np.float64), t, p


def test_13b_verify_accept_compact(cs, dm13, ow13):
    from paper_2510_26843_gb300.workload import DeviceKV

    n = 64
    kv = DeviceKV(dm13, P + 2 * n)
    kv.load_random_prefix(SEED, P)
    parent = synth.tree(SEED, n, 8)
    toks = synth.tokens(SEED, n, SH13.vocab)
    got, t, p = gpu_step(cs, dm13, kv, toks, parent)
    K_last, V_last = (x[:, P:P + n].clone() for x in kv.layer(SH13.n_layers - 1))
    acc = torch.zeros(n + 2, dtype=torch.int32, device="cuda")
    cs.accept_greedy(dm13.h, None, t, p, n, acc)
    cs.kv_compact(kv.h, acc)
    torch.cuda.synchronize()
    L = int(acc[0])
    gpu_path = acc[1:1 + L].cpu().tolist()
    assert cs.kv_length(kv.h) == (P + L, 0)
    K_new, V_new = kv.layer(SH13.n_layers - 1)
    for k, j in enumerate(gpu_path):
        assert torch.equal(K_new[:, P + k], K_last[:, j]) and torch.equal(V_new[:, P + k], V_last[:, j])
    assert cs.get_status(dm13.h) == 0

    ref = oracle.tree_step(ow13, oracle_cache(n), toks, parent)
    err = rel_err(got, ref)
    assert np.all(err < TOL_BF16), err.max()
    path, bonus = oracle.accept_greedy(oracle.argmax_lowest(ref), toks, parent)
    if np.all(oracle.top2_margin(ref)[path] >= MARGIN):
        assert gpu_path == path and int(acc[L + 1]) == bonus
    kv.close()


def test_13b_cascade_drafts(cs, dm13, ow13):
    """The sparse draft of a cascade round (W8A8, one of the two layers on) drafts a tree level by level:
    the second level is appended under the first, allowed because the same layer wrote the ancestors."""
    from paper_2510_26843_gb300.workload import DeviceKV

    kv = DeviceKV(dm13, P + 64)
    kv.load_random_prefix(SEED, P)
    okv = oracle_cache(64)
    m2 = np.array([1, 0], dtype=np.uint8)  # d2: one of two layers on
    lev1_parent, lev1_toks = np.array([-1, 0, 0, 1]), synth.tokens(SEED + 3, 4, SH13.vocab)
    got1, _, _ = gpu_step(cs, dm13, kv, lev1_toks, lev1_parent, mask=m2, mode=1)
    assert cs.get_status(dm13.h) == 0
    ref1 = oracle.tree_step(ow13, okv, lev1_toks, lev1_parent, skip_mask=m2, quant_mode=1)
    assert np.all(rel_err(got1, ref1) < TOL_INT8), rel_err(got1, ref1).max()
    # the next level hangs under tree slots 1..3; d2's active layer wrote their K/V, so d2 may append
    lev2_parent, lev2_toks = np.array([1, 2, 3, 3]), synth.tokens(SEED + 4, 4, SH13.vocab)
    got2, _, _ = gpu_step(cs, dm13, kv, lev2_toks, lev2_parent, mask=m2, mode=1)
    assert cs.get_status(dm13.h) == 0
    ref2 = oracle.tree_step(ow13, okv, lev2_toks, lev2_parent, skip_mask=m2, quant_mode=1)
    assert np.all(rel_err(got2, ref2) < TOL_INT8), rel_err(got2, ref2).max()
    kv.close()
