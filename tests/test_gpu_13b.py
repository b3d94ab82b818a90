"""GPU parity on the Llama-13B-shaped model (40 layers, d=5120, 40 heads x 128, F=13824, V=32000,
prefix 4096) against the CPU oracle, in the launch configuration the benchmark times (CUDA graphs +
programmatic dependent launch): one whole cascade round of the 13B configuration (Sec. 4.2), every
step of it compared with the oracle:

  * the sparse draft d2 (60% of layers skipped, W8A8) drafts the 64-node tree (depth <= 8) level by
    level, each level appended under the previous ones (allowed: d2's layers wrote the ancestors);
  * the tree is reset and the denser draft d1 (40% skipped, bf16; its layers contain d2's) re-checks
    all 64 nodes in one step;
  * the tree is reset and the full 40-layer model verifies all 64 nodes; greedy acceptance and
    compaction follow (moved K/V byte-identical to the tree slots they came from).

Tolerances: bf16 steps 2e-2 of the oracle's logit range; the 16-layer W8A8 draft levels against the
oracle with the bf16 cache (attn_bf16) at the fixed bound TOL_INT8_DEEP of test_gpu_7b.py; accepted
path and bonus bit-exact unless the oracle's top-2 margin on the path is below 1e-3.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

SEED = 1313
SH13 = synth.LLAMA13B
TOL_BF16, MARGIN = 2e-2, 1e-3
TOL_INT8_DEEP = 0.2  # as test_gpu_7b.TOL_INT8_DEEP
CASCADE_SKIP = (0.4, 0.6)  # d1 (bf16), d2 (W8A8)
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
    cs.set_options(dm.h, cs.OPT_PDL | cs.OPT_GRAPHS | cs.OPT_W4_TC | cs.OPT_W8_TC)
    yield dm
    dm.close()


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


def level_order(parent, toks):
    """The tree renumbered by depth (parents first) and each level's [start, end) node range."""
    n = len(parent)
    depth = [0] * n
    for i in range(1, n):
        depth[i] = depth[parent[i]] + 1
    order = sorted(range(n), key=lambda i: (depth[i], i))
    pos = {old: new for new, old in enumerate(order)}
    par = np.array([-1 if parent[o] < 0 else pos[int(parent[o])] for o in order], dtype=np.int64)
    tk = np.array([toks[o] for o in order], dtype=np.int64)
    levels, start = [], 0
    for dd in range(max(depth) + 1):
        cnt = depth.count(dd)
        levels.append((start, start + cnt))
        start += cnt
    return par, tk, levels


def test_13b_cascade_round(cs, dm13):
    from paper_2510_26843_gb300.workload import DeviceKV

    n = 64
    parent, toks, levels = level_order(synth.tree(SEED, n, 8), synth.tokens(SEED, n, SH13.vocab))
    m1, m2 = synth.skip_masks(SEED, SH13.n_layers, list(CASCADE_SKIP))
    assert np.all(m1[m2 > 0] > 0)  # nested: d2's layers are d1's
    kv = DeviceKV(dm13, P + 2 * n)
    kv.load_random_prefix(SEED, P)
    okv = oracle_cache(n)
    # int8 weights of d2's 16 layers are derived once for all levels
    w_d2 = oracle.Weights.from_seed(SEED, SH13, keep_layers=int(m2.sum()))
    w = oracle.Weights.from_seed(SEED, SH13, keep_layers=1)

    # d2 drafts the tree level by level (node ids of a level are tree slots a .. b-1)
    for a, b in levels:
        par = parent[a:b]
        got, _, _ = gpu_step(cs, dm13, kv, toks[a:b], par, mask=m2, mode=1)
        assert cs.get_status(dm13.h) == 0
        ref = oracle.tree_step(w_d2, okv, toks[a:b], par, skip_mask=m2, quant_mode=1, attn_bf16=True)
        err = rel_err(got, ref)
        print(f"13B d2 level [{a}, {b}): per-row error / logit range max {err.max():.4f}")
        assert np.all(err < TOL_INT8_DEEP), (a, err.max())
    del w_d2
    # d1 re-checks every node of the tree
    cs.kv_reset_tree(kv.h)
    okv.reset_tree()
    got, _, _ = gpu_step(cs, dm13, kv, toks, parent, mask=m1, mode=0)
    assert cs.get_status(dm13.h) == 0
    ref = oracle.tree_step(w, okv, toks, parent, skip_mask=m1)
    err = rel_err(got, ref)
    print(f"13B d1 re-check: max error {err.max():.4f}")
    assert np.all(err < TOL_BF16), err.max()
    # the full model verifies the tree; acceptance and compaction
    cs.kv_reset_tree(kv.h)
    okv.reset_tree()
    got, t, p = gpu_step(cs, dm13, kv, toks, parent)
    K_last, V_last = (x[:, P:P + n].clone() for x in kv.layer(SH13.n_layers - 1))
    acc = torch.zeros(n + 2, dtype=torch.int32, device="cuda")
    cs.accept_greedy(dm13.h, None, t, p, n, acc)
    cs.kv_compact(kv.h, acc)
    torch.cuda.synchronize()
    assert cs.get_status(dm13.h) == 0
    L = int(acc[0])
    gpu_path = acc[1:1 + L].cpu().tolist()
    assert cs.kv_length(kv.h) == (P + L, 0)
    K_new, V_new = kv.layer(SH13.n_layers - 1)
    for k, j in enumerate(gpu_path):
        assert torch.equal(K_new[:, P + k], K_last[:, j]) and torch.equal(V_new[:, P + k], V_last[:, j])
    ref = oracle.tree_step(w, okv, toks, parent)
    err = rel_err(got, ref)
    print(f"13B verify (40 layers): max error {err.max():.4f}")
    assert np.all(err < TOL_BF16), err.max()
    path, bonus = oracle.accept_greedy(oracle.argmax_lowest(ref), toks, parent)
    if np.all(oracle.top2_margin(ref)[path] >= MARGIN):
        assert gpu_path == path and int(acc[L + 1]) == bonus
    kv.close()


@pytest.mark.parametrize("n", [8, 64])
def test_13b_w8a8_tensor_core_path_equals_integer_path(cs, dm13, n):
    """The 40-layer 13B W8A8 step on both paths (K = 5120 and 13824: a gate/up output sums up to five
    exact 1024-column accumulators): the same codes and scales, exact int32 sums on both, so the
    logits are bitwise equal, at the 16- and 64-token tiles."""
    from paper_2510_26843_gb300.workload import DeviceKV

    parent = synth.tree(SEED + n, n, 8)
    toks = synth.tokens(SEED + n, n, SH13.vocab)
    base = cs.OPT_PDL | cs.OPT_GRAPHS | cs.OPT_W4_TC
    out = []
    for flags in (base | cs.OPT_W8_TC, base):
        cs.set_options(dm13.h, flags)
        kv = DeviceKV(dm13, P + 128)
        kv.load_random_prefix(SEED, P)
        got, _, _ = gpu_step(cs, dm13, kv, toks, parent, mode=1)
        assert cs.get_status(dm13.h) == 0
        kv.close()
        out.append(got)
    cs.set_options(dm13.h, base | cs.OPT_W8_TC)
    assert np.all(np.isfinite(out[0]))
    np.testing.assert_array_equal(out[0], out[1])
