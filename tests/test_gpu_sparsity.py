"""Activation sparsity on the GPU (App. C: the TEAL draft of the DSIA family).

* The rule itself, `casspec_sparsify_rows`, against `oracle.sparsify_rows` on the same fp32 values
  (hi + lo of the split activation): the set of zeroed entries is identical, bit for bit, including
  rows full of exact ties (the lower index kept) and rows of zeros; every other entry is unchanged.
* Whole steps with `casspec_set_act_sparsity` against `oracle.tree_step(act_sparsity=s)`.  Which entries
  a row loses is decided by comparing magnitudes, so an input whose z-th and (z+1)-th smallest
  magnitudes lie closer than the rounding difference between the two sides can lose either one.  The
  oracle shows it against itself: rounding only its attention operands to bf16 moves the tiny model's
  logits by up to 0.17 of their range at s = 0.5 (median up to 0.05).  So:
  - strict cases, within TOL_BF16 of the fp64 oracle: steps whose every decision has a relative margin
    (gap between those two magnitudes over the larger) well above the GPU's rounding of that input,
    asserted from the oracle's trace before the comparison: FFN-only layers at s = 0.99 (the gate/up
    and down inputs are the chain's fp32-accurate values; margins >= 5e-4) and one full layer at
    s = 0.99 (the attention output o, bf16 attention operands, changes by <= 5e-4 relative; its margin
    is 5e-3 on that tree);
  - the full model at s = 0.99, 0.5 and 0.2: within TOL_INT8_DEEP, the fixed bound for steps whose
    integer decisions follow the values (as for a W8A8 stack), with a median error under half the
    distance to the dense step (0.05 at s = 0.2, 0.21 at s = 0.5; the oracle's own bf16 variant has a
    median of up to 0.046);
  - s = 0.001 (z = floor(sK) = 0 for every K here): the sparsify launches run and zero nothing, and the
    logits equal the dense step's bit for bit; s = 0 again restores the dense step bit for bit;
* Quantised steps with sparsity (App. C's mixed drafts, W8A8 and W4A4): the selection is taken on the
  bf16 activation the quantiser then reads (the oracle's reading for quantised drafts):
  - s = 0.001 (nothing zeroed): the sparse path (norm -> bf16 row -> selection -> row quantiser) gives
    the fused norm-quantiser's codes, so the logits equal the dense quantised step's bit for bit;
  - FFN-only layers at s = 0.99: within TOL_INT8 of the oracle (the dense quantised bound);
  - the full model at s = 0.5 against the bf16-cache oracle: TOL_INT8_DEEP (W8A8) or TOL_W4 (W4A4,
    whose attention-output codes follow the GPU's bf16 probabilities), with a median under half the
    distance to the dense quantised step.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

SH = synth.TINY
SEED = 2468
TOL_BF16 = 2e-2
TOL_INT8_DEEP = 0.2  # as test_gpu_7b.TOL_INT8_DEEP
TOL_W4 = 0.3  # as test_gpu_step.TOL_W4


@pytest.fixture(scope="module")
def cs():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2510_26843_gb300 as m

    m.load_library()
    return m


def _split(v32: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """fp32 values -> (hi, lo) bf16 bit patterns with hi + lo == v in fp32 where representable."""
    hi = synth.bf16_bits_rne(v32)
    r = v32 - synth.bf16_to_f32(hi)
    lo = synth.bf16_bits_rne(r.astype(np.float32))
    return hi, lo


@pytest.mark.parametrize("K,n,s,kind", [(64, 3, 0.5, "ties"), (256, 17, 0.25, "ties"), (4096, 64, 0.5, "mixed"),
                                        (11008, 8, 0.9, "mixed"), (1000, 5, 0.999, "ties"), (16384, 2, 0.5, "zeros")])
def test_rule_matches_oracle(cs, K, n, s, kind):
    rng = np.random.default_rng(K + n)
    if kind == "ties":  # a handful of exact values: long runs of equal magnitudes of both signs
        v = rng.choice(np.array([0.0, 0.25, -0.25, 0.5, -0.5, 1.0, -2.0], dtype=np.float32), size=(n, K))
    elif kind == "zeros":
        v = np.zeros((n, K), dtype=np.float32)
        v[:, ::7] = rng.standard_normal((n, len(range(0, K, 7)))).astype(np.float32)
    else:  # normal values carried in both planes, with some ties
        v = rng.standard_normal((n, K)).astype(np.float32)
        v[:, ::5] = np.float32(0.75)
    hi, lo = _split(v)
    x = np.zeros((128, K), dtype=np.uint16)
    x[:n], x[64:64 + n] = hi, lo
    xd = torch.from_numpy(x.view(np.int16)).cuda()
    cs.sparsify_rows(xd, K, n, K, s)
    torch.cuda.synchronize()
    got = xd.cpu().numpy().view(np.uint16)
    vals = (synth.bf16_to_f32(hi).astype(np.float32) + synth.bf16_to_f32(lo).astype(np.float32)).astype(np.float64)
    ref = oracle.sparsify_rows(vals, s)
    zeroed_ref = (ref == 0.0) & (vals != 0.0)
    zeroed_gpu = (got[:n] == 0) & (got[64:64 + n] == 0) & ((hi != 0) | (lo != 0))
    assert np.array_equal(zeroed_gpu, zeroed_ref)
    keep = ~zeroed_ref
    assert np.array_equal(got[:n][keep], hi[keep]) and np.array_equal(got[64:64 + n][keep], lo[keep])
    assert np.all(got[n:64] == 0) and np.all(got[64 + n:] == 0)  # rows past n untouched


def _margin(trace: dict, s: float, keys) -> float:
    """Smallest relative gap, over the sparsified rows of the oracle step, between the z-th and the
    (z+1)-th smallest magnitude (exact ties excluded: both sides see the same values there and keep
    the lower index)."""
    m = 1.0
    for l in trace:
        for key in keys:
            if key in trace[l]:
                a = np.sort(np.abs(trace[l][key]), axis=1)
                z = int(np.floor(s * a.shape[1] + 1e-9))
                g = (a[:, z] - a[:, z - 1]) / a[:, z]
                g = g[g > 0]
                m = min(m, float(g.min()) if g.size else 1.0)
    return m


def test_sparse_steps_match_oracle(cs):
    from paper_2510_26843_gb300.workload import DeviceKV, DeviceModel

    dm = DeviceModel(SH, SEED, with_int8=True)
    ow = oracle.Weights.from_seed(SEED, SH, keep_layers=SH.n_layers)

    def run(s, toks, parent, mode=0, mask=None):
        kv = DeviceKV(dm, 256)
        kv.load_random_prefix(SEED, 96)
        n = len(toks)
        lg = torch.empty((n, SH.vocab), dtype=torch.float32, device="cuda")
        cs.set_act_sparsity(dm.h, s)
        t = torch.tensor(np.asarray(toks, dtype=np.int32), device="cuda")
        p = torch.tensor(np.asarray(parent, dtype=np.int32), device="cuda")
        rc = cs.tree_step(dm.h, kv.h, t, p, n, mask, mode, lg, check=False)
        torch.cuda.synchronize()
        kv.close()
        return rc, lg.cpu().numpy().astype(np.float64)

    def oracle_cache():
        okv = oracle.KVCache(SH.n_layers, SH.n_heads, SH.head_dim, 256)
        for l in range(SH.n_layers):
            k = synth.bf16_to_f32(synth.prefix_kv_bf16(SEED, SH, l, "k", 96)).astype(np.float64)
            v = synth.bf16_to_f32(synth.prefix_kv_bf16(SEED, SH, l, "v", 96)).astype(np.float64)
            okv.load_prefix(l, k, v)
        return okv

    def rel(a, ref):
        return np.max(np.abs(a - ref) / np.ptp(ref, axis=1, keepdims=True), axis=1)

    ffn_only = np.array([1 | cs.SKIP_ATTN, 1 | cs.SKIP_ATTN], np.uint8)
    first_full = np.array([1, 0], np.uint8)
    for tseed, mask, need in ((6, ffn_only, {"xn2": 5e-4, "u": 5e-4}), (77, ffn_only, {"xn2": 5e-4, "u": 5e-4}),
                              (7, first_full, {"xn": 1e-3, "o": 5e-3})):
        parent = synth.tree(tseed, 24, 6)
        toks = synth.tokens(tseed, 24, SH.vocab)
        tr = {}
        ref = oracle.tree_step(ow, oracle_cache(), toks, parent, skip_mask=mask, act_sparsity=0.99, trace=tr)
        for key, bound in need.items():
            assert _margin(tr, 0.99, (key,)) >= bound, (tseed, key)
        dense = oracle.tree_step(ow, oracle_cache(), toks, parent, skip_mask=mask)
        assert np.median(rel(dense, ref)) > 0.1  # the sparse step is far from the dense one
        rc, got = run(0.99, toks, parent, mask=mask)
        assert rc == 0
        assert np.all(rel(got, ref) < TOL_BF16), (tseed, rel(got, ref).max())

    for tseed in (SEED, 77):
        parent = synth.tree(tseed, 24, 6)
        toks = synth.tokens(tseed, 24, SH.vocab)
        dense = oracle.tree_step(ow, oracle_cache(), toks, parent)
        for s in (0.99, 0.5, 0.2):
            rc, got = run(s, toks, parent)
            assert rc == 0
            ref = oracle.tree_step(ow, oracle_cache(), toks, parent, act_sparsity=s)
            err = rel(got, ref)
            assert np.all(err < TOL_INT8_DEEP), (tseed, s, err.max())
            assert np.median(err) < 0.5 * np.median(rel(dense, ref)), (tseed, s, np.median(err))
    _, dense0 = run(0.0, toks, parent)
    _, none0 = run(0.001, toks, parent)
    _, dense1 = run(0.0, toks, parent)
    assert np.array_equal(dense0, none0) and np.array_equal(dense0, dense1)
    assert cs.get_status(dm.h) == 0
    dm.close()


def test_quantised_sparse_steps_match_oracle(cs):
    from paper_2510_26843_gb300.workload import DeviceKV, DeviceModel

    dm = DeviceModel(SH, SEED, with_int8=True)
    ow = oracle.Weights.from_seed(SEED, SH, keep_layers=SH.n_layers)
    TOL_INT8 = 5e-2

    def run(s, toks, parent, mode, mask=None):
        kv = DeviceKV(dm, 256)
        kv.load_random_prefix(SEED, 96)
        n = len(toks)
        lg = torch.empty((n, SH.vocab), dtype=torch.float32, device="cuda")
        cs.set_act_sparsity(dm.h, s)
        t = torch.tensor(np.asarray(toks, dtype=np.int32), device="cuda")
        p = torch.tensor(np.asarray(parent, dtype=np.int32), device="cuda")
        rc = cs.tree_step(dm.h, kv.h, t, p, n, mask, mode, lg, check=False)
        torch.cuda.synchronize()
        kv.close()
        assert rc == 0
        return lg.cpu().numpy().astype(np.float64)

    def oracle_cache():
        okv = oracle.KVCache(SH.n_layers, SH.n_heads, SH.head_dim, 256)
        for l in range(SH.n_layers):
            k = synth.bf16_to_f32(synth.prefix_kv_bf16(SEED, SH, l, "k", 96)).astype(np.float64)
            v = synth.bf16_to_f32(synth.prefix_kv_bf16(SEED, SH, l, "v", 96)).astype(np.float64)
            okv.load_prefix(l, k, v)
        return okv

    def rel(a, ref):
        return np.max(np.abs(a - ref) / np.ptp(ref, axis=1, keepdims=True), axis=1)

    ffn_only = np.array([1 | cs.SKIP_ATTN, 1 | cs.SKIP_ATTN], np.uint8)
    parent = synth.tree(6, 24, 6)
    toks = synth.tokens(6, 24, SH.vocab)
    for mode in (1, 2):
        dense_q = run(0.0, toks, parent, mode)
        np.testing.assert_array_equal(run(0.001, toks, parent, mode), dense_q)
        got = run(0.99, toks, parent, mode, mask=ffn_only)
        ref = oracle.tree_step(ow, oracle_cache(), toks, parent, skip_mask=ffn_only, quant_mode=mode,
                               act_sparsity=0.99)
        assert np.all(rel(got, ref) < TOL_INT8), (mode, rel(got, ref).max())
        got = run(0.5, toks, parent, mode)
        ref = oracle.tree_step(ow, oracle_cache(), toks, parent, quant_mode=mode, act_sparsity=0.5,
                               attn_bf16=True)
        dense = oracle.tree_step(ow, oracle_cache(), toks, parent, quant_mode=mode, attn_bf16=True)
        err = rel(got, ref)
        assert np.all(err < (TOL_INT8_DEEP if mode == 1 else TOL_W4)), (mode, err.max())
        assert np.median(err) < 0.5 * np.median(rel(dense, ref)), (mode, np.median(err))
    cs.set_act_sparsity(dm.h, 0.0)
    assert cs.get_status(dm.h) == 0
    dm.close()
