"""Pins of the CPU oracle against what the paper and the mathematics fix (no GPU).

Each test compares the oracle with something other than itself: a textbook causal forward written
with torch library routines (tests/torch_ref.py), closed forms, hand-derived fixtures, or brute
force.  Together they are chosen so that a dropped term, a wrong sign or index, or a transposed
operand anywhere in the oracle fails at least one of them.
"""
from __future__ import annotations

import itertools
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
import synth
from tests.torch_ref import CausalLM

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
SEED = 1234


# ------------------------------------------------------------------------------------------------
# generator
# ------------------------------------------------------------------------------------------------
def test_splitmix64_published_vector():
    # SplitMix64 seeded with 0 (state advanced by GAMMA before mixing): first outputs of the
    # reference generator.
    assert synth.u64(0, 0) == 0xE220A8397B1DCDAF
    assert synth.u64(0, 1) == 0x6E789E6AA1B965F4
    assert synth.u64(0, 2) == 0x06C45D188009454F


def test_fill_matches_scalar_definition_and_subranges():
    key = synth.stream_key(7, synth.K_WQKV, 3)
    full = synth.fill_normal_bf16(key, 0, 5000, 0.02)
    for i in [0, 1, 2, 999, 4999]:
        assert full[i] == synth.normal_bf16_scalar(key, i, 0.02)
    assert np.array_equal(full[1234:4321], synth.fill_normal_bf16(key, 1234, 4321 - 1234, 0.02))
    big = synth.bf16_to_f32(synth.fill_normal_bf16(key, 0, 1 << 20, 0.02))
    assert abs(big.std() - 0.02) < 2e-4 and abs(big.mean()) < 2e-4


# ------------------------------------------------------------------------------------------------
# elementwise pieces vs closed forms / library routines
# ------------------------------------------------------------------------------------------------
def test_rmsnorm_closed_form_and_library():
    x = np.array([[3.0, 4.0]])
    np.testing.assert_allclose(oracle.rmsnorm(x, np.ones(2), 0.0), [[3 / math.sqrt(12.5), 4 / math.sqrt(12.5)]])
    r = np.random.default_rng(0).standard_normal((5, 64))
    g = np.random.default_rng(1).standard_normal(64)
    ref = F.rms_norm(torch.from_numpy(r), (64,), torch.from_numpy(g), 1e-5).numpy()
    np.testing.assert_allclose(oracle.rmsnorm(r, g, 1e-5), ref, rtol=1e-12, atol=1e-12)


def test_rope_closed_form_and_properties():
    # h = 2: one pair rotated by angle pos (frequency base^0 = 1)
    out = oracle.rope(np.array([[1.0, 0.0], [1.0, 0.0]]), np.array([0, 3]), 10000.0)
    np.testing.assert_allclose(out, [[1.0, 0.0], [math.cos(3), math.sin(3)]], atol=1e-15)
    rng = np.random.default_rng(2)
    q, k = rng.standard_normal(128), rng.standard_normal(128)
    # norm preserved
    rq = oracle.rope(q[None], np.array([17]), 10000.0)[0]
    assert abs(np.linalg.norm(rq) - np.linalg.norm(q)) < 1e-12
    # q.k depends only on the position difference
    dots = [oracle.rope(q[None], np.array([m]), 1e4)[0] @ oracle.rope(k[None], np.array([m - 5]), 1e4)[0]
            for m in (5, 9, 100, 2047)]
    np.testing.assert_allclose(dots, dots[0], rtol=1e-10)
    # frequency index: pair j rotates by pos * base^(-2j/h)
    e = np.zeros(8)
    e[1] = 1.0  # pair (1, 5)
    r = oracle.rope(e[None], np.array([2]), 100.0)[0]
    ang = 2 * 100.0 ** (-2 * 1 / 8)
    np.testing.assert_allclose([r[1], r[5]], [math.cos(ang), math.sin(ang)], atol=1e-15)


def test_silu_closed_form():
    np.testing.assert_allclose(oracle.silu(np.array([0.0, 1.0, -1.0])),
                               [0.0, 1 / (1 + math.exp(-1)), -1 / (1 + math.exp(1))])
    x = np.linspace(-8, 8, 33)
    np.testing.assert_allclose(oracle.silu(x), F.silu(torch.from_numpy(x)).numpy(), rtol=1e-14)


# ------------------------------------------------------------------------------------------------
# quantisation
# ------------------------------------------------------------------------------------------------
def _nearest_f32(fr: Fraction) -> np.float32:
    c = np.float32(float(fr))
    cands = [np.nextafter(c, np.float32(-np.inf)), c, np.nextafter(c, np.float32(np.inf))]
    best = min(cands, key=lambda v: (abs(Fraction(float(v)) - fr), int(np.array(v).view(np.uint32)) & 1))
    return np.float32(best)


def _golden_quant_rows():
    rows = []
    for line in open(os.path.join(GOLDEN, "quant_rows.txt")):
        if line.startswith("#") or not line.strip():
            continue
        xs, qs = line.split("|")
        rows.append(([float(v) for v in xs.split()], [int(v) for v in qs.split()]))
    return rows


@pytest.mark.parametrize("which", ["f32", "f64"])
def test_quantizer_golden_rows(which):
    for xs, qs in _golden_quant_rows():
        x = np.array([xs], dtype=np.float32 if which == "f32" else np.float64)
        q, s = (oracle.quantize_rows_f32 if which == "f32" else oracle.quantize_rows_f64)(x)
        assert q.dtype == np.int8
        assert q[0].tolist() == qs, (xs, q[0].tolist(), qs)
        amax = max(abs(v) for v in xs)
        want = 0.0 if amax == 0 else (_nearest_f32(Fraction(amax) / 127) if which == "f32" else amax / 127)
        assert s[0] == want


def test_quantizer_properties_random():
    rng = np.random.default_rng(3)
    x = (rng.standard_normal((50, 300)) * rng.uniform(0.01, 10, (50, 1))).astype(np.float32)
    q, s = oracle.quantize_rows_f32(x)
    amax_idx = np.argmax(np.abs(x), axis=1)
    assert np.all(np.abs(q[np.arange(50), amax_idx]) == 127)
    assert np.all(np.sign(q[np.arange(50), amax_idx]) == np.sign(x[np.arange(50), amax_idx]))
    # every code is within half a step of x / scale (rounding error of one fp32 multiply)
    assert np.all(np.abs(q - x / s[:, None].astype(np.float64)) <= 0.5 + 1e-4)


def test_int4_quantizer_golden_rows_and_properties():
    for line in open(os.path.join(GOLDEN, "quant4_rows.txt")):
        if line.startswith("#") or not line.strip():
            continue
        xs, qs = line.split("|")
        x = np.array([[float(v) for v in xs.split()]], dtype=np.float32)
        want = [int(v) for v in qs.split()]
        for fn in (oracle.quantize_rows_f32, oracle.quantize_rows_f64):
            q, s = fn(x, 7)
            assert q[0].tolist() == want
            assert s[0] == float(np.max(np.abs(x))) / 7
    rng = np.random.default_rng(13)
    x = (rng.standard_normal((40, 200)) * rng.uniform(0.01, 10, (40, 1))).astype(np.float32)
    q, s = oracle.quantize_rows_f32(x, 7)
    i = np.argmax(np.abs(x), axis=1)
    assert np.all(np.abs(q[np.arange(40), i]) == 7) and np.abs(q).max() == 7
    assert np.all(np.abs(q - x / s[:, None].astype(np.float64)) <= 0.5 + 1e-5)


def test_sparsify_rows_bruteforce():
    """The floor(s K) smallest magnitudes become 0 (ties: the higher index goes first), checked against
    a plain selection loop on rows with many ties."""
    rng = np.random.default_rng(17)
    for _ in range(60):
        K = int(rng.integers(1, 24))
        x = rng.integers(-4, 5, (3, K)).astype(np.float64) * 0.5
        s = float(rng.choice([0.0, 0.25, 0.4, 0.5, 0.9]))
        got = oracle.sparsify_rows(x, s)
        z = int(math.floor(s * K + 1e-9))
        for r in range(3):
            kept = []
            for _ in range(K - z):  # repeatedly take the largest magnitude, lowest index on ties
                best = None
                for c in range(K):
                    if c in kept:
                        continue
                    if best is None or abs(x[r, c]) > abs(x[r, best]):
                        best = c
                kept.append(best)
            want = np.zeros(K)
            want[kept] = x[r, kept]
            assert np.array_equal(got[r], want), (x[r], s, got[r], want)
    assert np.array_equal(oracle.sparsify_rows(x, 0.0), x)


def test_w8a8_linear_bruteforce():
    rng = np.random.default_rng(4)
    qx = rng.integers(-127, 128, (3, 37), dtype=np.int64).astype(np.int8)
    qw = rng.integers(-127, 128, (5, 37), dtype=np.int64).astype(np.int8)
    sx, sw = rng.uniform(0.1, 1, 3), rng.uniform(0.1, 1, 5)
    y = oracle.linear_w8a8(qx, sx, qw, sw)
    for t, o in itertools.product(range(3), range(5)):
        acc = sum(int(qx[t, k]) * int(qw[o, k]) for k in range(37))
        assert y[t, o] == pytest.approx(acc * sx[t] * sw[o], rel=1e-15)
    # the integer sums are exact at the longest rows of the 13B shape, extreme codes included
    K = 13824
    qx = rng.integers(-127, 128, (4, K), dtype=np.int64)
    qx[0] = 127
    qw = rng.integers(-127, 128, (6, K), dtype=np.int64)
    qw[0] = 127
    qw[1] = -127
    y = oracle.linear_w8a8(qx.astype(np.int8), np.ones(4), qw.astype(np.int8), np.ones(6))
    exact = np.array([[int(np.dot(qx[t], qw[o])) for o in range(6)] for t in range(4)], dtype=np.int64)
    assert exact[0, 0] == K * 127 * 127
    assert np.array_equal(y, exact.astype(np.float64)) and np.array_equal(y.astype(np.int64), exact)


# ------------------------------------------------------------------------------------------------
# attention vs library sdpa
# ------------------------------------------------------------------------------------------------
def _kv(P, H=2, h=16, cap=64, layers=1):
    rng = np.random.default_rng(5)
    kv = oracle.KVCache(layers, H, h, cap)
    kv.load_prefix(0, rng.standard_normal((H, P, h)), rng.standard_normal((H, P, h)))
    return kv, rng


def test_attention_single_query_matches_sdpa():
    kv, rng = _kv(20)
    q = rng.standard_normal((1, 2, 16))
    kv.K[0][:, 20] = rng.standard_normal((2, 16))
    kv.V[0][:, 20] = rng.standard_normal((2, 16))
    kv.valid[0][20] = True
    o = oracle.tree_attention(q, kv, 0, [20], [frozenset([0])])
    K = torch.from_numpy(kv.K[0][:, :21])
    V = torch.from_numpy(kv.V[0][:, :21])
    ref = F.scaled_dot_product_attention(torch.from_numpy(q.transpose(1, 0, 2))[None], K[None], V[None])[0]
    np.testing.assert_allclose(o.transpose(1, 0, 2), ref.numpy(), rtol=1e-12, atol=1e-12)


def test_tree_attention_matches_masked_sdpa():
    P, n = 12, 6
    parent = np.array([-1, 0, 0, 1, 1, 2])
    kv, rng = _kv(P)
    q = rng.standard_normal((n, 2, 16))
    for i in range(n):
        kv.K[0][:, P + i] = rng.standard_normal((2, 16))
        kv.V[0][:, P + i] = rng.standard_normal((2, 16))
        kv.valid[0][P + i] = True
    depth, anc = oracle.tree_topology(parent, 0, [], [])
    assert depth == [0, 1, 1, 2, 2, 2]
    o = oracle.tree_attention(q, kv, 0, list(range(P, P + n)), anc)
    # explicit boolean mask built from the parent array by walking up
    mask = torch.zeros(n, P + n, dtype=torch.bool)
    mask[:, :P] = True
    for i in range(n):
        j = i
        while j != -1:
            mask[i, P + j] = True
            j = parent[j]
    K = torch.from_numpy(kv.K[0][:, :P + n])[None]
    V = torch.from_numpy(kv.V[0][:, :P + n])[None]
    ref = F.scaled_dot_product_attention(torch.from_numpy(q.transpose(1, 0, 2))[None], K, V, attn_mask=mask)[0]
    np.testing.assert_allclose(o.transpose(1, 0, 2), ref.numpy(), rtol=1e-12, atol=1e-12)


def test_tree_topology_rejects_bad_parents():
    for bad in ([0], [-1, 1], [-1, 5], [-1, -2]):
        with pytest.raises(ValueError):
            oracle.tree_topology(np.array(bad), 0, [], [])


# ------------------------------------------------------------------------------------------------
# whole step vs textbook causal decoding (tiny model)
# ------------------------------------------------------------------------------------------------
SH = synth.TINY


@pytest.fixture(scope="module")
def tiny():
    w = oracle.Weights.from_seed(SEED, SH, keep_layers=SH.n_layers)
    ref = CausalLM(SH, SEED)
    prefix = synth.prefix_tokens(SEED, 64, SH.vocab)
    return w, ref, prefix


def _prefilled(w, prefix, cap=256, mask=None):
    """Oracle cache after committing `prefix` via one chain tree step + compaction."""
    kv = oracle.KVCache(SH.n_layers, SH.n_heads, SH.head_dim, cap)
    logits = oracle.tree_step(w, kv, prefix, synth.chain(len(prefix)), skip_mask=mask)
    oracle.kv_compact(kv, list(range(len(prefix))))
    return kv, logits


def _root_path(parent, i):
    path = []
    while i != -1:
        path.append(i)
        i = parent[i]
    return path[::-1]


def test_chain_prefill_equals_causal_forward(tiny):
    w, ref, prefix = tiny
    _, logits = _prefilled(w, prefix)
    want = ref.forward(prefix)
    rng = np.ptp(want, axis=1, keepdims=True)
    assert np.max(np.abs(logits - want) / rng) < 1e-10


@pytest.mark.parametrize("tree_seed", [0, 1, 2])
def test_tree_nodes_equal_causal_decode_of_their_root_path(tiny, tree_seed):
    w, ref, prefix = tiny
    kv, _ = _prefilled(w, prefix)
    parent = synth.tree(tree_seed, 8, 4)
    toks = synth.tokens(tree_seed, 8, SH.vocab)
    logits = oracle.tree_step(w, kv, toks, parent)
    for i in range(8):
        seq = np.concatenate([prefix, toks[_root_path(parent, i)]])
        want = ref.forward(seq)[-1]
        assert np.max(np.abs(logits[i] - want)) / np.ptp(want) < 1e-10, i


def test_n1_equals_single_token_decode(tiny):
    w, ref, prefix = tiny
    kv, _ = _prefilled(w, prefix)
    logits = oracle.tree_step(w, kv, np.array([17]), np.array([-1]))
    want = ref.forward(np.concatenate([prefix, [17]]))[-1]
    assert np.max(np.abs(logits[0] - want)) / np.ptp(want) < 1e-10


def test_appended_draft_levels_equal_one_shot_tree(tiny):
    """Drafting a tree level by level (T > 0 appends) gives the same logits as one call."""
    w, ref, prefix = tiny
    parent = synth.tree(5, 8, 3)
    toks = synth.tokens(5, 8, SH.vocab)
    kv1, _ = _prefilled(w, prefix)
    one = oracle.tree_step(w, kv1, toks, parent)
    kv2, _ = _prefilled(w, prefix)
    parts = [oracle.tree_step(w, kv2, toks[a:b], parent[a:b]) for a, b in ((0, 1), (1, 4), (4, 8))]
    np.testing.assert_allclose(np.concatenate(parts), one, rtol=1e-12, atol=1e-12)


def test_sibling_permutation_and_nonancestor_perturbation(tiny):
    w, ref, prefix = tiny
    parent = np.array([-1, 0, 0, 0, 1, 2])
    toks = np.array([5, 6, 7, 8, 9, 10])
    kv, _ = _prefilled(w, prefix)
    base = oracle.tree_step(w, kv, toks, parent)
    # swap siblings 1 and 2 (and re-point child 4 -> 2's position, child 5 -> 1's)
    perm = [0, 2, 1, 3, 5, 4]  # new node k is old node perm[k]
    inv = {old: new for new, old in enumerate(perm)}
    parent2 = np.array([-1 if parent[o] == -1 else inv[parent[o]] for o in perm])
    kv, _ = _prefilled(w, prefix)
    out2 = oracle.tree_step(w, kv, toks[perm], parent2)
    np.testing.assert_allclose(out2, base[perm], rtol=1e-12, atol=1e-12)
    # changing node 3's token (not an ancestor of 1, 2, 4, 5) leaves those rows unchanged
    t3 = toks.copy()
    t3[3] = 999
    kv, _ = _prefilled(w, prefix)
    out3 = oracle.tree_step(w, kv, t3, parent)
    for i in (0, 1, 2, 4, 5):
        np.testing.assert_allclose(out3[i], base[i], rtol=1e-12, atol=1e-12)
    assert np.max(np.abs(out3[3] - base[3])) > 1e-3


def test_skip_mask_all_off_is_closed_form(tiny):
    w, ref, prefix = tiny
    kv = oracle.KVCache(SH.n_layers, SH.n_heads, SH.head_dim, 128)
    toks = np.array([1, 2, 3])
    out = oracle.tree_step(w, kv, toks, np.array([-1, 0, 1]), skip_mask=np.zeros(SH.n_layers, np.uint8))
    e = torch.from_numpy(synth.bf16_to_f32(synth.weight_bf16(SEED, SH, "embed")).astype(np.float64))[toks]
    lm = torch.from_numpy(synth.bf16_to_f32(synth.weight_bf16(SEED, SH, "lm_head")).astype(np.float64))
    want = F.linear(F.rms_norm(e, (SH.d_model,), None, SH.rms_eps), lm).numpy()
    np.testing.assert_allclose(out, want, rtol=1e-12, atol=1e-12)
    assert not any(v.any() for v in kv.valid)  # no layer wrote K/V


def test_skip_one_layer_equals_model_without_it(tiny):
    w, ref, prefix = tiny
    mask = np.array([1, 0], dtype=np.uint8)
    kv, _ = _prefilled(w, prefix, mask=mask)
    toks = synth.tokens(9, 4, SH.vocab)
    parent = synth.chain(4)
    out = oracle.tree_step(w, kv, toks, parent, skip_mask=mask)
    want = ref.forward(np.concatenate([prefix, toks]), layers_on=mask)[-4:]
    assert np.max(np.abs(out - want) / np.ptp(want, axis=1, keepdims=True)) < 1e-10
    # all on == no mask
    kv1, _ = _prefilled(w, prefix)
    kv2, _ = _prefilled(w, prefix)
    np.testing.assert_array_equal(oracle.tree_step(w, kv1, toks, parent, skip_mask=np.ones(2, np.uint8)),
                                  oracle.tree_step(w, kv2, toks, parent))


@pytest.mark.parametrize("mode", [0, 1])
def test_layer_input_override_composes(tiny, mode):
    """x0 replaces the embedding as the first layer's input: the embedding rows themselves give the
    default result bit for bit, and layer 1 run alone from the residual layer 0 left (traced) gives
    the two-layer result (same caches), in bf16 and W8A8 mode."""
    w, ref, prefix = tiny
    toks, parent = synth.tokens(21, 6, SH.vocab), synth.tree(21, 6, 3)
    kv1, _ = _prefilled(w, prefix)
    kv2, _ = _prefilled(w, prefix)
    tr = {}
    full = oracle.tree_step(w, kv1, toks, parent, quant_mode=mode, trace=tr)
    same = oracle.tree_step(w, kv2, toks, parent, quant_mode=mode, x0=w.f64("embed")[toks])
    np.testing.assert_array_equal(full, same)
    kv3, _ = _prefilled(w, prefix)
    only1 = np.array([0, 1], dtype=np.uint8)
    tail = oracle.tree_step(w, kv3, toks, parent, skip_mask=only1, quant_mode=mode, x0=tr[0]["x"])
    np.testing.assert_array_equal(full, tail)
    np.testing.assert_array_equal(kv3.K[1], kv1.K[1])  # layer 1 wrote the same K/V
    assert "u" in tr[1] and tr[1]["u"].shape == (6, SH.ffn)


def _gains(name, layer):
    """Distinct seeded RMSNorm gains per (norm, layer)."""
    kind = {"attn_norm": 1, "ffn_norm": 2, "final_norm": 3}[name]
    return np.random.default_rng(100 * max(layer, 0) + kind).uniform(0.5, 1.5, SH.d_model)


def _weights_with(zero: tuple | None = None):
    """Tiny weights with the gains above, optionally with one matrix (name, layer) zeroed."""
    def get(name, layer):
        bits = synth.weight_bf16(SEED, SH, name, layer)
        return np.zeros_like(bits) if zero == (name, layer) else bits

    return oracle.Weights(SH, get, _gains, keep_layers=SH.n_layers)


@pytest.mark.parametrize("mask,blocks", [
    ([1, 1], [(True, True), (True, True)]),
    ([1 | 2, 1], [(False, True), (True, True)]),  # layer 0 without attention
    ([1, 1 | 4], [(True, True), (True, False)]),  # layer 1 without FFN
    ([1 | 4, 1 | 2], [(True, False), (False, True)]),
])
def test_gains_and_sub_blocks_match_causal_forward(tiny, mask, blocks):
    """Chain prefill with non-unit gains (each norm its own) and sub-block masks against the
    textbook causal forward given the same gains and sub-block switches: the RMSNorm of each block
    uses that block's gains and a skipped block is dropped from the residual stream."""
    _, _, prefix = tiny
    ref = CausalLM(SH, SEED, gains=_gains)
    kv = oracle.KVCache(SH.n_layers, SH.n_heads, SH.head_dim, 128)
    got = oracle.tree_step(_weights_with(), kv, prefix[:40], synth.chain(40), skip_mask=np.array(mask, np.uint8))
    want = ref.forward(prefix[:40], blocks=blocks)
    assert np.max(np.abs(got - want) / np.ptp(want, axis=1, keepdims=True)) < 1e-10


@pytest.mark.parametrize("layer", [0, 1])
@pytest.mark.parametrize("block", ["attn", "ffn"])
def test_skipped_sub_block_equals_zeroed_output_matrix(tiny, layer, block):
    """Skipping a layer's attention (FFN) block gives exactly the model whose output projection Wo
    (down projection Wd) of that layer is zero: the block adds nothing to the residual stream.  The
    gains differ per norm, so running the other block with the wrong norm would show.  A skipped
    attention block writes no K/V in that layer."""
    _, _, prefix = tiny
    flag, name = (oracle.SKIP_ATTN, "wo") if block == "attn" else (oracle.SKIP_FFN, "wd")
    mask = np.ones(SH.n_layers, np.uint8)
    mask[layer] |= flag
    w_skip, w_zero = _weights_with(), _weights_with((name, layer))
    kv_s, pre_s = _prefilled(w_skip, prefix, mask=mask)
    kv_z, pre_z = _prefilled(w_zero, prefix)
    np.testing.assert_array_equal(pre_s, pre_z)
    toks, parent = synth.tokens(21, 8, SH.vocab), synth.tree(21, 8, 4)
    got = oracle.tree_step(w_skip, kv_s, toks, parent, skip_mask=mask)
    want = oracle.tree_step(w_zero, kv_z, toks, parent)
    np.testing.assert_array_equal(got, want)
    P = len(prefix)
    for l in range(SH.n_layers):
        written = bool(kv_s.valid[l][P:P + 8].all())
        assert written == (l != layer or block == "ffn")
        assert not kv_s.valid[l][P:P + 8].any() or written
    # and the skipped block changes the result (the pin is not vacuous)
    kv_f, _ = _prefilled(w_skip, prefix)
    assert np.max(np.abs(oracle.tree_step(w_skip, kv_f, toks, parent) - got)) > 1e-3


def test_both_sub_blocks_skipped_is_the_layer_off(tiny):
    w, _, prefix = tiny
    toks, parent = synth.tokens(22, 6, SH.vocab), synth.tree(22, 6, 3)
    both = np.array([1 | oracle.SKIP_ATTN | oracle.SKIP_FFN, 1], np.uint8)
    off = np.array([0, 1], np.uint8)
    kv1, _ = _prefilled(w, prefix, mask=off)
    kv2, _ = _prefilled(w, prefix, mask=off)
    np.testing.assert_array_equal(oracle.tree_step(w, kv1, toks, parent, skip_mask=both),
                                  oracle.tree_step(w, kv2, toks, parent, skip_mask=off))
    assert oracle.layer_blocks(1) == (True, True) and oracle.layer_blocks(0) == (False, False)


def test_int8_mode_close_to_bf16_mode(tiny):
    """W8A8 draft logits stay within the quantisation error of the full-precision model."""
    w, ref, prefix = tiny
    toks, parent = synth.tokens(3, 8, SH.vocab), synth.tree(3, 8, 4)
    kv1, _ = _prefilled(w, prefix)
    kv2, _ = _prefilled(w, prefix)
    a = oracle.tree_step(w, kv1, toks, parent)
    b = oracle.tree_step(w, kv2, toks, parent, quant_mode=1)
    err = np.max(np.abs(a - b) / np.ptp(a, axis=1, keepdims=True))
    assert 1e-5 < err < 0.1, err


def test_w4a4_and_activation_sparsity_modes(tiny):
    """W4A4 (App. C, QSpec's bit width) and TEAL activation sparsity: sparsity 0 is the dense
    model exactly; one projection with a single kept input is that input times one weight column;
    W4A4 moves the logits more than W8A8 and less than the whole logit range."""
    w, ref, prefix = tiny
    toks, parent = synth.tokens(3, 8, SH.vocab), synth.tree(3, 8, 4)
    runs = {}
    for key, kw in {"bf16": {}, "s0": {"act_sparsity": 0.0}, "w8": {"quant_mode": 1}, "w4": {"quant_mode": 2},
                    "s50": {"act_sparsity": 0.5}, "w4s50": {"quant_mode": 2, "act_sparsity": 0.5}}.items():
        kv, _ = _prefilled(w, prefix)
        runs[key] = oracle.tree_step(w, kv, toks, parent, **kw)
    np.testing.assert_array_equal(runs["s0"], runs["bf16"])

    def err(a):
        return np.max(np.abs(a - runs["bf16"]) / np.ptp(runs["bf16"], axis=1, keepdims=True))

    assert err(runs["w8"]) < err(runs["w4"]) < 1.0
    assert err(runs["s50"]) > 1e-3 and err(runs["w4s50"]) > 1e-3
    x = np.zeros((1, SH.d_model))
    x[0, 5], x[0, 9] = -3.0, 0.25
    from oracle import casspec_oracle

    y = casspec_oracle._linear(x, w, "wo", 0, (0, 1.0 - 1.0 / SH.d_model))  # keep one input of d
    np.testing.assert_allclose(y[0], -3.0 * w.f64("wo", 0)[:, 5], rtol=0, atol=0)
    with pytest.raises(ValueError):
        oracle.tree_step(w, oracle.KVCache(SH.n_layers, SH.n_heads, SH.head_dim, 128), toks, parent, quant_mode=3)


def test_quantised_sparsity_selects_on_the_bf16_activation(tiny):
    """In a quantised draft the selection is taken on the bf16 activation the quantiser reads: two
    inputs of different fp64 magnitude that round to the same bf16 value tie, and the lower index is
    kept, where the bf16 draft keeps the larger fp64 one.  With one input kept, the W8A8 projection
    is that input's code (127) times the weight column's codes, scaled."""
    w, _, _ = tiny
    from oracle import casspec_oracle

    d = SH.d_model
    x = np.zeros((1, d))
    x[0, 5], x[0, 9] = 1.0 + 2.0 ** -12, 1.0 + 2.0 ** -11  # both round to 1.0 in bf16
    keep_one = 1.0 - 1.0 / d
    y16 = casspec_oracle._linear(x, w, "wo", 0, (0, keep_one))
    np.testing.assert_array_equal(y16[0], x[0, 9] * w.f64("wo", 0)[:, 9])
    y8 = casspec_oracle._linear(x, w, "wo", 0, (1, keep_one))
    qw, sw = w.intq("wo", 0, 127)
    kept = np.zeros((1, d))
    kept[0, 5] = 1.0  # the selection under test: index 5, as bf16 (the quantiser's own scale rule)
    qx, sx = oracle.quantize_rows_f32(kept, 127)
    assert qx[0, 5] == 127 and np.count_nonzero(qx) == 1
    want = (127.0 * qw[:, 5].astype(np.float64)) * float(sx[0]) * sw
    np.testing.assert_allclose(y8[0], want, rtol=1e-15, atol=0)
    assert not np.allclose(qw[:, 5], qw[:, 9])


def test_attn_bf16_rounds_only_the_attention_operands(tiny):
    """attn_bf16 stores bf16 K/V and uses bf16 q: the cache entries it writes are bf16 values,
    everything else is the fp64 model, and the logits move by about the bf16 rounding."""
    w, ref, prefix = tiny
    toks, parent = synth.tokens(5, 8, SH.vocab), synth.tree(5, 8, 4)
    kv1, _ = _prefilled(w, prefix)
    kv2, _ = _prefilled(w, prefix)
    tr1, tr2 = {}, {}
    a = oracle.tree_step(w, kv1, toks, parent, trace=tr1)
    b = oracle.tree_step(w, kv2, toks, parent, trace=tr2, attn_bf16=True)
    P = len(prefix)
    for l in range(SH.n_layers):
        new_k = kv2.K[l][:, P:P + 8]
        assert np.array_equal(new_k, oracle.round_bf16(new_k))
        assert np.array_equal(tr2[l]["q"], oracle.round_bf16(tr2[l]["q"]))
        assert not np.array_equal(kv1.K[l][:, P:P + 8], oracle.round_bf16(kv1.K[l][:, P:P + 8]))
    # layer 0's normalised input does not depend on attention: identical
    assert np.array_equal(tr1[0]["xn"], tr2[0]["xn"])
    err = np.max(np.abs(a - b) / np.ptp(a, axis=1, keepdims=True))
    assert 1e-6 < err < 1e-2, err


# ------------------------------------------------------------------------------------------------
# acceptance vs brute force; losslessness; compaction
# ------------------------------------------------------------------------------------------------
def _brute_accept(argmax, tokens, parent):
    n = len(parent)
    kids = {i: [c for c in range(n) if parent[c] == i] for i in range(n)}
    leaves = [i for i in range(n) if not kids[i]]
    best = None
    for leaf in leaves:
        path = _root_path(parent, leaf)
        m = 0
        while m + 1 < len(path) and tokens[path[m + 1]] == argmax[path[m]]:
            m += 1
        cand = path[: m + 1]
        key = (len(cand), -cand[-1])
        if best is None or key > best[0]:
            best = (key, cand)
    return best[1], int(argmax[best[1][-1]])


def test_accept_greedy_bruteforce_random_and_planted():
    rng = np.random.default_rng(6)
    for trial in range(400):
        n = int(rng.integers(1, 9))
        parent = synth.tree(trial, n, int(rng.integers(1, 5)))
        vocab = 3 if trial % 2 else 50
        argmax = rng.integers(0, vocab, n)
        toks = rng.integers(0, vocab, n)
        if trial % 3 == 0 and n > 1:  # plant a path
            leaf = int(rng.integers(0, n))
            path = _root_path(parent, leaf)
            for a, b in zip(path, path[1:]):
                toks[b] = argmax[a]
        assert oracle.accept_greedy(argmax, toks, parent) == _brute_accept(argmax, toks, parent)


def test_accept_rejects_multiple_roots():
    with pytest.raises(ValueError):
        oracle.accept_greedy(np.zeros(3), np.zeros(3), np.array([-1, -1, 0]))


def test_greedy_speculative_equals_greedy_autoregressive(tiny):
    """Sec. 5.1: speculative decoding with greedy tree verification is lossless."""
    w, ref, prefix = tiny
    steps = 64
    # greedy AR with the textbook model
    seq = list(prefix)
    for _ in range(steps):
        seq.append(int(np.argmax(ref.forward(np.array(seq))[-1])))
    truth = seq[len(prefix):]
    # speculative: prefill, then rounds of (tree verify, accept, compact)
    kv, logits = _prefilled(w, prefix, cap=len(prefix) + steps + 16)
    out = [int(oracle.argmax_lowest(logits[-1:])[0])]
    rng = np.random.default_rng(7)
    rnd = 0
    while len(out) < steps:
        parent = synth.tree(100 + rnd, 8, 4)
        toks = rng.integers(0, SH.vocab, 8)
        toks[0] = out[-1]
        # plant the true continuation along one branch so deep acceptance happens
        leaf = int(rng.integers(0, 8))
        path = _root_path(parent, leaf)
        k = len(out)
        for depth, node in enumerate(path[1:], start=1):
            if k - 1 + depth < len(truth) and rng.random() < 0.8:
                toks[node] = truth[k - 1 + depth]
        lg = oracle.tree_step(w, kv, toks, parent)
        acc, bonus = oracle.accept_greedy(oracle.argmax_lowest(lg), toks, parent)
        oracle.kv_compact(kv, acc)
        out.extend(int(toks[a]) for a in acc[1:])
        out.append(bonus)
        rnd += 1
    assert out[:steps] == truth
    assert rnd < steps  # some rounds accepted more than the root


def test_compaction_equals_causal_cache(tiny):
    w, ref, prefix = tiny
    parent = np.array([-1, 0, 0, 2, 2, 3, 1, 5])
    toks = synth.tokens(11, 8, SH.vocab)
    for a, b in ((0, 2), (2, 3), (3, 5)):  # plant path 0-2-3-5, one depth level per pass
        kv, _ = _prefilled(w, prefix)
        toks[b] = oracle.argmax_lowest(oracle.tree_step(w, kv, toks, parent))[a]
    kv, _ = _prefilled(w, prefix)
    lg = oracle.tree_step(w, kv, toks, parent)
    acc, bonus = oracle.accept_greedy(oracle.argmax_lowest(lg), toks, parent)
    assert acc == [0, 2, 3, 5]
    oracle.kv_compact(kv, acc)
    assert kv.P == len(prefix) + 4 and kv.T == 0
    _, cache = ref.forward(np.concatenate([prefix, toks[acc]]), return_kv=True)
    for l in range(SH.n_layers):
        k_ref, v_ref = (t.numpy() for t in cache[l])
        np.testing.assert_allclose(kv.K[l][:, :kv.P], k_ref, rtol=1e-9, atol=1e-10)
        np.testing.assert_allclose(kv.V[l][:, :kv.P], v_ref, rtol=1e-9, atol=1e-10)


# ------------------------------------------------------------------------------------------------
# top-K candidates (tree expansion, Sec. 4.2)
# ------------------------------------------------------------------------------------------------
def test_topk_softmax_against_brute_force_and_torch():
    rng = np.random.default_rng(3)
    x = rng.normal(0, 3, (5, 40))
    x[2, 7] = x[2, 3] = x[2].max() + 1.0  # an exact tie at the top: the lower id first
    idx, prob = oracle.topk_softmax(x, 4)
    for r in range(5):
        order = sorted(range(40), key=lambda j: (-x[r, j], j))[:4]
        assert list(idx[r]) == order
    assert list(idx[2][:2]) == [3, 7]
    ref = torch.softmax(torch.tensor(x), dim=1).numpy()
    assert np.allclose(prob, np.take_along_axis(ref, idx, axis=1), rtol=1e-12, atol=0)
    # k larger than the row: every token, in order
    idx2, prob2 = oracle.topk_softmax(x[:, :3], 8)
    assert idx2.shape == (5, 3) and np.allclose(prob2.sum(axis=1), 1.0)

