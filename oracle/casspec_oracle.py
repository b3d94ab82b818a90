"""CPU fp64 oracle of the CAS-Spec token-tree decode step.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU
baseline / reference arm may import or run this module.  The CUDA library never calls it and it
shares no code with it; its only shared dependency is the seeded input module ``synth`` (which
holds no step of the method).

What it computes (CAS-Spec, arXiv 2510.26843):
  * one forward pass of a Llama-style decoder over the n nodes of a token tree against a prefix KV
    cache -- the tree-attention draft/verify pass of Sec. 4.2 ("tree attention allows ... parallel
    verification of different branches"; "tree-based parallel draft generation"), run by the target
    model and by its DSIA drafts (Sec. 4.1, Def. 4.1);
  * DSIA layer sparsity (Sec. 4.1, "skipping a subset of transformer layers"): a switched-off
    layer is the identity on the residual stream and writes no K/V; the same at the granularity of
    a layer's attention or FFN sub-block (Sec. 4.1 names both granularities): a skipped attention
    block adds nothing to the residual stream and writes no K/V, a skipped FFN block adds nothing;
  * DSIA activation quantisation (Sec. 4.1 and App. C, QSpec-style W?A? drafts): W8A8 and W4A4,
    per output channel symmetric weights and per-token dynamic symmetric activations on the inputs
    of Wqkv, Wo, Wgate/Wup and Wdown; attention, K/V and the LM head stay in floating point;
  * DSIA activation sparsity (Sec. 4.1 and App. C, TEAL): the smallest-magnitude share of each
    projection input is zeroed per token;
  * lossless greedy verification (Sec. 5.1: output identical to autoregressive decoding): the
    longest root-to-leaf path whose tokens equal the target's argmax, plus the bonus token;
  * compaction of the accepted path's K/V into the committed cache.

Readings where the paper is silent (each also listed in the design notes):
  * architecture: pre-norm RMSNorm, rotary position embedding (rotate-half pairs (j, j + h/2),
    angle pos * base^(-2j/h)), SwiGLU FFN, multi-head attention, untied LM head, no biases;
  * tree positions: a node at depth t (root depth 0, Alg. 1: the root is the last bonus token) sits
    at position P + t, P = committed prefix length;
  * tree mask: every node sees the whole prefix and exactly its ancestors and itself;
  * argmax ties go to the lowest token id; among children carrying the same token the lowest node
    index is taken; the root (node 0) is always accepted, so L >= 1;
  * quantisation: q = rint(x * (127 / amax)) with ties to even, clamped to [-127, 127], scale
    amax / 127; amax = 0 gives q = 0 and scale 0.  Weights are quantised with this rule evaluated
    in fp32 (IEEE round-to-nearest division and multiply, no fused multiply-add) from the bf16
    weights; activations are quantised with the same fp32 rule from their bf16 rounding (the
    precision in which the draft stores them), so both sides take the integer decisions alike.

Everything here is fp64 unless stated; bf16 inputs are widened exactly.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Callable

import numpy as np

import synth

# ----------------------------------------------------------------------------------------------
# elementwise pieces
# ----------------------------------------------------------------------------------------------


def rmsnorm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * g."""
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * np.asarray(g, dtype=np.float64)


def rope(x: np.ndarray, pos: np.ndarray, base: float) -> np.ndarray:
    """Rotate-half rotary embedding of x[..., n, h] at integer positions pos[n].

    For j < h/2 the pair (x_j, x_{j+h/2}) is rotated by angle pos * base^(-2j/h).
    """
    x = np.asarray(x, dtype=np.float64)
    h = x.shape[-1]
    half = h // 2
    inv_freq = base ** (-2.0 * np.arange(half, dtype=np.float64) / h)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv_freq[None, :]  # [n, half]
    c, s = np.cos(ang), np.sin(ang)
    a, b = x[..., :half], x[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


# ----------------------------------------------------------------------------------------------
# int8 quantisation (App. C activation-quantisation DSIA; W8A8 reading)
# ----------------------------------------------------------------------------------------------


def quantize_rows_f32(x: np.ndarray, qmax: int = 127) -> tuple[np.ndarray, np.ndarray]:
    """Symmetric per-row quantisation evaluated in fp32 (qmax 127: int8; 7: int4).

    x: fp32 rows [r, c] (bf16 inputs widened exactly).  Returns (q int8 [r, c], scale fp32 [r]).
    inv = qmax / amax (fp32 division), t = x * inv (fp32 multiply), q = rint(t) (ties to even),
    clamp to +-qmax; scale = amax / qmax (fp32 division).  amax = 0 -> q = 0, scale = 0.
    """
    x = np.asarray(x, dtype=np.float32)
    qm = np.float32(qmax)
    amax = np.max(np.abs(x), axis=-1)
    safe = np.where(amax > 0, amax, np.float32(1.0)).astype(np.float32)
    inv = (qm / safe).astype(np.float32)
    t = (x * inv[:, None]).astype(np.float32)
    q = np.clip(np.rint(t), -qmax, qmax).astype(np.int8)
    q[amax == 0] = 0
    scale = np.where(amax > 0, (amax / qm).astype(np.float32), np.float32(0.0)).astype(np.float32)
    return q, scale


def quantize_rows_f64(x: np.ndarray, qmax: int = 127) -> tuple[np.ndarray, np.ndarray]:
    """The same rule evaluated in fp64 (end-to-end oracle activations)."""
    x = np.asarray(x, dtype=np.float64)
    amax = np.max(np.abs(x), axis=-1)
    safe = np.where(amax > 0, amax, 1.0)
    q = np.clip(np.rint(x * (qmax / safe)[:, None]), -qmax, qmax).astype(np.int8)
    q[amax == 0] = 0
    scale = np.where(amax > 0, amax / qmax, 0.0)
    return q, scale


def sparsify_rows(x: np.ndarray, s: float) -> np.ndarray:
    """Activation sparsity by magnitude (the TEAL DSIA of App. C): per row of length K, the
    floor(s * K) entries of smallest magnitude become 0 and the others are kept; among equal
    magnitudes the lower index is kept."""
    x = np.array(x, dtype=np.float64, copy=True)
    K = x.shape[-1]
    z = int(math.floor(s * K + 1e-9))
    if z <= 0:
        return x
    for r in range(x.shape[0]):
        order = sorted(range(K), key=lambda c: (-abs(x[r, c]), c))
        x[r, order[K - z:]] = 0.0
    return x


def linear_w8a8(qx: np.ndarray, sx: np.ndarray, qw: np.ndarray, sw: np.ndarray) -> np.ndarray:
    """y[t, o] = (sum_k qx[t, k] * qw[o, k]) * sx[t] * sw[o]; the integer sum is exact.

    The codes are integers of magnitude <= 127, so every partial sum of the dot product is an integer
    below K * 127^2 < 2^53: the fp64 matrix product returns the exact integer sum in any summation
    order (the same value as an int64 sum; pinned against an int64 brute force)."""
    K = qx.shape[-1]
    assert K * 127 * 127 < 2 ** 53
    acc = qx.astype(np.float64) @ qw.astype(np.float64).T
    return acc.astype(np.float64) * np.asarray(sx, dtype=np.float64)[:, None] * np.asarray(sw, dtype=np.float64)[None, :]


# ----------------------------------------------------------------------------------------------
# weights
# ----------------------------------------------------------------------------------------------


class Weights:
    """Weight provider: bf16 bit arrays from `get(name, layer)`; widened to fp64 on use.

    Names: embed [V, d], wqkv [3d, d] (Wq; Wk; Wv stacked by rows), wo [d, d], wg [F, d], wu [F, d],
    wd [d, F], lm_head [V, d] -- all [out, in].  Gains come from `gain(name, layer)`.
    Recently used layers are kept (`keep_layers`) so tiny models are generated once.
    """

    def __init__(self, shape: synth.ModelShape, get: Callable[[str, int], np.ndarray],
                 gain: Callable[[str, int], np.ndarray] | None = None, keep_layers: int = 2):
        self.shape = shape
        self._get = get
        self._gain = gain or (lambda name, layer: np.ones(shape.d_model, dtype=np.float32))
        self._keep = keep_layers
        self._cache: dict = {}
        self._order: list = []

    @staticmethod
    def from_seed(seed: int, shape: synth.ModelShape, keep_layers: int = 2) -> "Weights":
        return Weights(shape, lambda name, layer: synth.weight_bf16(seed, shape, name, layer),
                       keep_layers=keep_layers)

    def _cached(self, key, make):
        """Memoise per (kind, layer, name); keep only the `keep_layers` most recent layers."""
        if key in self._cache:
            return self._cache[key]
        layer = key[1]
        if layer >= 0 and layer not in self._order:
            self._order.append(layer)
            while len(self._order) > self._keep:
                old = self._order.pop(0)
                for k in [k for k in self._cache if k[1] == old]:
                    del self._cache[k]
        v = make()
        self._cache[key] = v
        return v

    def bits(self, name: str, layer: int = -1) -> np.ndarray:
        return self._cached(("bits", layer, name), lambda: self._get(name, max(layer, 0)))

    def f64(self, name: str, layer: int = -1) -> np.ndarray:
        return self._cached(("f64", layer, name),
                            lambda: synth.bf16_to_f32(self.bits(name, layer)).astype(np.float64))

    def int8(self, name: str, layer: int) -> tuple[np.ndarray, np.ndarray]:
        """Per-output-channel int8 weights and fp32 scales (quantize_rows_f32 of the bf16 rows)."""
        return self.intq(name, layer, 127)

    def intq(self, name: str, layer: int, qmax: int) -> tuple[np.ndarray, np.ndarray]:
        """Per-output-channel weights with codes in [-qmax, qmax] (127: int8, 7: int4) and scales."""
        return self._cached((f"i{qmax}", layer, name),
                            lambda: quantize_rows_f32(synth.bf16_to_f32(self.bits(name, layer)), qmax))

    def gain(self, name: str, layer: int = -1) -> np.ndarray:
        return np.asarray(self._gain(name, layer), dtype=np.float64)


# ----------------------------------------------------------------------------------------------
# KV cache and tree state
# ----------------------------------------------------------------------------------------------


@dataclass
class KVCache:
    """Committed prefix [0, P) plus tree slots [P, P + T); K/V per layer as fp64 [H, cap, h].

    valid[l][s] records which slots hold K/V written for layer l (prefix stand-ins count as valid).
    depth[j], anc[j] describe tree slot j (anc = set of tree slots on the root path, incl. j).
    """

    n_layers: int
    n_heads: int
    head_dim: int
    capacity: int
    P: int = 0
    T: int = 0
    K: list = field(default_factory=list)
    V: list = field(default_factory=list)
    valid: list = field(default_factory=list)
    depth: list = field(default_factory=list)
    anc: list = field(default_factory=list)

    def __post_init__(self):
        shp = (self.n_heads, self.capacity, self.head_dim)
        self.K = [np.zeros(shp) for _ in range(self.n_layers)]
        self.V = [np.zeros(shp) for _ in range(self.n_layers)]
        self.valid = [np.zeros(self.capacity, dtype=bool) for _ in range(self.n_layers)]

    def load_prefix(self, layer: int, k: np.ndarray, v: np.ndarray):
        """Install a stand-in prefix ([H, P, h] each) for `layer`; sets P."""
        p = k.shape[1]
        self.K[layer][:, :p] = k
        self.V[layer][:, :p] = v
        self.valid[layer][:p] = True
        self.P = p

    def reset_tree(self):
        self.T = 0
        self.depth, self.anc = [], []
        for l in range(self.n_layers):
            self.valid[l][self.P:] = False


def tree_topology(parent: np.ndarray, T: int, depth_prev: list, anc_prev: list) -> tuple[list, list]:
    """Depth and ancestor set of new nodes i (tree slot T + i) given parent_idx in tree-slot space.

    parent -1 makes a node a root child of the committed prefix (depth 0); otherwise the parent must
    be an existing slot < T + i.  Raises ValueError on an invalid parent.
    """
    depth, anc = list(depth_prev), list(anc_prev)
    for i, p in enumerate(int(v) for v in parent):
        j = T + i
        if p == -1:
            depth.append(0)
            anc.append(frozenset([j]))
        elif 0 <= p < j:
            depth.append(depth[p] + 1)
            anc.append(anc[p] | {j})
        else:
            raise ValueError(f"parent_idx[{i}] = {p} not in [-1, {j})")
    return depth[T:], anc[T:]


# ----------------------------------------------------------------------------------------------
# the tree step
# ----------------------------------------------------------------------------------------------


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bf16 value (ties to even) via fp32; returned as fp32."""
    u = np.ascontiguousarray(np.asarray(x, dtype=np.float64).astype(np.float32)).view(np.uint32)
    u = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) & np.uint32(0xFFFF0000)
    return u.view(np.float32)


QMAX = {1: 127, 2: 7}  # quant_mode -> largest code: W8A8, W4A4


def _linear(x: np.ndarray, w: Weights, name: str, layer: int, lin: tuple) -> np.ndarray:
    """One projection of a draft: lin = (quant_mode, activation sparsity).  The sparsity rule
    applies to the projection's input first (in a quantised mode to its bf16 value, the value the
    quantiser reads); a quantised mode then quantises that input."""
    mode, sparsity = lin
    if sparsity > 0.0:
        # a quantised draft stores its activation in bf16 and quantises that value (reading of App. C
        # above), so its magnitude selection is taken on the same bf16 value; a bf16 draft selects on
        # the activation itself
        x = sparsify_rows(round_bf16(x) if mode in QMAX else x, sparsity)
    if mode in QMAX:
        # The quantiser's integer decisions are taken on the activation as the draft stores it
        # (bf16) with the fp32 rule, i.e. in the kernel's precision.
        qx, sx = quantize_rows_f32(round_bf16(x), QMAX[mode])
        qw, sw = w.intq(name, layer, QMAX[mode])
        return linear_w8a8(qx, sx, qw, sw)
    return x @ w.f64(name, layer).T


def tree_attention(q: np.ndarray, kv: KVCache, layer: int, slots: list, anc: list) -> np.ndarray:
    """Masked softmax attention of new nodes.

    q: [n, H, h] (already rotated).  Node i attends to prefix slots [0, P) and to tree slots
    P + j for j in anc[i].  Returns o [n, H, h].
    """
    n, H, h = q.shape
    P = kv.P
    cap = len(kv.valid[layer])
    visible = np.zeros((n, cap), dtype=bool)
    visible[:, :P] = True
    for i in range(n):
        for j in anc[i]:
            visible[i, P + j] = True
    assert np.all(kv.valid[layer][visible.any(axis=0)]), "attended slot has no K/V in this layer"
    out = np.empty((n, H, h))
    cols = np.nonzero(visible.any(axis=0))[0]
    for hd in range(H):
        keys = kv.K[layer][hd, cols]  # [c, h]
        vals = kv.V[layer][hd, cols]
        s = q[:, hd, :] @ keys.T / math.sqrt(h)  # [n, c]
        s = np.where(visible[:, cols], s, -np.inf)
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p /= p.sum(axis=1, keepdims=True)
        out[:, hd, :] = p @ vals
    return out


SKIP_ATTN = 0x2  # skip-mask flag: the layer's attention block is skipped
SKIP_FFN = 0x4  # skip-mask flag: the layer's FFN block is skipped


def layer_blocks(code: int) -> tuple[bool, bool]:
    """(attention on, FFN on) for one skip-mask byte: 0 switches the whole layer off; otherwise
    each sub-block runs unless its flag is set."""
    code = int(code)
    if code == 0:
        return False, False
    return not code & SKIP_ATTN, not code & SKIP_FFN


def tree_step(w: Weights, kv: KVCache, tokens: np.ndarray, parent: np.ndarray,
              skip_mask: np.ndarray | None = None, quant_mode: int = 0,
              trace: dict | None = None, attn_bf16: bool = False, act_sparsity: float = 0.0,
              x0: np.ndarray | None = None) -> np.ndarray:
    """One draft/verify pass over n new tree nodes; returns logits [n, V] (fp64).

    The nodes occupy tree slots T .. T+n-1 (cache slots P+T .. P+T+n-1); each active layer writes
    their K/V there.  skip_mask[l] == 0 switches layer l off (Sec. 4.1 layer sparsity); a non-zero
    byte keeps it on except for the sub-blocks whose flag it carries: SKIP_ATTN (the attention
    block: no residual update, no K/V written) and SKIP_FFN (the FFN block).
    quant_mode 1 runs the W8A8 draft, 2 the W4A4 draft (App. C: QSpec's bit width; codes +-7 with the
    same rule); act_sparsity s > 0 zeroes the floor(s K) smallest-magnitude inputs of every projection
    (App. C: TEAL activation sparsity), before any quantisation.  `trace`, if given, receives
    per-layer intermediates.
    attn_bf16 rounds q and the K/V written to the cache to bf16 (a bf16 cache and bf16 attention
    operands).  It is a perturbation of the size of bf16 storage, used by tests to measure how far
    the method's own output moves under it; the reference result keeps it off.
    x0 [n, d], if given, is the residual stream entering the first layer in place of the tokens'
    embedding rows (a test feeds one layer the input another implementation gave it).
    """
    sh = w.shape
    tokens = np.asarray(tokens, dtype=np.int64)
    parent = np.asarray(parent, dtype=np.int64)
    n = len(tokens)
    if kv.P + kv.T + n > kv.capacity:
        raise ValueError("KV capacity exceeded")
    depth, anc = tree_topology(parent, kv.T, kv.depth, kv.anc)
    pos = np.array([kv.P + t for t in depth], dtype=np.int64)
    slots = [kv.P + kv.T + i for i in range(n)]
    all_anc = kv.anc + anc
    mask = np.ones(sh.n_layers, dtype=np.uint8) if skip_mask is None else np.asarray(skip_mask)
    if quant_mode not in (0, 1, 2) or not 0.0 <= act_sparsity < 1.0:
        raise ValueError("quant_mode must be 0, 1 or 2 and act_sparsity in [0, 1)")
    lin = (quant_mode, float(act_sparsity))

    x = w.f64("embed")[tokens] if x0 is None else np.array(x0, dtype=np.float64).reshape(n, sh.d_model)  # [n, d]
    for l in range(sh.n_layers):
        attn_on, ffn_on = layer_blocks(mask[l])
        if attn_on:
            x = _attention_block(x, w, kv, l, lin, pos, slots, all_anc, n, attn_bf16, trace)
        if ffn_on:
            xn2 = rmsnorm(x, w.gain("ffn_norm", l), sh.rms_eps)
            if trace is not None:
                trace.setdefault(l, {})["xn2"] = xn2
            g = _linear(xn2, w, "wg", l, lin)
            u = _linear(xn2, w, "wu", l, lin)
            hgu = silu(g) * u
            if trace is not None:
                trace.setdefault(l, {})["u"] = hgu
            x = x + _linear(hgu, w, "wd", l, lin)
        if trace is not None and (attn_on or ffn_on):
            trace.setdefault(l, {})["x"] = x.copy()
    xf = rmsnorm(x, w.gain("final_norm"), sh.rms_eps)
    logits = xf @ w.f64("lm_head").T
    kv.depth = kv.depth + depth
    kv.anc = kv.anc + anc
    kv.T += n
    return logits


def _attention_block(x, w, kv, l, lin, pos, slots, all_anc, n, attn_bf16, trace):
    """x + Wo . TreeAttention(RoPE(Wq xn), RoPE(Wk xn), Wv xn) with xn = RMSNorm(x); writes the
    nodes' K/V of layer l."""
    sh = w.shape
    d, H, h = sh.d_model, sh.n_heads, sh.head_dim
    xn = rmsnorm(x, w.gain("attn_norm", l), sh.rms_eps)
    qkv = _linear(xn, w, "wqkv", l, lin)
    q = rope(qkv[:, :d].reshape(n, H, h).transpose(1, 0, 2), pos, sh.rope_base).transpose(1, 0, 2)
    k = rope(qkv[:, d:2 * d].reshape(n, H, h).transpose(1, 0, 2), pos, sh.rope_base).transpose(1, 0, 2)
    v = qkv[:, 2 * d:].reshape(n, H, h)
    if attn_bf16:
        q, k, v = round_bf16(q), round_bf16(k), round_bf16(v)
    for i, s in enumerate(slots):
        kv.K[l][:, s] = k[i]
        kv.V[l][:, s] = v[i]
        kv.valid[l][s] = True
    o = tree_attention(q, kv, l, slots, [all_anc[kv.T + i] for i in range(n)]).reshape(n, d)
    if trace is not None:
        trace.setdefault(l, {}).update({"xn": xn, "q": q, "k": k, "v": v, "o": o})
    return x + _linear(o, w, "wo", l, lin)


# ----------------------------------------------------------------------------------------------
# greedy acceptance and compaction
# ----------------------------------------------------------------------------------------------


def argmax_lowest(logits: np.ndarray) -> np.ndarray:
    """Row argmax with ties to the lowest index."""
    return np.argmax(np.asarray(logits), axis=-1).astype(np.int64)


def top2_margin(logits: np.ndarray) -> np.ndarray:
    s = np.sort(np.asarray(logits, dtype=np.float64), axis=-1)
    return s[:, -1] - s[:, -2]


def accept_greedy(argmax: np.ndarray, tokens: np.ndarray, parent: np.ndarray) -> tuple[list, int]:
    """Longest accepted root-to-node path (node indices, root first) and the bonus token.

    Node 0 is the root (the last committed bonus token, Alg. 1; always accepted).  A node matches
    when its parent matches and its token equals the parent's argmax (greedy verification: the
    target would have emitted exactly that token there, Sec. 5.1 losslessness).  The accepted node
    is the deepest matching node (lowest index among equally deep ones); the path is its root path
    and the bonus token is the target's argmax at that node.
    """
    parent = [int(p) for p in parent]
    n = len(parent)
    if n == 0 or parent[0] != -1 or any(not (0 <= p < c) for c, p in enumerate(parent) if c > 0):
        raise ValueError("node 0 must be the only root and parent[c] < c")
    depth = [0] * n
    match = [True] + [False] * (n - 1)
    for c in range(1, n):
        p = parent[c]
        depth[c] = depth[p] + 1
        match[c] = match[p] and int(tokens[c]) == int(argmax[p])
    best = max((c for c in range(n) if match[c]), key=lambda c: (depth[c], -c))
    path = [best]
    while path[-1] != 0:
        path.append(parent[path[-1]])
    path.reverse()
    return path, int(argmax[best])


def kv_compact(kv: KVCache, path: list) -> None:
    """Move the accepted tree slots to committed slots P .. P+L-1 in every layer; P += L; T = 0."""
    P = kv.P
    for l in range(kv.n_layers):
        src_k = [kv.K[l][:, P + j].copy() for j in path]
        src_v = [kv.V[l][:, P + j].copy() for j in path]
        ok = [bool(kv.valid[l][P + j]) for j in path]
        for k, j in enumerate(path):
            kv.K[l][:, P + k] = src_k[k]
            kv.V[l][:, P + k] = src_v[k]
            kv.valid[l][P + k] = ok[k]
    kv.P = P + len(path)
    kv.reset_tree()


def topk_softmax(logits: np.ndarray, k: int) -> tuple[np.ndarray, np.ndarray]:
    """K-best candidates per row for tree expansion (Sec. 4.2, Algorithm 1: top-K tokens of each drafted
    position; their normalised probabilities rank siblings): the k largest logits of each row (ties to
    the lower token id), and their softmax probabilities over the whole row, in fp64."""
    x = np.asarray(logits, dtype=np.float64)
    k = min(k, x.shape[1])
    idx = np.argsort(-x, axis=1, kind="stable")[:, :k]
    m = x.max(axis=1, keepdims=True)
    z = np.exp(x - m).sum(axis=1, keepdims=True)
    prob = np.exp(np.take_along_axis(x, idx, axis=1) - m) / z
    return idx.astype(np.int64), prob
