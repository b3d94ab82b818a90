"""Seeded synthetic inputs for the CAS-Spec tree step (weights, prefix K/V, token trees, skip masks).

This module is the only code shared by the CUDA path's callers (tests, bench) and the CPU oracle.
It holds input generation only: no step of the decoder, the tree mask, quantisation or acceptance.

Generator: SplitMix64 (Vigna 2015) used counter-style.  A stream is identified by a 64-bit key
derived from (seed, stream id); element i of the stream is ``mix(key + (i+1) * GAMMA)``.  Bulk
normal fills run in ``fill.c`` (compiled on first use with the system C compiler); the same
per-element definition is restated in ``normal_bf16_scalar`` for the pin tests.

Workload recipe (the shapes follow the paper's Llama-2-7B / 13B / Vicuna evaluation, Sec. 5.1):
  * weights N(0, 0.02) as bf16 (Irwin-Hall(4) approximation of a normal deviate);
  * RMSNorm gains 1.0;
  * prefix K/V N(0, 1) bf16 stand-ins for a real prompt's cache;
  * token ids uniform over the vocabulary;
  * trees: node 0 is the root (parent -1); node i > 0 draws its parent uniformly from the earlier
    nodes whose depth is below ``max_depth`` and whose child count is below ``max_branch``;
  * skip masks: exactly floor(f * L) layers off, chosen uniformly without replacement; masks of
    one cascade share one permutation, so a sparser draft's active layers are a subset of a denser one's.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
import threading
from dataclasses import dataclass

import numpy as np

GAMMA = 0x9E3779B97F4A7C15
MASK64 = (1 << 64) - 1

# stream kinds (high bits of a stream id)
K_EMBED, K_WQKV, K_WO, K_WG, K_WU, K_WD, K_LM_HEAD = 1, 2, 3, 4, 5, 6, 7
K_PREFIX_K, K_PREFIX_V, K_TOKENS, K_TREE, K_MASK, K_PREFIX_TOKENS = 8, 9, 10, 11, 12, 13

WEIGHT_STD = 0.02


def mix64(z: int) -> int:
    """SplitMix64 output function (finaliser)."""
    z &= MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
    return z ^ (z >> 31)


def stream_key(seed: int, kind: int, layer: int = 0, sub: int = 0) -> int:
    """Key of stream (kind, layer, sub) under `seed`."""
    sid = (kind << 40) | (layer << 20) | sub
    return mix64(mix64((seed + GAMMA) & MASK64) ^ ((sid * 0xD1B54A32D192ED03) & MASK64))


def u64(key: int, i: int) -> int:
    """Element i of stream `key` (uniform 64-bit)."""
    return mix64((key + (i + 1) * GAMMA) & MASK64)


class Counter:
    """Sequential reader over one stream (used for the small discrete draws)."""

    def __init__(self, key: int):
        self.key, self.i = key, 0

    def next(self) -> int:
        v = u64(self.key, self.i)
        self.i += 1
        return v

    def below(self, m: int) -> int:
        """Uniform integer in [0, m) by multiply-shift on the high 32 bits."""
        return ((self.next() >> 32) * m) >> 32


# ----------------------------------------------------------------------------------------------
# normal deviates as bf16
# ----------------------------------------------------------------------------------------------
_IH_SIGMA = math.sqrt(((1 << 32) - 1) / 3.0)  # std of a sum of four uniform 16-bit integers


def normal_scale(std: float) -> np.float32:
    return np.float32(std / _IH_SIGMA)


def bf16_bits_rne(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit pattern, round to nearest even (finite inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    return ((u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)).astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """bf16 bit pattern -> exact fp32 value."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_bf16_scalar(key: int, i: int, std: float) -> int:
    """Element i of a normal stream as a bf16 bit pattern (pure-Python restatement of fill.c)."""
    z = u64(key, i)
    s = (z & 0xFFFF) + ((z >> 16) & 0xFFFF) + ((z >> 32) & 0xFFFF) + (z >> 48)
    f = np.float32(s - 131070) * normal_scale(std)
    return int(bf16_bits_rne(np.array([f], dtype=np.float32))[0])


_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "_libsynth.so")
_lib = None
_lib_lock = threading.Lock()


def build_fill_library(force: bool = False) -> str:
    """Compile fill.c into _libsynth.so next to it (plain C, no target-specific flags)."""
    src = os.path.join(_HERE, "fill.c")
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(src):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-shared", "-fPIC", "-pthread", "-o", tmp, src])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _fill_lib():
    global _lib
    with _lib_lock:
        if _lib is None:
            lib = ctypes.CDLL(build_fill_library())
            lib.synth_fill_normal_bf16.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_size_t,
                                                   ctypes.c_float, ctypes.c_void_p, ctypes.c_int]
            lib.synth_fill_normal_bf16.restype = None
            _lib = lib
    return _lib


def fill_normal_bf16(key: int, start: int, count: int, std: float, out: np.ndarray | None = None) -> np.ndarray:
    """Elements [start, start+count) of a normal stream as bf16 bit patterns (uint16)."""
    if out is None:
        out = np.empty(count, dtype=np.uint16)
    assert out.dtype == np.uint16 and out.flags.c_contiguous and out.size == count
    _fill_lib().synth_fill_normal_bf16(key, start, count, float(normal_scale(std)),
                                       out.ctypes.data, min(os.cpu_count() or 1, 32))
    return out


# ----------------------------------------------------------------------------------------------
# model weights
# ----------------------------------------------------------------------------------------------
@dataclass(frozen=True)
class ModelShape:
    n_layers: int
    d_model: int
    n_heads: int
    head_dim: int
    ffn: int
    vocab: int
    rope_base: float = 10000.0
    rms_eps: float = 1e-5


TINY = ModelShape(2, 256, 4, 64, 688, 1024)
LLAMA7B = ModelShape(32, 4096, 32, 128, 11008, 32000)
LLAMA13B = ModelShape(40, 5120, 40, 128, 13824, 32000)

WEIGHT_KINDS = {"embed": K_EMBED, "wqkv": K_WQKV, "wo": K_WO, "wg": K_WG, "wu": K_WU, "wd": K_WD,
                "lm_head": K_LM_HEAD}


def weight_shape(shape: ModelShape, name: str) -> tuple[int, int]:
    d, f, v = shape.d_model, shape.ffn, shape.vocab
    return {"embed": (v, d), "wqkv": (3 * d, d), "wo": (d, d), "wg": (f, d), "wu": (f, d),
            "wd": (d, f), "lm_head": (v, d)}[name]


def weight_bf16(seed: int, shape: ModelShape, name: str, layer: int = 0,
                rows: tuple[int, int] | None = None) -> np.ndarray:
    """Weight tensor `name` of `layer` as bf16 bits [rows, cols] (row-major, [out, in] convention).

    `rows=(r0, r1)` returns only that row range (same bytes as the full tensor's rows).
    Wqkv stacks Wq, Wk, Wv along rows; embed and lm_head ignore `layer`.
    """
    nr, nc = weight_shape(shape, name)
    r0, r1 = rows if rows is not None else (0, nr)
    key = stream_key(seed, WEIGHT_KINDS[name], layer if name not in ("embed", "lm_head") else 0)
    out = fill_normal_bf16(key, r0 * nc, (r1 - r0) * nc, WEIGHT_STD)
    return out.reshape(r1 - r0, nc)


def gains(shape: ModelShape) -> np.ndarray:
    """RMSNorm gains (all 1.0: N(0, 0.02) gains would collapse the residual signal)."""
    return np.ones(shape.d_model, dtype=np.float32)


def prefix_kv_bf16(seed: int, shape: ModelShape, layer: int, which: str, prefix_len: int) -> np.ndarray:
    """Stand-in prefix cache: K or V of `layer` as bf16 bits [n_heads, prefix_len, head_dim], N(0, 1)."""
    kind = K_PREFIX_K if which == "k" else K_PREFIX_V
    key = stream_key(seed, kind, layer)
    n = shape.n_heads * prefix_len * shape.head_dim
    return fill_normal_bf16(key, 0, n, 1.0).reshape(shape.n_heads, prefix_len, shape.head_dim)


# ----------------------------------------------------------------------------------------------
# discrete inputs
# ----------------------------------------------------------------------------------------------
def tokens(seed: int, n: int, vocab: int, sub: int = 0) -> np.ndarray:
    c = Counter(stream_key(seed, K_TOKENS, 0, sub))
    return np.array([c.below(vocab) for _ in range(n)], dtype=np.int32)


def prefix_tokens(seed: int, n: int, vocab: int) -> np.ndarray:
    c = Counter(stream_key(seed, K_PREFIX_TOKENS))
    return np.array([c.below(vocab) for _ in range(n)], dtype=np.int32)


def tree(seed: int, n: int, max_depth: int, max_branch: int | None = None, sub: int = 0) -> np.ndarray:
    """parent_idx[n] of a random rooted tree in topological order (parent[0] = -1, parent[i] < i)."""
    c = Counter(stream_key(seed, K_TREE, 0, sub))
    parent = [-1]
    depth = [0]
    kids = [0]
    for i in range(1, n):
        ok = [p for p in range(i) if depth[p] < max_depth and (max_branch is None or kids[p] < max_branch)]
        if not ok:
            raise ValueError("tree constraints admit no parent")
        p = ok[c.below(len(ok))]
        parent.append(p)
        depth.append(depth[p] + 1)
        kids[p] += 1
        kids.append(0)
    return np.array(parent, dtype=np.int32)


def chain(n: int) -> np.ndarray:
    """parent_idx of a chain (node i's parent is i-1)."""
    return np.arange(-1, n - 1, dtype=np.int32)


def skip_masks(seed: int, n_layers: int, fractions_off: list[float]) -> list[np.ndarray]:
    """Nested layer-skip masks: mask[j][l] = 0 for the first floor(f_j * L) layers of one seeded
    permutation, 1 otherwise.  Larger fractions switch off supersets of smaller ones."""
    c = Counter(stream_key(seed, K_MASK))
    perm = list(range(n_layers))
    for i in range(n_layers - 1, 0, -1):  # Fisher-Yates
        j = c.below(i + 1)
        perm[i], perm[j] = perm[j], perm[i]
    out = []
    for f in fractions_off:
        m = np.ones(n_layers, dtype=np.uint8)
        m[perm[: int(math.floor(f * n_layers + 1e-9))]] = 0
        out.append(m)
    return out
