"""Python binding of libcasspec (include/casspec.h): argument marshalling only.

Every function mirrors the C entry point of the same name without the ``casspec_`` prefix.
Device buffers are torch CUDA tensors (passed by data pointer); streams are torch.cuda.Stream
objects or raw handles.  Loading fails loudly if the CUDA library has not been built: there is no
fallback implementation.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libcasspec.so")

OK, E_INVAL, E_SHAPE, E_CAPACITY, E_CUDA, E_TREE, E_TIMEOUT, E_STATE = 0, -1, -2, -3, -4, -5, -6, -7
MAX_TREE = 64
TOPK_MAX = 8
DYTC_MAX_CLASS = 4  # latency-model classes (one regression per step arithmetic)
DYTC_WORK = 24 * MAX_TREE  # int32 entries of casspec_dytc_round's device scratch
SKIP_ATTN, SKIP_FFN = 0x2, 0x4  # skip-mask flags on a non-zero byte: drop the attention / FFN block
OPT_PDL, OPT_GRAPHS, OPT_TEST_STALL, OPT_W4_TC, OPT_W8_TC = 1, 2, 4, 8, 16

(T_EMBED, T_LM_HEAD, T_FINAL_NORM, T_ATTN_NORM, T_FFN_NORM, T_WQKV, T_WO, T_WG, T_WU, T_WD,
 T_WQKV_Q, T_WO_Q, T_WG_Q, T_WU_Q, T_WD_Q, T_WQKV_S, T_WO_S, T_WG_S, T_WU_S, T_WD_S,
 T_RESIDUAL, T_ACT_Q, T_ACT_S,
 T_WQKV_Q4, T_WO_Q4, T_WG_Q4, T_WU_Q4, T_WD_Q4, T_WQKV_S4, T_WO_S4, T_WG_S4, T_WU_S4, T_WD_S4,
 T_WQKV_F8, T_WO_F8, T_WG_F8, T_WU_F8, T_WD_F8) = range(38)

EXPORTS = [
    "casspec_model_bytes", "casspec_create_model", "casspec_destroy_model", "casspec_set_stream",
    "casspec_set_options", "casspec_set_act_sparsity", "casspec_sparsify_rows", "casspec_tensor", "casspec_quantize_weights", "casspec_kv_bytes", "casspec_kv_create",
    "casspec_kv_destroy", "casspec_kv_layer", "casspec_kv_set_prefix", "casspec_kv_reset_tree", "casspec_kv_length",
    "casspec_tree_step", "casspec_argmax", "casspec_accept_greedy", "casspec_kv_compact", "casspec_get_status",
    "casspec_status_string", "casspec_linear_workspace_bytes", "casspec_linear_bf16", "casspec_linear_bf16_static", "casspec_linear_bf16_static_status",
    "casspec_rmsnorm",
    "casspec_quantize_rows", "casspec_quantize_rows4", "casspec_profile", "casspec_profile_read", "casspec_launch_count",
    "casspec_ewif_sd", "casspec_ewif_hc", "casspec_ewif_vc", "casspec_dytc_objective", "casspec_dytc_create",
    "casspec_dytc_destroy", "casspec_dytc_get_params", "casspec_dytc_set_cost", "casspec_dytc_alpha", "casspec_dytc_cost", "casspec_dytc_best_config",
    "casspec_dytc_record", "casspec_dytc_end_step", "casspec_dytc_tree_reset", "casspec_dytc_tree_plan",
    "casspec_dytc_tree_extend", "casspec_dytc_tree_begin", "casspec_dytc_tree_add", "casspec_vc_accept", "casspec_dytc_tree_get", "casspec_dytc_round", "casspec_latency_fit", "casspec_step_bytes", "casspec_dytc_observe", "casspec_dytc_fit_costs", "casspec_pld_draft", "casspec_topk",
]
K_QKV, K_ATTN, K_WO, K_GATEUP, K_DOWN, K_LMHEAD, K_OTHER, K_COUNT = range(8)


class ModelConfig(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("d_model", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("ffn", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("rope_base", ctypes.c_float), ("rms_eps", ctypes.c_float), ("with_int8", ctypes.c_int32)]


class DytcParams(ctypes.Structure):
    _fields_ = [("n_cfg", ctypes.c_int32), ("alpha_dn", ctypes.c_double), ("c_dn", ctypes.c_double),
                ("k_max", ctypes.c_int32), ("t_min", ctypes.c_double), ("m_max", ctypes.c_int32),
                ("lambda_", ctypes.c_double), ("window", ctypes.c_int32), ("topk", ctypes.c_int32),
                ("p_tree", ctypes.c_double)]


class DraftCfg(ctypes.Structure):
    _fields_ = [("skip_mask", ctypes.c_void_p), ("quant_mode", ctypes.c_int32), ("pld_n_max", ctypes.c_int32),
                ("vc", ctypes.c_int32)]


class CasspecError(RuntimeError):
    def __init__(self, fn: str, rc: int):
        super().__init__(f"{fn} failed: {rc} ({status_string(rc)})")
        self.rc = rc


_lib = None
_P = ctypes.c_void_p
_I = ctypes.c_int
_SZ = ctypes.c_size_t
_D = ctypes.c_double


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libcasspec.so (raises if it is missing: build it with __graft_entry__.build())."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: the CUDA library must be built (python -c 'import __graft_entry__ as g; g.build()')")
    lib = ctypes.CDLL(path)
    sig = {
        "casspec_model_bytes": (_SZ, [ctypes.POINTER(ModelConfig)]),
        "casspec_ewif_sd": (_D, [_D, _D, _I]),
        "casspec_ewif_hc": (_D, [_D, _D, _I, _D, _D, _I]),
        "casspec_ewif_vc": (_D, [_D, _D, _D, _D, _I, _I]),
        "casspec_dytc_objective": (_D, [_D, _D, _I, _D, _D]),
        "casspec_dytc_create": (_I, [ctypes.POINTER(DytcParams), ctypes.POINTER(_D), ctypes.POINTER(_D), ctypes.POINTER(_P)]),
        "casspec_dytc_destroy": (None, [_P]),
        "casspec_dytc_get_params": (_I, [_P, ctypes.POINTER(DytcParams)]),
        "casspec_dytc_set_cost": (_I, [_P, _I, _D]),
        "casspec_dytc_alpha": (_I, [_P, _I, ctypes.POINTER(_D)]),
        "casspec_dytc_cost": (_I, [_P, _I, ctypes.POINTER(_D)]),
        "casspec_dytc_best_config": (_I, [_P, ctypes.POINTER(_I), ctypes.POINTER(_I), ctypes.POINTER(_D)]),
        "casspec_dytc_record": (_I, [_P, _I, _I]),
        "casspec_dytc_end_step": (_I, [_P]),
        "casspec_dytc_tree_reset": (_I, [_P]),
        "casspec_dytc_tree_plan": (_I, [_P, ctypes.POINTER(_I), ctypes.POINTER(_I), ctypes.POINTER(_I)]),
        "casspec_dytc_tree_extend": (_I, [_P, _I, _I, _I, ctypes.POINTER(ctypes.c_int32)]),
        "casspec_vc_accept": (_I, [ctypes.POINTER(ctypes.c_int32), _I, ctypes.POINTER(ctypes.c_int32),
                                   ctypes.POINTER(ctypes.c_int32)]),
        "casspec_dytc_tree_begin": (_I, [_P, _I, _I, ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(_I)]),
        "casspec_dytc_tree_add": (_I, [_P, _I, _I, ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_float), _I]),
        "casspec_pld_draft": (_I, [_P, _I, _I, _I, _I, _P, _P]),
        "casspec_topk": (_I, [_P, _I, _I, _I, _P, _P, _P]),
        "casspec_step_bytes": (_D, [ctypes.POINTER(ModelConfig), _P, _I, _I, _I]),
        "casspec_dytc_observe": (_I, [_P, _I, _D, _D]),
        "casspec_dytc_fit_costs": (_I, [_P, ctypes.POINTER(_I), ctypes.POINTER(_D), _D, ctypes.POINTER(_D),
                                        ctypes.POINTER(_D), _D, ctypes.POINTER(_D)]),
        "casspec_latency_fit": (_I, [ctypes.POINTER(_D), ctypes.POINTER(_D), _I, ctypes.POINTER(_D), ctypes.POINTER(_D), _D,
                                     ctypes.POINTER(_D), ctypes.POINTER(_D)]),
        "casspec_dytc_round": (_I, [_P, _P, _P, ctypes.POINTER(DraftCfg), ctypes.c_int32, _P, _I, _P, _P,
                                    ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(_I), ctypes.POINTER(_I)]),
        "casspec_dytc_tree_get": (_I, [_P, ctypes.POINTER(_I), ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int32),
                                       ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(_D)]),
        "casspec_create_model": (_I, [ctypes.POINTER(ModelConfig), _P, _SZ, ctypes.POINTER(_P)]),
        "casspec_destroy_model": (None, [_P]),
        "casspec_set_stream": (_I, [_P, _P]),
        "casspec_set_options": (_I, [_P, ctypes.c_uint, ctypes.POINTER(ctypes.c_uint)]),
        "casspec_set_act_sparsity": (_I, [_P, ctypes.c_float]),
        "casspec_sparsify_rows": (_I, [_P, _I, _I, _I, ctypes.c_float, _P]),
        "casspec_tensor": (_I, [_P, _I, _I, ctypes.POINTER(_P), ctypes.POINTER(_SZ)]),
        "casspec_quantize_weights": (_I, [_P]),
        "casspec_kv_bytes": (_SZ, [ctypes.POINTER(ModelConfig), _I]),
        "casspec_kv_create": (_I, [_P, _I, _P, _SZ, ctypes.POINTER(_P)]),
        "casspec_kv_destroy": (None, [_P]),
        "casspec_kv_layer": (_I, [_P, _I, ctypes.POINTER(_P), ctypes.POINTER(_P), ctypes.POINTER(_I)]),
        "casspec_kv_set_prefix": (_I, [_P, _I]),
        "casspec_kv_reset_tree": (_I, [_P]),
        "casspec_kv_length": (_I, [_P, ctypes.POINTER(_I), ctypes.POINTER(_I)]),
        "casspec_tree_step": (_I, [_P, _P, _P, _P, _I, _P, _I, _P]),
        "casspec_argmax": (_I, [_P, ctypes.POINTER(_P), ctypes.POINTER(_P)]),
        "casspec_accept_greedy": (_I, [_P, _P, _P, _P, _I, _P]),
        "casspec_kv_compact": (_I, [_P, _P]),
        "casspec_get_status": (_I, [_P, ctypes.POINTER(_I)]),
        "casspec_status_string": (ctypes.c_char_p, [_I]),
        "casspec_linear_workspace_bytes": (_SZ, [_I, _I, _I]),
        "casspec_linear_bf16": (_I, [_P, _I, _I, _P, _I, _P, _I, _P, _SZ, _P]),
        "casspec_linear_bf16_static": (_I, [_P, _I, _I, _P, _I, _P, _I, _P]),
        "casspec_linear_bf16_static_status": (_I, [_P, ctypes.POINTER(_I)]),
        "casspec_rmsnorm": (_I, [_P, _P, _I, _I, ctypes.c_float, _P, _P, _P, _P]),
        "casspec_quantize_rows": (_I, [_P, _I, _I, _P, _P, _P]),
        "casspec_quantize_rows4": (_I, [_P, _I, _I, _P, _P, _P]),
        "casspec_profile": (_I, [_P, _I]),
        "casspec_profile_read": (_I, [_P, _I, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(_I)]),
        "casspec_launch_count": (_I, [_P, ctypes.POINTER(ctypes.c_uint64)]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def _ptr(t) -> int | None:
    """Device pointer of a torch tensor (or None / raw int)."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(s) -> int | None:
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(fn: str, rc: int) -> None:
    if rc != OK:
        raise CasspecError(fn, rc)


def config(n_layers, d_model, n_heads, head_dim, ffn, vocab, rope_base=10000.0, rms_eps=1e-5, with_int8=0):
    return ModelConfig(n_layers, d_model, n_heads, head_dim, ffn, vocab, rope_base, rms_eps, int(with_int8))


def model_bytes(cfg: ModelConfig) -> int:
    return load_library().casspec_model_bytes(ctypes.byref(cfg))


def create_model(cfg: ModelConfig, dev_mem) -> int:
    h = _P()
    _check("casspec_create_model",
           load_library().casspec_create_model(ctypes.byref(cfg), _ptr(dev_mem), dev_mem.numel() * dev_mem.element_size(),
                                               ctypes.byref(h)))
    return h.value


def destroy_model(m: int) -> None:
    load_library().casspec_destroy_model(m)


def set_stream(m: int, stream) -> None:
    _check("casspec_set_stream", load_library().casspec_set_stream(m, _stream(stream)))


def set_options(m: int, flags: int) -> int:
    old = ctypes.c_uint()
    _check("casspec_set_options", load_library().casspec_set_options(m, flags, ctypes.byref(old)))
    return old.value


def set_act_sparsity(m: int, s: float) -> None:
    """casspec_set_act_sparsity: the activation sparsity s of the model's bf16 steps (0: dense)."""
    _check("casspec_set_act_sparsity", load_library().casspec_set_act_sparsity(m, float(s)))


def sparsify_rows(x_split, ld: int, n: int, K: int, s: float, stream=None) -> None:
    """casspec_sparsify_rows: the sparsity rule on a split activation [128][ld] bf16, in place."""
    _check("casspec_sparsify_rows", load_library().casspec_sparsify_rows(_ptr(x_split), ld, n, K, float(s),
                                                                          _stream(stream)))


def tensor(m: int, tensor_id: int, layer: int = 0) -> tuple[int, int]:
    p, nb = _P(), _SZ()
    _check("casspec_tensor", load_library().casspec_tensor(m, tensor_id, layer, ctypes.byref(p), ctypes.byref(nb)))
    return p.value, nb.value


def quantize_weights(m: int) -> None:
    _check("casspec_quantize_weights", load_library().casspec_quantize_weights(m))


def kv_bytes(cfg: ModelConfig, max_ctx: int) -> int:
    return load_library().casspec_kv_bytes(ctypes.byref(cfg), max_ctx)


def kv_create(m: int, max_ctx: int, dev_mem) -> int:
    h = _P()
    _check("casspec_kv_create", load_library().casspec_kv_create(m, max_ctx, _ptr(dev_mem),
                                                                 dev_mem.numel() * dev_mem.element_size(), ctypes.byref(h)))
    return h.value


def kv_destroy(kv: int) -> None:
    load_library().casspec_kv_destroy(kv)


def kv_layer(kv: int, layer: int) -> tuple[int, int, int]:
    k, v, ld = _P(), _P(), _I()
    _check("casspec_kv_layer", load_library().casspec_kv_layer(kv, layer, ctypes.byref(k), ctypes.byref(v), ctypes.byref(ld)))
    return k.value, v.value, ld.value


def kv_set_prefix(kv: int, P: int) -> None:
    _check("casspec_kv_set_prefix", load_library().casspec_kv_set_prefix(kv, P))


def kv_reset_tree(kv: int) -> None:
    _check("casspec_kv_reset_tree", load_library().casspec_kv_reset_tree(kv))


def kv_length(kv: int) -> tuple[int, int]:
    P, T = _I(), _I()
    _check("casspec_kv_length", load_library().casspec_kv_length(kv, ctypes.byref(P), ctypes.byref(T)))
    return P.value, T.value


def tree_step(m: int, kv: int, tokens, parent_idx, n: int, skip_mask=None, quant_mode: int = 0, logits_out=None,
              check: bool = True) -> int:
    mask = None
    if skip_mask is not None:
        mask = np.ascontiguousarray(np.asarray(skip_mask, dtype=np.uint8))
    rc = load_library().casspec_tree_step(m, kv, _ptr(tokens), _ptr(parent_idx), n,
                                          None if mask is None else mask.ctypes.data, quant_mode, _ptr(logits_out))
    if check:
        _check("casspec_tree_step", rc)
    return rc


def argmax(m: int) -> tuple[int, int]:
    a, g = _P(), _P()
    _check("casspec_argmax", load_library().casspec_argmax(m, ctypes.byref(a), ctypes.byref(g)))
    return a.value, g.value


def accept_greedy(m: int, logits, tokens, parent_idx, n: int, accepted_out) -> None:
    _check("casspec_accept_greedy",
           load_library().casspec_accept_greedy(m, _ptr(logits), _ptr(tokens), _ptr(parent_idx), n, _ptr(accepted_out)))


def kv_compact(kv: int, accepted_out, check: bool = True) -> int:
    rc = load_library().casspec_kv_compact(kv, _ptr(accepted_out))
    if check:
        _check("casspec_kv_compact", rc)
    return rc


def get_status(m: int) -> int:
    st = _I()
    _check("casspec_get_status", load_library().casspec_get_status(m, ctypes.byref(st)))
    return st.value


def status_string(rc: int) -> str:
    try:
        return load_library().casspec_status_string(rc).decode()
    except RuntimeError:
        return str(rc)


def linear_workspace_bytes(N: int, K: int, n: int) -> int:
    return load_library().casspec_linear_workspace_bytes(N, K, n)


def linear_bf16(W, N: int, K: int, X, n: int, Y, ldy: int, workspace, stream=None) -> None:
    _check("casspec_linear_bf16",
           load_library().casspec_linear_bf16(_ptr(W), N, K, _ptr(X), n, _ptr(Y), ldy, _ptr(workspace),
                                              workspace.numel() * workspace.element_size(), _stream(stream)))


def linear_bf16_static(W, N: int, K: int, X, n: int, Y, ldy: int, stream=None) -> None:
    _check("casspec_linear_bf16_static",
           load_library().casspec_linear_bf16_static(_ptr(W), N, K, _ptr(X), n, _ptr(Y), ldy, _stream(stream)))


def linear_bf16_static_status(stream=None) -> int:
    """Status word of the latest casspec_linear_bf16_static call on the current device (syncs)."""
    st = _I()
    _check("casspec_linear_bf16_static_status",
           load_library().casspec_linear_bf16_static_status(_stream(stream), ctypes.byref(st)))
    return st.value


def rmsnorm(x, g, n: int, d: int, eps: float, y=None, q=None, s=None, stream=None) -> None:
    _check("casspec_rmsnorm", load_library().casspec_rmsnorm(_ptr(x), _ptr(g), n, d, eps, _ptr(y), _ptr(q), _ptr(s),
                                                             _stream(stream)))


def quantize_rows(x, n: int, d: int, q, s, stream=None) -> None:
    _check("casspec_quantize_rows", load_library().casspec_quantize_rows(_ptr(x), n, d, _ptr(q), _ptr(s), _stream(stream)))


def quantize_rows4(x, n: int, d: int, q4, s, stream=None) -> None:
    """casspec_quantize_rows4: codes in [-7, 7], two per byte (q4: [n][d / 2] uint8)."""
    _check("casspec_quantize_rows4", load_library().casspec_quantize_rows4(_ptr(x), n, d, _ptr(q4), _ptr(s),
                                                                            _stream(stream)))


def unpack_int4(b: np.ndarray, K: int) -> np.ndarray:
    """Codes of int4 rows ([rows][K / 2] bytes, column 2j in the low nibble of byte j) as int8 [rows][K]."""
    b = np.asarray(b, dtype=np.uint8).reshape(-1, K // 2)
    lo, hi = (b & 0x0F).astype(np.int16), (b >> 4).astype(np.int16)
    out = np.empty((b.shape[0], K), dtype=np.int8)
    out[:, 0::2] = np.where(lo > 7, lo - 16, lo)
    out[:, 1::2] = np.where(hi > 7, hi - 16, hi)
    return out


def decode_e4m3_codes(b: np.ndarray) -> np.ndarray:
    """Integer codes in [-16, 16] from their FP8 e4m3 bytes (sign, 4 exponent bits with bias 7, 3
    fraction bits); only exact integers are expected."""
    b = np.asarray(b, dtype=np.uint8)
    e = ((b >> 3) & 15).astype(np.int64)
    f = (b & 7).astype(np.int64)
    mag = np.where(e == 0, 0, ((8 + f) << np.maximum(e - 7, 0)) >> 3)
    return np.where(b & 0x80, -mag, mag).astype(np.int8)


def profile(m: int, enable: bool) -> None:
    _check("casspec_profile", load_library().casspec_profile(m, int(enable)))


def profile_read(m: int, kind: int) -> tuple[float, int]:
    """(total device ms, launches) of kernel kind `kind` since profiling was enabled."""
    t, c = ctypes.c_double(), _I()
    _check("casspec_profile_read", load_library().casspec_profile_read(m, kind, ctypes.byref(t), ctypes.byref(c)))
    return t.value, c.value


def launch_count(m: int) -> int:
    c = ctypes.c_uint64()
    _check("casspec_launch_count", load_library().casspec_launch_count(m, ctypes.byref(c)))
    return c.value


# ------------------------------------------------------------------------------------------------
# DyTC scheduling (host code in the library; no GPU work)
# ------------------------------------------------------------------------------------------------
def ewif_sd(alpha: float, c: float, k: int) -> float:
    return load_library().casspec_ewif_sd(alpha, c, k)


def ewif_hc(a1: float, c1: float, k1: int, a2: float, c2: float, k2: int) -> float:
    return load_library().casspec_ewif_hc(a1, c1, k1, a2, c2, k2)


def ewif_vc(alpha: float, alpha12: float, c1: float, c2: float, n: int, k: int) -> float:
    return load_library().casspec_ewif_vc(alpha, alpha12, c1, c2, n, k)


def dytc_objective(alpha: float, c: float, k: int, alpha_dn: float, c_dn: float) -> float:
    return load_library().casspec_dytc_objective(alpha, c, k, alpha_dn, c_dn)


def vc_accept(proposals, argmax) -> list[int]:
    """casspec_vc_accept: d_i's drafted tokens of one vertical-cascade round (host lists)."""
    j = len(proposals)
    p = (ctypes.c_int32 * max(j, 1))(*[int(x) for x in proposals])
    a = (ctypes.c_int32 * (j + 1))(*[int(x) for x in argmax[: j + 1]])
    out = (ctypes.c_int32 * (j + 1))()
    rc = load_library().casspec_vc_accept(p, j, a, out)
    if rc < 0:
        raise CasspecError("casspec_vc_accept", rc)
    return list(out[:rc])


def pld_draft(tokens, L: int, n_min: int, n_max: int, k: int, out, stream=None) -> None:
    """casspec_pld_draft: tokens dev int32 [L], out dev int32 [2 + k] = {match length, count, tokens}."""
    _check("casspec_pld_draft", load_library().casspec_pld_draft(_ptr(tokens), L, n_min, n_max, k, _ptr(out),
                                                                   _stream(stream)))


def topk(logits, n: int, V: int, K: int, idx_out, prob_out, stream=None) -> None:
    """casspec_topk: logits dev fp32 [n][V] -> idx_out dev int32 [n][K], prob_out dev fp32 [n][K]."""
    _check("casspec_topk", load_library().casspec_topk(_ptr(logits), n, V, K, _ptr(idx_out), _ptr(prob_out),
                                                         _stream(stream)))


def latency_fit(x, y, mu0, sd0, noise_sd: float) -> tuple[list[float], list[float]]:
    """Posterior mean [w0, w1] and covariance (row-major 2 x 2) of latency = w0 + w1 * bytes."""
    m = len(x)
    xa, ya = (_D * max(m, 1))(*[float(v) for v in x]), (_D * max(m, 1))(*[float(v) for v in y])
    mu, sd = (_D * 2)(*[float(v) for v in mu0]), (_D * 2)(*[float(v) for v in sd0])
    w, cov = (_D * 2)(), (_D * 4)()
    _check("casspec_latency_fit", load_library().casspec_latency_fit(xa, ya, m, mu, sd, float(noise_sd), w, cov))
    return list(w), list(cov)


def step_bytes(cfg: ModelConfig, skip_mask=None, quant_mode: int = 0, n: int = 1, P: int = 0) -> float:
    """casspec_step_bytes: algorithmic bytes of one tree step of this configuration."""
    mk = None if skip_mask is None else np.ascontiguousarray(np.asarray(skip_mask, dtype=np.uint8))
    v = load_library().casspec_step_bytes(ctypes.byref(cfg), None if mk is None else mk.ctypes.data, int(quant_mode),
                                          int(n), int(P))
    if v < 0:
        raise CasspecError("casspec_step_bytes", E_INVAL)
    return v


def draft_cfgs(cfgs):
    """casspec_draft_cfg array for casspec_dytc_round, and the mask arrays it points into (keep them
    alive for the call).  Each entry: (skip_mask or None, quant_mode) for a model draft,
    ("pld", n_max) for the prompt lookup, ("vc", skip_mask or None, quant_mode, n_max) for the
    vertical cascade of that model draft over the prompt lookup."""
    masks, items = [], []
    for cfg in cfgs:
        kind = cfg[0] if isinstance(cfg[0], str) else None
        if kind == "pld":
            masks.append(None)
            items.append(DraftCfg(None, 0, int(cfg[1]), 0))
            continue
        a, b, n_vc = (cfg[1], cfg[2], int(cfg[3])) if kind == "vc" else (cfg[0], cfg[1], 0)
        mk = None if a is None else np.ascontiguousarray(np.asarray(a, dtype=np.uint8))
        masks.append(mk)
        items.append(DraftCfg(None if mk is None else mk.ctypes.data, int(b), n_vc, int(n_vc > 0)))
    return (DraftCfg * len(items))(*items), masks


class Dytc:
    """Owner of one native DyTC scheduler (casspec_dytc_*)."""

    def __init__(self, alphas, costs, alpha_dn: float, c_dn: float, k_max: int, t_min: float, m_max: int,
                 lam: float = 0.7, window: int = 20, topk: int = 1, p_tree: float = 1.0):
        lib = load_library()
        n = len(alphas)
        p = DytcParams(n, alpha_dn, c_dn, k_max, t_min, m_max, lam, window, topk, p_tree)
        a = (_D * n)(*alphas)
        c = (_D * n)(*costs)
        h = _P()
        _check("casspec_dytc_create", lib.casspec_dytc_create(ctypes.byref(p), a, c, ctypes.byref(h)))
        self.h, self.m_max, self.n_cfg = h.value, m_max, n

    def close(self) -> None:
        if self.h:
            load_library().casspec_dytc_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_cost(self, cfg: int, cost: float) -> None:
        _check("casspec_dytc_set_cost", load_library().casspec_dytc_set_cost(self.h, cfg, cost))

    def alpha(self, cfg: int) -> float:
        v = _D()
        _check("casspec_dytc_alpha", load_library().casspec_dytc_alpha(self.h, cfg, ctypes.byref(v)))
        return v.value

    def cost(self, cfg: int) -> float:
        v = _D()
        _check("casspec_dytc_cost", load_library().casspec_dytc_cost(self.h, cfg, ctypes.byref(v)))
        return v.value

    def best_config(self) -> tuple[int | None, int, float]:
        s, k, v = _I(), _I(), _D()
        _check("casspec_dytc_best_config",
               load_library().casspec_dytc_best_config(self.h, ctypes.byref(s), ctypes.byref(k), ctypes.byref(v)))
        return (None if s.value < 0 else s.value), k.value, v.value

    def record(self, cfg: int, accepted: bool) -> None:
        _check("casspec_dytc_record", load_library().casspec_dytc_record(self.h, cfg, int(bool(accepted))))

    def end_step(self) -> None:
        _check("casspec_dytc_end_step", load_library().casspec_dytc_end_step(self.h))

    def tree_reset(self) -> None:
        _check("casspec_dytc_tree_reset", load_library().casspec_dytc_tree_reset(self.h))

    def tree_plan(self) -> tuple[int, int, int] | None:
        leaf, s, k = _I(), _I(), _I()
        rc = load_library().casspec_dytc_tree_plan(self.h, ctypes.byref(leaf), ctypes.byref(s), ctypes.byref(k))
        if rc < 0:
            raise CasspecError("casspec_dytc_tree_plan", rc)
        return (leaf.value, s.value, k.value) if rc == 1 else None

    def tree_extend(self, leaf: int, cfg: int, tokens) -> int:
        t = (ctypes.c_int32 * len(tokens))(*[int(x) for x in tokens])
        rc = load_library().casspec_dytc_tree_extend(self.h, leaf, cfg, len(tokens), t)
        if rc < 0:
            raise CasspecError("casspec_dytc_tree_extend", rc)
        return rc

    def observe(self, cls: int, bytes_moved: float, us: float) -> None:
        """Record one measured step of arithmetic class `cls` (its quant_mode)."""
        _check("casspec_dytc_observe",
               load_library().casspec_dytc_observe(self.h, int(cls), float(bytes_moved), float(us)))

    def fit_costs(self, cfg_class, cfg_bytes, target_bytes: float, mu0, sd0, noise_sd: float) -> list[list[float]]:
        """Refit each class's latency model to its observed steps and reset every configuration's cost;
        returns the fitted w of every class."""
        cc = (_I * self.n_cfg)(*[int(v) for v in cfg_class])
        cb = (_D * self.n_cfg)(*[float(v) for v in cfg_bytes])
        mu, sd = (_D * 2)(*[float(v) for v in mu0]), (_D * 2)(*[float(v) for v in sd0])
        w = (_D * (2 * DYTC_MAX_CLASS))()
        _check("casspec_dytc_fit_costs",
               load_library().casspec_dytc_fit_costs(self.h, cc, cb, float(target_bytes), mu, sd, float(noise_sd), w))
        return [[w[2 * k], w[2 * k + 1]] for k in range(DYTC_MAX_CLASS)]

    def tree_begin(self, leaf: int, siblings: bool = True) -> list[int]:
        br, nb = (ctypes.c_int32 * MAX_TREE)(), _I()
        _check("casspec_dytc_tree_begin",
               load_library().casspec_dytc_tree_begin(self.h, leaf, int(bool(siblings)), br, ctypes.byref(nb)))
        return list(br[: nb.value])

    def tree_add(self, node: int, cfg: int, tokens, probs) -> int:
        """Candidates (rank order) of one drafted position below `node`; returns the top-1 child,
        0 when the tree is full."""
        kc = len(tokens)
        t = (ctypes.c_int32 * kc)(*[int(x) for x in tokens])
        p = (ctypes.c_float * kc)(*[float(x) for x in probs])
        rc = load_library().casspec_dytc_tree_add(self.h, node, cfg, t, p, kc)
        if rc < 0:
            raise CasspecError("casspec_dytc_tree_add", rc)
        return rc

    def tree_get(self) -> dict:
        m = self.m_max
        n = _I()
        par, tok, cfg = (ctypes.c_int32 * m)(), (ctypes.c_int32 * m)(), (ctypes.c_int32 * m)()
        pacc = (_D * m)()
        _check("casspec_dytc_tree_get", load_library().casspec_dytc_tree_get(self.h, ctypes.byref(n), par, tok, cfg, pacc))
        k = n.value
        return {"parent": list(par[:k]), "token": list(tok[:k]), "cfg": list(cfg[:k]), "p_acc": list(pacc[:k])}

    def round(self, m: int, kv: int, cfgs, root_token: int, dev_work, history=None, hist_len: int = 0,
              dev_logits=None) -> tuple[list[int], int]:
        """One DyTC round (casspec_dytc_round).  cfgs: per configuration (skip_mask or None, quant_mode)
        for a model draft, ("pld", n_max) for the prompt-lookup draft, or ("vc", skip_mask, quant_mode,
        n_max) for the vertical cascade of that model draft over the prompt lookup; history: torch int32 CUDA
        tensor of the committed tokens (hist_len valid, the last = root_token, room for MAX_TREE more);
        dev_work: torch int32 CUDA tensor of DYTC_WORK entries; dev_logits: torch fp32 CUDA tensor of
        MAX_TREE x vocab (needed when topk > 1).  Returns the committed tokens (the last is the bonus
        token) and the number of drafted nodes."""
        arr, masks = draft_cfgs(cfgs)
        out = (ctypes.c_int32 * MAX_TREE)()
        n, nd = _I(), _I()
        _check("casspec_dytc_round", load_library().casspec_dytc_round(self.h, m, kv, arr, int(root_token), _ptr(history),
                                                                       int(hist_len), _ptr(dev_work), _ptr(dev_logits), out,
                                                                       ctypes.byref(n), ctypes.byref(nd)))
        return list(out[: n.value]), nd.value

