"""Synthetic device workloads for the tree step: a model whose weights come from the seeded input
generator (`synth`) and a KV cache with a stand-in prefix.  Input staging only -- every step of the
decoder runs in the CUDA library."""
from __future__ import annotations

import numpy as np
import torch

import synth

from . import (T_EMBED, T_LM_HEAD, T_WD, T_WG, T_WO, T_WQKV, T_WU, config, create_model, destroy_model,
               kv_bytes, kv_create, kv_destroy, kv_layer, kv_set_prefix, model_bytes, quantize_weights,
               set_stream, tensor)

_LAYER_TENSORS = [("wqkv", T_WQKV), ("wo", T_WO), ("wg", T_WG), ("wu", T_WU), ("wd", T_WD)]


class DeviceModel:
    """A model in one torch-owned device buffer with weights from synth.weight_bf16(seed, shape, ...)."""

    def __init__(self, shape: synth.ModelShape, seed: int, with_int8: bool = False, device: str = "cuda"):
        self.shape, self.seed = shape, seed
        self.cfg = config(shape.n_layers, shape.d_model, shape.n_heads, shape.head_dim, shape.ffn, shape.vocab,
                          shape.rope_base, shape.rms_eps, with_int8)
        self.mem = torch.empty(model_bytes(self.cfg), dtype=torch.uint8, device=device)
        self.h = create_model(self.cfg, self.mem)
        set_stream(self.h, torch.cuda.current_stream())
        self._upload()
        if with_int8:
            quantize_weights(self.h)

    def slot(self, tensor_id: int, layer: int = 0) -> torch.Tensor:
        """uint8 view of the device bytes of one weight tensor."""
        ptr, nb = tensor(self.h, tensor_id, layer)
        off = ptr - self.mem.data_ptr()
        return self.mem[off:off + nb]

    def _put(self, tensor_id: int, layer: int, bits: np.ndarray) -> None:
        self.slot(tensor_id, layer).copy_(torch.from_numpy(np.ascontiguousarray(bits).view(np.uint8).reshape(-1)))

    def _upload(self) -> None:
        sh, s = self.shape, self.seed
        self._put(T_EMBED, 0, synth.weight_bf16(s, sh, "embed"))
        self._put(T_LM_HEAD, 0, synth.weight_bf16(s, sh, "lm_head"))
        for l in range(sh.n_layers):
            for name, tid in _LAYER_TENSORS:
                self._put(tid, l, synth.weight_bf16(s, sh, name, l))
        torch.cuda.synchronize()

    def close(self) -> None:
        if self.h:
            destroy_model(self.h)
            self.h = 0


class DeviceKV:
    """KV cache for `model` with `max_ctx` slots in one torch-owned device buffer."""

    def __init__(self, model: DeviceModel, max_ctx: int):
        self.model = model
        self.mem = torch.empty(kv_bytes(model.cfg, max_ctx), dtype=torch.uint8, device=model.mem.device)
        self.h = kv_create(model.h, max_ctx, self.mem)
        _, _, self.ctx = kv_layer(self.h, 0)

    def layer(self, l: int) -> tuple[torch.Tensor, torch.Tensor]:
        """(K, V) of layer l as int16 views [H][ctx][hd] (bf16 bit patterns)."""
        sh = self.model.shape
        k, v, ld = kv_layer(self.h, l)
        n = sh.n_heads * ld * sh.head_dim
        out = []
        for p in (k, v):
            off = p - self.mem.data_ptr()
            out.append(self.mem[off:off + 2 * n].view(torch.int16).view(sh.n_heads, ld, sh.head_dim))
        return out[0], out[1]

    def load_random_prefix(self, seed: int, P: int) -> None:
        """Install the N(0, 1) stand-in prefix of synth.prefix_kv_bf16 in every layer; sets P."""
        sh = self.model.shape
        for l in range(sh.n_layers):
            K, V = self.layer(l)
            for which, dst in (("k", K), ("v", V)):
                bits = synth.prefix_kv_bf16(seed, sh, l, which, P)
                dst[:, :P, :].copy_(torch.from_numpy(bits.view(np.int16)))
        kv_set_prefix(self.h, P)
        torch.cuda.synchronize()

    def close(self) -> None:
        if self.h:
            kv_destroy(self.h)
            self.h = 0


def bf16_bits_to_float(t: torch.Tensor) -> np.ndarray:
    """int16 tensor of bf16 bit patterns -> float32 numpy array (exact)."""
    return synth.bf16_to_f32(t.cpu().numpy().view(np.uint16))
