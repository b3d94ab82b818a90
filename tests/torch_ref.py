"""Textbook causal Llama forward in torch (CPU, fp64) used to pin the oracle.

It is written independently of the oracle: library routines for RMSNorm, linear layers, SiLU and
causal scaled-dot-product attention, and rotary embedding as a complex multiplication
(pair (x_j, x_{j+h/2}) read as x_j + i x_{j+h/2}, multiplied by exp(i * pos * base^(-2j/h))).
A full-sequence causal forward gives, at every position, the logits of token-by-token
autoregressive decoding, which is what a token tree must reproduce node by node.
"""
from __future__ import annotations

import numpy as np
import torch
import torch.nn.functional as F

import synth


class CausalLM:
    def __init__(self, shape: synth.ModelShape, seed: int, gains=None):
        """gains(name, layer) -> [d] RMSNorm gains ("attn_norm", "ffn_norm", "final_norm"); ones
        if None."""
        self.sh = shape
        one = lambda name, layer: np.ones(shape.d_model)  # noqa: E731
        self.gain = lambda name, layer=-1: torch.as_tensor(  # noqa: E731
            np.asarray((gains or one)(name, layer), dtype=np.float64))
        get = lambda name, layer=0: torch.from_numpy(  # noqa: E731
            synth.bf16_to_f32(synth.weight_bf16(seed, shape, name, layer)).astype(np.float64))
        self.embed = get("embed")
        self.lm_head = get("lm_head")
        self.layers = []
        d = shape.d_model
        for l in range(shape.n_layers):
            wqkv = get("wqkv", l)
            self.layers.append(dict(wq=wqkv[:d], wk=wqkv[d:2 * d], wv=wqkv[2 * d:], wo=get("wo", l),
                                    wg=get("wg", l), wu=get("wu", l), wd=get("wd", l)))

    def _rope(self, x: torch.Tensor, pos: torch.Tensor) -> torch.Tensor:
        # x: [H, S, h]
        h = x.shape[-1]
        half = h // 2
        freq = self.sh.rope_base ** (-2.0 * torch.arange(half, dtype=torch.float64) / h)
        rot = torch.polar(torch.ones(len(pos), half, dtype=torch.float64), pos[:, None].double() * freq[None])
        z = torch.complex(x[..., :half], x[..., half:]) * rot
        return torch.cat([z.real, z.imag], dim=-1)

    def forward(self, tokens, layers_on=None, return_kv: bool = False, blocks=None):
        """Logits [S, V] of a causal forward over `tokens` (positions 0..S-1).  layers_on[l] false
        drops layer l; blocks[l] = (attention on, FFN on) drops single sub-blocks."""
        sh = self.sh
        d = sh.d_model
        toks = torch.as_tensor(np.asarray(tokens), dtype=torch.long)
        S = len(toks)
        pos = torch.arange(S)
        x = self.embed[toks]
        kv = []
        for l, W in enumerate(self.layers):
            attn, ffn = (True, True) if blocks is None else blocks[l]
            if layers_on is not None and not layers_on[l]:
                attn = ffn = False
            if not attn:
                kv.append(None)
            if attn:
                x = self._attention(x, W, l, pos, kv)
            if ffn:
                xn = F.rms_norm(x, (d,), self.gain("ffn_norm", l), sh.rms_eps)
                x = x + F.linear(F.silu(F.linear(xn, W["wg"])) * F.linear(xn, W["wu"]), W["wd"])
        logits = F.linear(F.rms_norm(x, (d,), self.gain("final_norm"), sh.rms_eps), self.lm_head)
        return (logits.numpy(), kv) if return_kv else logits.numpy()

    def _attention(self, x, W, l, pos, kv):
        sh = self.sh
        d, H, h = sh.d_model, sh.n_heads, sh.head_dim
        S = x.shape[0]
        xn = F.rms_norm(x, (d,), self.gain("attn_norm", l), sh.rms_eps)
        q = F.linear(xn, W["wq"]).view(S, H, h).transpose(0, 1)
        k = F.linear(xn, W["wk"]).view(S, H, h).transpose(0, 1)
        v = F.linear(xn, W["wv"]).view(S, H, h).transpose(0, 1)
        q, k = self._rope(q, pos), self._rope(k, pos)
        kv.append((k, v))
        a = F.scaled_dot_product_attention(q[None], k[None], v[None], is_causal=True)[0]
        return x + F.linear(a.transpose(0, 1).reshape(S, d), W["wo"])
