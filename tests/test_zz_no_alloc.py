"""casspec_linear_bf16_static (no workspace, static device scratch) against casspec_linear_bf16.

Collected last (file name) so that it also runs after every other GPU test in one process; it must
pass on its own in a fresh process too.  Both entry points run the same stream-K tcgen05 kernel
with a fixed fix-up order, so they agree within the linear op's tolerance (and in practice
bitwise), on two calls in a row; each call is also held to the fp64 product of the bf16 operands,
and its status word must report no expired wait.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cs():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2510_26843_gb300 as m

    m.load_library()
    return m


def _rand_bf16(seed, shape, std):
    key = synth.stream_key(seed, 99)
    return synth.fill_normal_bf16(key, 0, int(np.prod(shape)), std).reshape(shape)


def _dev(bits):
    return torch.from_numpy(bits.view(np.int16).copy()).cuda()


@pytest.mark.parametrize("N,K,n", [(384, 256, 8), (1000, 688, 37), (4096, 4096, 64), (12288, 4096, 1)])
def test_static_matches_workspace_entry_point(cs, N, K, n):
    W = _rand_bf16(11, (N, K), 0.02)
    X = _rand_bf16(12, (n, K), 1.0)
    Wd, Xd = _dev(W), _dev(X)
    ws = torch.zeros(cs.linear_workspace_bytes(N, K, n), dtype=torch.uint8, device="cuda")
    ref = torch.full((n, N), float("nan"), dtype=torch.float32, device="cuda")
    cs.linear_bf16(Wd, N, K, Xd, n, ref, N, ws)
    Xf, Wf = synth.bf16_to_f32(X).astype(np.float64), synth.bf16_to_f32(W).astype(np.float64)
    scale = torch.from_numpy(np.abs(Xf) @ np.abs(Wf).T)
    exact = torch.from_numpy(Xf @ Wf.T)  # the fp64 product of the bf16 operands
    for _ in range(2):  # two calls in a row through the same static scratch
        got = torch.full((n, N), float("nan"), dtype=torch.float32, device="cuda")
        cs.linear_bf16_static(Wd, N, K, Xd, n, got, N)
        assert cs.linear_bf16_static_status() == 0  # no bounded wait expired
        torch.cuda.synchronize()
        g, r = got.cpu().double(), ref.cpu().double()
        assert torch.isfinite(g).all()
        assert float(((g - r).abs() / (scale + 1e-30)).max()) < 2e-4
        assert float(((g - exact).abs() / (scale + 1e-30)).max()) < 2e-4


def test_static_rejects_sizes_beyond_its_scratch(cs):
    K, n = 64, 4
    W = torch.zeros(40000, K, dtype=torch.int16, device="cuda")
    X = torch.zeros(n, K, dtype=torch.int16, device="cuda")
    Y = torch.zeros(n, 40000, dtype=torch.float32, device="cuda")
    with pytest.raises(cs.CasspecError) as e:
        cs.linear_bf16_static(W, 40000, K, X, n, Y, 40000)  # 313 output tiles > the static slots
    assert e.value.rc == cs.E_CAPACITY
    with pytest.raises(cs.CasspecError) as e:
        cs.linear_bf16_static(W, 128, K, X, 65, Y, 40000)
    assert e.value.rc == cs.E_SHAPE
