"""casspec_topk (K-best candidates per logit row for tree expansion, Sec. 4.2) against the oracle:
token ids exact (lower id first on ties), probabilities within 1e-5 relative."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cs():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2510_26843_gb300 as m

    m.load_library()
    return m


def _run(cs, x, K):
    n, V = x.shape
    xd = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).cuda()
    idx = torch.full((n, K), -7, dtype=torch.int32, device="cuda")
    prob = torch.full((n, K), -1.0, dtype=torch.float32, device="cuda")
    cs.topk(xd, n, V, K, idx, prob)
    torch.cuda.synchronize()
    return idx.cpu().numpy(), prob.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("n,V,K", [(64, 32000, 8), (64, 32000, 1), (7, 1024, 4), (3, 257, 8), (1, 5, 8)])
def test_topk_matches_oracle(cs, n, V, K):
    rng = np.random.default_rng(n * 1000 + V + K)
    x = rng.normal(0.0, 3.0, (n, V)).astype(np.float32)
    if V > 10:
        x[0, 5] = x[0, 9] = x[0, 2] = x[0].max() + 0.5  # a three-way tie at the top
    idx, prob = _run(cs, x, K)
    ref_i, ref_p = oracle.topk_softmax(x.astype(np.float64), K)
    kk = ref_i.shape[1]
    assert (idx[:, :kk] == ref_i).all()
    assert np.allclose(prob[:, :kk], ref_p, rtol=1e-5, atol=0)
    if kk < K:
        assert (idx[:, kk:] == -1).all() and (prob[:, kk:] == 0).all()
    if V > 10:
        assert list(idx[0, :3]) == [2, 5, 9][: min(3, K)] or K < 3


def test_topk_rejects_bad_arguments(cs):
    x = torch.zeros(2, 16, device="cuda")
    i = torch.zeros(2, 8, dtype=torch.int32, device="cuda")
    p = torch.zeros(2, 8, device="cuda")
    for n, V, K in [(0, 16, 4), (2, 0, 4), (2, 16, 0), (2, 16, 9)]:
        with pytest.raises(cs.CasspecError):
            cs.topk(x, n, V, K, i, p)
