"""Per-kernel parity on the GPU, through the C ABI, against the CPU oracle (fp64 / fp32 spec)."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cs():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2510_26843_gb300 as m

    m.load_library()
    return m


def _bf16_dev(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda()


def _rand_bf16(seed: int, shape, std=1.0) -> np.ndarray:
    n = int(np.prod(shape))
    return synth.fill_normal_bf16(synth.stream_key(seed, 99, 0, hash(shape) & 0xFFFF), 0, n, std).reshape(shape)


LINEAR_SHAPES = [
    (384, 256, 8),      # several tiles, tiny K: every tile split across CTAs
    (1000, 688, 37),    # ragged N (last tile partial), ragged K (last k-block partial), ragged n
    (4096, 4096, 64),   # 7B Wo
    (12288, 4096, 1),   # 7B Wqkv, single token
    (4096, 11008, 16),  # 7B Wd
    (32000, 4096, 64),  # 7B LM head
]


@pytest.mark.parametrize("N,K,n", LINEAR_SHAPES)
def test_linear_bf16_matches_fp64(cs, N, K, n):
    W = _rand_bf16(1, (N, K), 0.02)
    X = _rand_bf16(2, (n, K), 1.0)
    ws = torch.zeros(cs.linear_workspace_bytes(N, K, n), dtype=torch.uint8, device="cuda")
    Y = torch.full((n, N), float("nan"), dtype=torch.float32, device="cuda")
    Wd, Xd = _bf16_dev(W), _bf16_dev(X)
    cs.linear_bf16(Wd, N, K, Xd, n, Y, N, ws)
    torch.cuda.synchronize()
    got = Y.cpu().numpy().astype(np.float64)
    ref = synth.bf16_to_f32(X).astype(np.float64) @ synth.bf16_to_f32(W).astype(np.float64).T
    # fp32 accumulation of exact bf16 products: error grows like sqrt(K) ulps of the partial sums
    scale = np.abs(synth.bf16_to_f32(X)).astype(np.float64) @ np.abs(synth.bf16_to_f32(W)).astype(np.float64).T
    assert np.all(np.isfinite(got))
    assert np.max(np.abs(got - ref) / (scale + 1e-30)) < 2e-4
    # deterministic: a second call gives the same bits, and the workspace counters are back to zero
    Y2 = torch.empty_like(Y)
    cs.linear_bf16(Wd, N, K, Xd, n, Y2, N, ws)
    torch.cuda.synchronize()
    assert torch.equal(Y, Y2)
    assert int(ws[:4096].sum()) == 0


def test_linear_bf16_rejects_bad_arguments(cs):
    ws = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    W = torch.zeros(128, 64, dtype=torch.int16, device="cuda")
    X = torch.zeros(4, 64, dtype=torch.int16, device="cuda")
    Y = torch.zeros(4, 128, dtype=torch.float32, device="cuda")
    with pytest.raises(cs.CasspecError) as e:
        cs.linear_bf16(W, 128, 64, X, 65, Y, 128, ws)
    assert e.value.rc == cs.E_SHAPE
    with pytest.raises(cs.CasspecError) as e:
        cs.linear_bf16(W, 128, 60, X, 4, Y, 128, ws)  # K % 8 != 0
    assert e.value.rc == cs.E_SHAPE
    small = torch.zeros(16, dtype=torch.uint8, device="cuda")
    with pytest.raises(cs.CasspecError) as e:
        cs.linear_bf16(W, 128, 64, X, 4, Y, 128, small)
    assert e.value.rc == cs.E_CAPACITY


@pytest.mark.parametrize("n,d", [(1, 256), (7, 4096), (64, 5120), (3, 11008)])
def test_rmsnorm_and_quant_match_oracle(cs, n, d):
    rng = np.random.default_rng(n * 1000 + d)
    x = (rng.standard_normal((n, d)) * rng.uniform(0.1, 30, (n, 1))).astype(np.float32)
    x[0, :5] = [1e-3, 0, -4, 7.5, 2]
    g = rng.uniform(0.5, 1.5, d).astype(np.float32)
    xd, gd = torch.from_numpy(x).cuda(), torch.from_numpy(g).cuda()
    y = torch.empty(n, d, dtype=torch.int16, device="cuda")
    q = torch.empty(n, d, dtype=torch.int8, device="cuda")
    s = torch.empty(n, dtype=torch.float32, device="cuda")
    cs.rmsnorm(xd, gd, n, d, 1e-5, y, q, s)
    torch.cuda.synchronize()
    yb = synth.bf16_to_f32(y.cpu().numpy().view(np.uint16))
    ref = oracle.rmsnorm(x.astype(np.float64), g, 1e-5)
    # bf16 output: within one bf16 rounding (2^-8 relative) of the fp64 normalised value
    assert np.max(np.abs(yb - ref) / (np.abs(ref) + 1e-30)) <= 2.0 ** -8 + 1e-6
    # the quantisation of the GPU's own bf16 rows is bit-exact (codes and scales)
    q_ref, s_ref = oracle.quantize_rows_f32(yb)
    assert np.array_equal(q.cpu().numpy(), q_ref)
    assert np.array_equal(s.cpu().numpy(), s_ref)


def test_quantize_rows_bit_exact_including_golden_rows(cs):
    rows = []
    for line in open("tests/golden/quant_rows.txt"):
        if line.startswith("#") or not line.strip():
            continue
        rows.append([float(v) for v in line.split("|")[0].split()])
    width = 16
    x = np.zeros((len(rows) + 40, width), dtype=np.float32)
    for i, r in enumerate(rows):
        x[i, :len(r)] = r
    rng = np.random.default_rng(5)
    x[len(rows):] = rng.standard_normal((40, width)) * 3
    bits = synth.bf16_bits_rne(x)
    xb = synth.bf16_to_f32(bits)
    q = torch.empty(x.shape, dtype=torch.int8, device="cuda")
    s = torch.empty(x.shape[0], dtype=torch.float32, device="cuda")
    cs.quantize_rows(_bf16_dev(bits), x.shape[0], width, q, s)
    torch.cuda.synchronize()
    q_ref, s_ref = oracle.quantize_rows_f32(xb)
    assert np.array_equal(q.cpu().numpy(), q_ref)
    assert np.array_equal(s.cpu().numpy(), s_ref)


def test_quantize_rows4_bit_exact(cs):
    """W4A4 activation codes (App. C): the int4 rule on bf16 rows, bit-exact against the oracle's
    fp32 rule with qmax 7, including rows with exact .5 ties and a zero row."""
    width = 32
    rng = np.random.default_rng(9)
    x = (rng.standard_normal((48, width)) * rng.uniform(0.1, 20, (48, 1))).astype(np.float32)
    x[0, :6] = [7, 3.5, -3.5, 0.5, -0.5, 2.5]  # amax 7: the codes are x itself, ties to even
    x[1, :] = 0.0
    bits = synth.bf16_bits_rne(x)
    xb = synth.bf16_to_f32(bits)
    q4 = torch.empty(x.shape[0], width // 2, dtype=torch.uint8, device="cuda")
    s = torch.empty(x.shape[0], dtype=torch.float32, device="cuda")
    cs.quantize_rows4(_bf16_dev(bits), x.shape[0], width, q4, s)
    torch.cuda.synchronize()
    q_ref, s_ref = oracle.quantize_rows_f32(xb, 7)
    assert np.array_equal(cs.unpack_int4(q4.cpu().numpy(), width), q_ref)
    assert np.array_equal(s.cpu().numpy(), s_ref)
