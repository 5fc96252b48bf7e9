"""The projection GEMM building block (tcgen05 / TMEM / TMA for bf16, SIMT
for fp32) against numpy fp64 matmul of the same bf16 operands, through the C
ABI (ravel_gemm).  Shapes cover single and multiple tiles, ragged token /
feature / K tails, split-K (partials exchanged through shared memory for token
slices of 4..32, through L2 for wider ones), persistent launches on one SM
or on SM pairs (one 256-row MMA per K step across two CTAs) and every
epilogue."""
import numpy as np
import pytest

import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def handles():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34170_gb300 import build, ravel_create, ravel_destroy
    build.build()
    hs = {}
    for dt in ("bf16", "fp32"):
        cfg = synth.ExpertConfig(layers=1, width=64, n_q_heads=1, n_kv_heads=1, head_dim=64, mlp_dim=64, slots=2,
                                 action_dim=2, prefix=1, fop_tokens=0, batch=1, dtype=dt)
        hs[dt] = ravel_create(cfg, synth.make_weights(cfg))
    yield hs
    for h in hs.values():
        ravel_destroy(h)


def _rand(shape, seed, scale=1.0):
    return synth.round_bf16(np.random.default_rng(seed).standard_normal(shape).astype(np.float32) * scale)


SHAPES = [(1, 128, 64), (7, 100, 200), (50, 2560, 1024), (66, 1024, 2048), (50, 1024, 4096), (130, 384, 192),
          (300, 256, 512), (3200, 1024, 1024), (51, 3000, 1024), (4224, 2560, 1024), (3200, 1024, 2048),
          (3200, 1024, 4096), (2900, 2048, 704)]


@pytest.mark.parametrize("M,N,K", SHAPES)
@pytest.mark.parametrize("epi", [0, 1, 2])
def test_gemm_bf16(handles, M, N, K, epi):
    from paper_2609_34170_gb300 import ravel_gemm
    X, W = _rand((M, K), 1), _rand((N, K), 2, 0.05)
    bias = np.random.default_rng(3).standard_normal(N).astype(np.float32)
    ref = X.astype(np.float64) @ W.astype(np.float64).T + bias
    dev = lambda a, dt=torch.bfloat16: torch.from_numpy(a).to("cuda", dt)  # noqa: E731
    init = np.random.default_rng(4).standard_normal((M, N)).astype(np.float32)
    out = dev(init, torch.float32)
    ravel_gemm(handles["bf16"], dev(X), dev(W), epi, out, dev(bias, torch.float32))
    got = out.cpu().numpy().astype(np.float64)
    if epi == 1:
        ref = ref / (1 + np.exp(-ref))
    if epi == 2:
        ref = ref + init
    scale = np.sqrt(K) * 0.05 + 1
    np.testing.assert_allclose(got, ref, rtol=1e-4, atol=1e-4 * scale)


@pytest.mark.parametrize("M,N,K", [(50, 256, 1024), (50, 8192, 1024), (66, 4096, 1024), (66, 8192, 1024),
                                   (300, 1024, 256), (3200, 2048, 1024), (3200, 8192, 1024)])
@pytest.mark.parametrize("with_bias", [False, True])
def test_gemm_geglu_bf16(handles, M, N, K, with_bias):
    from paper_2609_34170_gb300 import ravel_gemm
    X, W = _rand((M, K), 5), _rand((N, K), 6, 0.05)
    bias = np.random.default_rng(9).standard_normal(N).astype(np.float32) if with_bias else np.zeros(N, np.float32)
    ref_all = X.astype(np.float64) @ W.astype(np.float64).T + bias   # bias of each gate / up row, before GELU
    blocks = ref_all.reshape(M, N // 128, 2, 64)
    g, u = blocks[:, :, 0].reshape(M, N // 2), blocks[:, :, 1].reshape(M, N // 2)
    ref = 0.5 * g * (1 + np.tanh(np.sqrt(2 / np.pi) * (g + 0.044715 * g ** 3))) * u
    out = torch.zeros((M, N // 2), device="cuda", dtype=torch.bfloat16)
    ravel_gemm(handles["bf16"], torch.from_numpy(X).to("cuda", torch.bfloat16),
               torch.from_numpy(W).to("cuda", torch.bfloat16), 3, out,
               torch.from_numpy(bias).cuda() if with_bias else None)
    got = out.float().cpu().numpy()
    np.testing.assert_allclose(got, ref, rtol=1e-2, atol=1e-2 * (np.abs(ref).max() + 1e-3))


def test_gemm_bf16_output_and_determinism(handles):
    from paper_2609_34170_gb300 import ravel_gemm
    M, N, K = 50, 1024, 4096      # split-K across the grid
    X, W = _rand((M, K), 7), _rand((N, K), 8, 0.05)
    Xd, Wd = torch.from_numpy(X).to("cuda", torch.bfloat16), torch.from_numpy(W).to("cuda", torch.bfloat16)
    outs = []
    for _ in range(3):
        o = torch.zeros((M, N), device="cuda", dtype=torch.bfloat16)
        ravel_gemm(handles["bf16"], Xd, Wd, 0, o)
        outs.append(o)
    assert all(torch.equal(outs[0], o) for o in outs[1:])
    ref = X.astype(np.float64) @ W.astype(np.float64).T
    np.testing.assert_allclose(outs[0].float().cpu().numpy(), ref, rtol=1e-2, atol=1e-2)


def test_gemm_two_sm_is_deterministic(handles):
    # the persistent two-SM kernel: every launch gives the same bits
    from paper_2609_34170_gb300 import ravel_gemm
    M, N, K = 3200, 1024, 4096
    X, W = _rand((M, K), 11), _rand((N, K), 12, 0.05)
    Xd, Wd = torch.from_numpy(X).to("cuda", torch.bfloat16), torch.from_numpy(W).to("cuda", torch.bfloat16)
    outs = []
    for _ in range(3):
        o = torch.zeros((M, N), device="cuda", dtype=torch.float32)
        ravel_gemm(handles["bf16"], Xd, Wd, 0, o)
        outs.append(o)
    assert all(torch.equal(outs[0], o) for o in outs[1:])
    ref = X.astype(np.float64) @ W.astype(np.float64).T
    np.testing.assert_allclose(outs[0].cpu().numpy(), ref, rtol=1e-4, atol=1e-4 * (np.sqrt(K) * 0.05 + 1))


@pytest.mark.parametrize("M,N,K", [(10, 100, 256), (66, 300, 200)])
def test_gemm_fp32_simt(handles, M, N, K):
    from paper_2609_34170_gb300 import ravel_gemm
    rng = np.random.default_rng(9)
    X, W = rng.standard_normal((M, K)).astype(np.float32), rng.standard_normal((N, K)).astype(np.float32)
    out = torch.zeros((M, N), device="cuda")
    ravel_gemm(handles["fp32"], torch.from_numpy(X).cuda(), torch.from_numpy(W).cuda(), 0, out)
    np.testing.assert_allclose(out.cpu().numpy(), X.astype(np.float64) @ W.astype(np.float64).T, rtol=1e-5,
                               atol=1e-4)
