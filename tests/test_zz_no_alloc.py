"""The allocation-free GEMM entry point (ravel_gemm_noalloc) against the
handle-based one (ravel_gemm), through the C ABI.

ravel_gemm_noalloc exists for callers that cannot allocate device memory and
so cannot create a handle (whose creation allocates the split-K workspace).
Its split-K scratch is a fixed device array inside the library that every
call reuses, so this test calls it twice in a row on each shape and checks
that both calls agree with ravel_gemm within the GEMM tests' tolerances:
the second call must not see stale counters or partial sums from the first.
The file is named so that pytest collects it last."""
import numpy as np
import pytest

import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

# (M, N, K, epi): split-K residual accumulate, split-K store, fused GeGLU,
# many token tiles (no split) -- the plans that touch the scratch differently
CASES = [(50, 1024, 4096, 2), (66, 2560, 1024, 0), (50, 8192, 1024, 3), (3200, 1024, 1024, 1)]


def _rand(shape, seed, scale=1.0):
    return synth.round_bf16(np.random.default_rng(seed).standard_normal(shape).astype(np.float32) * scale)


def test_noalloc_gemm_matches_handle_gemm_on_consecutive_calls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34170_gb300 import build, ravel_create, ravel_destroy, ravel_gemm, ravel_gemm_noalloc
    build.build()
    cfg = synth.ExpertConfig(layers=1, width=64, n_q_heads=1, n_kv_heads=1, head_dim=64, mlp_dim=64, slots=2,
                             action_dim=2, prefix=1, fop_tokens=0, batch=1, dtype="bf16")
    h = ravel_create(cfg, synth.make_weights(cfg))
    try:
        for i, (M, N, K, epi) in enumerate(CASES):
            X = torch.from_numpy(_rand((M, K), 10 + i)).to("cuda", torch.bfloat16)
            W = torch.from_numpy(_rand((N, K), 20 + i, 0.05)).to("cuda", torch.bfloat16)
            bias = torch.from_numpy(_rand((N,), 30 + i)).cuda()
            if epi == 3:
                shape, dt, rtol = (M, N // 2), torch.bfloat16, 1e-2
            else:
                shape, dt, rtol = (M, N), torch.float32, 1e-4
            init = torch.from_numpy(_rand(shape, 40 + i)).to("cuda", dt)
            ref = init.clone()
            ravel_gemm(h, X, W, epi, ref, bias)
            for call in range(2):
                out = init.clone()
                ravel_gemm_noalloc(X, W, epi, out, bias)
                torch.cuda.synchronize()
                r, o = ref.float().cpu().numpy(), out.float().cpu().numpy()
                np.testing.assert_allclose(o, r, rtol=rtol, atol=rtol * (np.abs(r).max() + 1e-3),
                                           err_msg=f"case {(M, N, K, epi)} call {call}")
    finally:
        ravel_destroy(h)


def test_noalloc_gemm_rejects_oversized_and_bad_arguments():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34170_gb300 import build, load
    build.build()
    L = load()
    X = torch.zeros((8, 64), device="cuda", dtype=torch.bfloat16)
    out = torch.zeros((8, 128), device="cuda")
    p = X.data_ptr()
    # N above the stated maximum -> RAVEL_ESHAPE; K not a multiple of 8 -> RAVEL_EINVAL
    assert L.ravel_gemm_noalloc(p, 8, 64, 64, p, 262145, 64, 0, out.data_ptr(), 262145, 0, None, None) == 2
    assert L.ravel_gemm_noalloc(p, 8, 60, 64, p, 8, 64, 0, out.data_ptr(), 128, 0, None, None) == 1
    assert L.ravel_gemm_noalloc(None, 8, 64, 64, p, 8, 64, 0, out.data_ptr(), 128, 0, None, None) == 1
