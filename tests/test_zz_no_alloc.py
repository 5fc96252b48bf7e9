"""The allocation-free GEMM entry point (ravel_gemm_noalloc), through the C ABI.

ravel_gemm_noalloc is for callers that cannot allocate device memory -- code
running inside another runtime's memory pool with raw allocation disabled,
plugin hosts that forbid cudaMalloc, control loops that must not touch the
allocator after start-up -- and so cannot create a handle (whose creation
allocates the split-K workspace).  Its split-K scratch is a fixed device array
inside the library that every call reuses.  This file checks:

* each shape twice in a row, against numpy fp64 of the same bf16 operands and
  against the handle-based ravel_gemm, with calls of different split plans
  (tile counts, split counts, no split) interleaved, so that a call that saw
  stale counters or partial sums of an earlier one would fail;
* that a bounded wait that runs out inside one of its GEMMs is reported by
  ravel_gemm_noalloc_status (and then cleared), not lost;
* that a first call on a capturing stream is refused without any set-up
  (checked in a fresh process, where no call has run yet);
* the size limits and argument checks.

The file is named so that pytest collects it last."""
import os
import subprocess
import sys

import numpy as np
import pytest

import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# (M, N, K, epi): split-K residual accumulate (8 tiles), split-K store (20
# tiles), fused GeGLU, many token tiles (no split), a ragged split plan, and
# the first plan again after the others
CASES = [(50, 1024, 4096, 2), (66, 2560, 1024, 0), (50, 8192, 1024, 3), (3200, 1024, 1024, 1),
         (130, 384, 192, 2), (50, 1024, 4096, 2)]


def _rand(shape, seed, scale=1.0):
    return synth.round_bf16(np.random.default_rng(seed).standard_normal(shape).astype(np.float32) * scale)


def _reference(X, W, bias, epi, init):
    """fp64 product of the bf16 operands with the epilogue applied on the host."""
    r = X.astype(np.float64) @ W.astype(np.float64).T + bias
    if epi == 1:
        return r / (1 + np.exp(-r))
    if epi == 2:
        return r + init
    if epi == 3:
        M, N = r.shape
        blocks = r.reshape(M, N // 128, 2, 64)
        g, u = blocks[:, :, 0].reshape(M, N // 2), blocks[:, :, 1].reshape(M, N // 2)
        return 0.5 * g * (1 + np.tanh(np.sqrt(2 / np.pi) * (g + 0.044715 * g ** 3))) * u
    return r


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34170_gb300 import build, load
    build.build()
    load()


def test_noalloc_first_call_under_capture_is_refused():
    # a fresh process: the first call on the device must not run its set-up
    # while the stream is being captured
    code = r"""
import torch, sys
sys.path.insert(0, %r)
from paper_2609_34170_gb300 import load
L = load()
X = torch.zeros((16, 64), device="cuda", dtype=torch.bfloat16)
W = torch.zeros((128, 64), device="cuda", dtype=torch.bfloat16)
out = torch.zeros((16, 128), device="cuda")
s = torch.cuda.Stream()
g = torch.cuda.CUDAGraph()
with torch.cuda.graph(g, stream=s):
    out.add_(1.0)
    st = L.ravel_gemm_noalloc(X.data_ptr(), 16, 64, 64, W.data_ptr(), 128, 64, 0, out.data_ptr(), 128, 0, None,
                              s.cuda_stream)
    st2 = L.ravel_gemm_noalloc_status(s.cuda_stream)
print("STATUS", st, st2)
""" % ROOT
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert "STATUS 1 1" in r.stdout, r.stdout + r.stderr[-2000:]


def test_noalloc_gemm_matches_fp64_and_handle_gemm_on_consecutive_calls():
    from paper_2609_34170_gb300 import (ravel_create, ravel_destroy, ravel_gemm, ravel_gemm_noalloc,
                                        ravel_gemm_noalloc_status)
    cfg = synth.ExpertConfig(layers=1, width=64, n_q_heads=1, n_kv_heads=1, head_dim=64, mlp_dim=64, slots=2,
                             action_dim=2, prefix=1, fop_tokens=0, batch=1, dtype="bf16")
    h = ravel_create(cfg, synth.make_weights(cfg))
    try:
        for i, (M, N, K, epi) in enumerate(CASES):
            Xh, Wh = _rand((M, K), 10 + i), _rand((N, K), 20 + i, 0.05)
            bias_h = _rand((N,), 30 + i)
            X = torch.from_numpy(Xh).to("cuda", torch.bfloat16)
            W = torch.from_numpy(Wh).to("cuda", torch.bfloat16)
            bias = torch.from_numpy(bias_h).cuda()
            if epi == 3:
                shape, dt, rtol = (M, N // 2), torch.bfloat16, 1e-2
            else:
                shape, dt, rtol = (M, N), torch.float32, 1e-4
            init_h = _rand(shape, 40 + i)
            init = torch.from_numpy(init_h).to("cuda", dt)
            want = _reference(Xh, Wh, bias_h, epi, init_h.astype(np.float64))
            ref = init.clone()
            ravel_gemm(h, X, W, epi, ref, bias)
            for call in range(2):
                out = init.clone()
                ravel_gemm_noalloc(X, W, epi, out, bias)
                torch.cuda.synchronize()
                r, o = ref.float().cpu().numpy(), out.float().cpu().numpy()
                tol = rtol * (np.abs(want).max() + 1e-3)
                np.testing.assert_allclose(o, want, rtol=rtol, atol=tol, err_msg=f"fp64 {(M, N, K, epi)} call {call}")
                np.testing.assert_allclose(o, r, rtol=rtol, atol=tol, err_msg=f"ravel_gemm {(M, N, K, epi)} call {call}")
        assert ravel_gemm_noalloc_status() == 0
    finally:
        ravel_destroy(h)


def test_noalloc_timeout_is_reported_not_lost():
    from paper_2609_34170_gb300 import (RAVEL_FAULT_WITHHOLD_ARRIVAL, ravel_debug_inject, ravel_gemm_noalloc,
                                        ravel_gemm_noalloc_status)
    M, N, K = 16, 128, 64                          # a single CTA without a cluster
    Xh, Wh = _rand((M, K), 1), _rand((N, K), 2, 0.05)
    X, W = torch.from_numpy(Xh).to("cuda", torch.bfloat16), torch.from_numpy(Wh).to("cuda", torch.bfloat16)
    out = torch.zeros((M, N), device="cuda")
    ravel_debug_inject(None, RAVEL_FAULT_WITHHOLD_ARRIVAL, 1)
    ravel_gemm_noalloc(X, W, 0, out)              # gives up after 2 ms
    assert ravel_gemm_noalloc_status() == 8       # RAVEL_ETIMEOUT, then cleared
    assert ravel_gemm_noalloc_status() == 0
    for _ in range(2):
        out.zero_()
        ravel_gemm_noalloc(X, W, 0, out)
        torch.cuda.synchronize()
        np.testing.assert_allclose(out.cpu().numpy(), Xh.astype(np.float64) @ Wh.astype(np.float64).T,
                                   rtol=1e-4, atol=1e-4)
    assert ravel_gemm_noalloc_status() == 0


def test_noalloc_gemm_rejects_oversized_and_bad_arguments():
    from paper_2609_34170_gb300 import load
    L = load()
    X = torch.zeros((8, 64), device="cuda", dtype=torch.bfloat16)
    out = torch.zeros((8, 128), device="cuda")
    p = X.data_ptr()
    # N above the stated maximum -> RAVEL_ESHAPE; K not a multiple of 8 -> RAVEL_EINVAL
    assert L.ravel_gemm_noalloc(p, 8, 64, 64, p, 262145, 64, 0, out.data_ptr(), 262145, 0, None, None) == 2
    assert L.ravel_gemm_noalloc(p, 8, 60, 64, p, 8, 64, 0, out.data_ptr(), 128, 0, None, None) == 1
    assert L.ravel_gemm_noalloc(None, 8, 64, 64, p, 8, 64, 0, out.data_ptr(), 128, 0, None, None) == 1
