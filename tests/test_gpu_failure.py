"""Failure paths of the step, through the C ABI, without a GPU fault.

* A prefix length out of range in the device context state: the attention
  kernels refuse it (they compute nothing and raise the device error word) and
  a later call returns RAVEL_EDEVICE.
* A bounded mbarrier wait that runs out: a single-CTA GEMM launch waits for an
  arrival that nobody makes, gives up after 2 ms, drains its copies and exits;
  a later call returns RAVEL_ETIMEOUT.
Both faults are injected from the host (ravel_debug_inject); every wait
involved is bounded, and the handle stays usable after ravel_reset.
"""
import numpy as np
import pytest

import synth
from tests._harness import Case, check_step, gpu_session

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34170_gb300 import build, load
    build.build()
    load()


def _ragged(dtype):
    return synth.ExpertConfig(layers=2, width=192, n_q_heads=6, n_kv_heads=2, head_dim=40, mlp_dim=320, slots=7,
                              action_dim=5, prefix=45, fop_tokens=3, batch=2, dtype=dtype)


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_bad_prefix_length_surfaces_as_edevice(dtype):
    from paper_2609_34170_gb300 import RAVEL_FAULT_PREFIX_LEN, RavelError, ravel_debug_inject
    case = Case(_ragged(dtype))
    s = gpu_session(case)
    check_step(case, s, label="before the fault")
    ravel_debug_inject(s.handle, RAVEL_FAULT_PREFIX_LEN)
    s.step(case.t, case.fop, case.delta)          # enqueued; the kernels refuse the length
    torch.cuda.synchronize()
    with pytest.raises(RavelError) as ei:
        s.step(case.t, case.fop, case.delta)
    assert ei.value.status == 7                   # RAVEL_EDEVICE
    with pytest.raises(RavelError) as ei:
        s.counters()
    assert ei.value.status == 7
    # a reset clears the error word and a new context a valid state: parity again
    s.reset(case.seeds)
    s.set_context(case.k, case.v, case.P)
    check_step(case, s, label="after reset")
    s.close()


def _rand(shape, seed, scale=1.0):
    return synth.round_bf16(np.random.default_rng(seed).standard_normal(shape).astype(np.float32) * scale)


def test_withheld_arrival_times_out_and_surfaces_as_etimeout():
    from paper_2609_34170_gb300 import (RAVEL_FAULT_WITHHOLD_ARRIVAL, RavelError, ravel_create, ravel_debug_inject,
                                        ravel_destroy, ravel_gemm, ravel_reset)
    cfg = synth.ExpertConfig(layers=1, width=64, n_q_heads=1, n_kv_heads=1, head_dim=64, mlp_dim=64, slots=2,
                             action_dim=2, prefix=1, fop_tokens=0, batch=1, dtype="bf16")
    h = ravel_create(cfg, synth.make_weights(cfg))
    try:
        M, N, K = 16, 128, 64                      # one tile, one K block: a single CTA, no cluster
        X, W = _rand((M, K), 1), _rand((N, K), 2, 0.05)
        Xd, Wd = torch.from_numpy(X).to("cuda", torch.bfloat16), torch.from_numpy(W).to("cuda", torch.bfloat16)
        ref = X.astype(np.float64) @ W.astype(np.float64).T
        out = torch.zeros((M, N), device="cuda")
        ravel_debug_inject(h, RAVEL_FAULT_WITHHOLD_ARRIVAL, 1)
        ravel_gemm(h, Xd, Wd, 0, out)              # gives up after 2 ms
        torch.cuda.synchronize()
        with pytest.raises(RavelError) as ei:
            ravel_gemm(h, Xd, Wd, 0, out)
        assert ei.value.status == 8                # RAVEL_ETIMEOUT
        # the context is intact: after a reset the same GEMM is correct
        buf = torch.empty((1, cfg.slots, cfg.action_dim), device="cuda")
        ravel_reset(h, 1, synth.robot_seeds(1, 1), buf)
        out.zero_()
        ravel_gemm(h, Xd, Wd, 0, out)
        torch.cuda.synchronize()
        np.testing.assert_allclose(out.cpu().numpy(), ref, rtol=1e-4, atol=1e-4)
    finally:
        ravel_destroy(h)
