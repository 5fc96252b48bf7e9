"""Per-robot context swaps through the C ABI (ravel_set_context_robots).

In the paper every robot's VLM context is refreshed asynchronously, whenever
its own VLM pass completes (Method, "Asynchronous Context Updates"): robots
then run with contexts of different ages and lengths.  The library keeps a
double-buffered context per robot; a swap for some robots leaves the others'
contexts untouched.  Each step is held to the step tolerances of the oracle
run with every robot's own context and prefix length.
"""
import numpy as np
import pytest

import synth
from oracle import expert
from tests._harness import TOL, Case, rel_l2

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34170_gb300 import build, load
    build.build()
    load()


def _cfg(dtype):
    return synth.ExpertConfig(layers=2, width=192, n_q_heads=6, n_kv_heads=2, head_dim=40, mlp_dim=320, slots=7,
                              action_dim=5, prefix=45, fop_tokens=3, batch=3, dtype=dtype)


class _Contexts:
    """The oracle's view: every robot's current K/V rows and prefix length."""

    def __init__(self, cfg, k, v, P):
        L, B, Hkv, _, hd = k.shape
        self.k = np.zeros((L, B, Hkv, cfg.prefix, hd), k.dtype)
        self.v = np.zeros_like(self.k)
        self.P = np.zeros(B, np.int64)
        self.install(list(range(B)), k, v, P)

    def install(self, robots, k, v, P):
        for i, b in enumerate(robots):
            self.k[:, b] = 0
            self.v[:, b] = 0
            self.k[:, b, :, :P] = k[:, i, :, :P]
            self.v[:, b, :, :P] = v[:, i, :, :P]
            self.P[b] = P


def _step_and_check(case, s, ctx, label):
    buf0 = s.buffer.cpu().numpy().copy()
    cnt0 = np.asarray(s.counters(), np.uint64)
    s.step(case.t, case.fop, case.delta, want_velocity=True)
    torch.cuda.synchronize()
    rel_o, new_o, cnt_o, vel_o = expert.roll_step(case.cfg, case.W, buf0, case.t, ctx.k, ctx.v, ctx.P, case.fop,
                                                  case.delta, case.seeds, cnt0)
    tol_a, tol_v = TOL[case.cfg.dtype]
    err_a = float(np.max(np.abs(s.released.cpu().numpy() - rel_o)))
    err_v = rel_l2(s.velocity.cpu().numpy(), vel_o)
    assert err_a <= tol_a, f"{label}: released max-abs {err_a:.3e}"
    assert err_v <= tol_v, f"{label}: velocity rel-L2 {err_v:.3e}"
    np.testing.assert_array_equal(s.counters(), cnt_o)
    return vel_o


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_some_robots_swap_while_the_others_keep_their_context(dtype):
    from paper_2609_34170_gb300 import RollingSession
    cfg = _cfg(dtype)
    case = Case(cfg)
    s = RollingSession(cfg, case.W, 0, cfg.batch, cfg.prefix)
    s.reset(case.seeds)
    s.set_context(case.k, case.v, case.P)
    ctx = _Contexts(cfg, case.k, case.v, case.P)
    _step_and_check(case, s, ctx, "all robots, context A")
    # robots 0 and 2 receive context B (shorter), robot 1 keeps A
    kb, vb = synth.make_context(cfg, 3000, 2, 30)
    s.set_context_robots([2, 0], kb, vb, 30)
    ctx.install([2, 0], kb, vb, 30)
    _step_and_check(case, s, ctx, "robots 0, 2 on B")
    # robot 1 receives context C (much shorter); 0 and 2 keep B
    kc, vc = synth.make_context(cfg, 4000, 1, 12)
    s.set_context_robots([1], kc, vc, 12)
    ctx.install([1], kc, vc, 12)
    _step_and_check(case, s, ctx, "robot 1 on C")
    # and a step with no swap reuses every robot's context
    _step_and_check(case, s, ctx, "no swap")
    s.close()


def test_per_robot_swap_rules():
    from paper_2609_34170_gb300 import RavelError, RollingSession
    cfg = _cfg("bf16")
    case = Case(cfg)
    s = RollingSession(cfg, case.W, 0, cfg.batch, cfg.prefix)
    s.reset(case.seeds)
    # robots 0 and 1 only: a step needs every robot's context
    kb, vb = synth.make_context(cfg, 3000, 2, 20)
    s.set_context_robots([0, 1], kb, vb, 20)
    with pytest.raises(RavelError, match="ENOCONTEXT"):
        s.step(case.t, case.fop, case.delta)
    kc, vc = synth.make_context(cfg, 4000, 1, 20)
    s.set_context_robots([2], kc, vc, 20)
    # robot 0's swap is still pending: a second one for it is refused
    with pytest.raises(RavelError, match="EBUSY"):
        s.set_context_robots([0], kc, vc, 20)
    with pytest.raises(RavelError, match="EINVAL"):
        s.set_context_robots([1, 1], kb, vb, 20)
    with pytest.raises(RavelError, match="EINVAL"):
        s.set_context_robots([3], kc, vc, 20)
    ctx = _Contexts(cfg, case.k, case.v, case.P)   # replaced below
    ctx.install([0, 1], kb, vb, 20)
    ctx.install([2], kc, vc, 20)
    _step_and_check(case, s, ctx, "contexts assembled from two calls")
    s.close()
