"""A slot-time schedule per robot (ravel_config.per_robot_times), through the
C ABI, against the fp64 oracle.

Robots that run rolling inference at different rates or with different
schedules carry their own slot times t_bj: the conditioning (App. A.1), the
Euler step dt_bj (Eq. 3) and the relative shift (1 - t_bj) then follow each
robot's schedule.  Steps are held to the step tolerances of the oracle run
with the same [B, H] slot times.
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
                              action_dim=5, prefix=45, fop_tokens=3, batch=3, dtype=dtype, per_robot_times=1)


def _schedules(H, shift):
    base = (np.arange(H) + 1) / H
    tb = np.stack([base, base ** 2, np.sqrt(base)])
    return np.roll(tb, shift, axis=0).astype(np.float32)


def _session(case):
    from paper_2609_34170_gb300 import RollingSession
    s = RollingSession(case.cfg, case.W, 0, case.B, case.cfg.prefix)
    s.reset(case.seeds)
    s.set_context(case.k, case.v, case.P)
    return s


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("relative", [False, True])
def test_schedule_per_robot_matches_oracle(dtype, relative):
    cfg = _cfg(dtype)
    case = Case(cfg)
    s = _session(case)
    A = cfg.action_dim
    mask = np.array([1.0, 1.0, 0.0, 1.0, 1.0][:A], np.float32)
    if relative:
        s.set_relative_dims(mask)
    rng = np.random.default_rng(11)
    tol_a, tol_v = TOL[dtype]
    for step in range(3):
        tb = _schedules(cfg.slots, step)    # the robots trade schedules every step
        state = rng.standard_normal((case.B, A)).astype(np.float32) if relative else None
        buf0 = s.buffer.cpu().numpy().copy()
        cnt0 = np.asarray(s.counters(), np.uint64)
        s.step(tb, case.fop, case.delta, want_velocity=True, state=state)
        torch.cuda.synchronize()
        rel_o, new_o, cnt_o, vel_o = expert.roll_step(cfg, case.W, buf0, tb, case.k, case.v, case.P, case.fop,
                                                      case.delta, case.seeds, cnt0, state=state,
                                                      rel_mask=mask if relative else None)
        err_a = float(np.max(np.abs(s.released.cpu().numpy() - rel_o)))
        err_v = rel_l2(s.velocity.cpu().numpy(), vel_o)
        assert err_a <= tol_a, f"step {step}: released max-abs {err_a:.3e}"
        assert err_v <= tol_v, f"step {step}: velocity rel-L2 {err_v:.3e}"
        assert float(np.max(np.abs(s.buffer.cpu().numpy()[:, :-1] - new_o[:, :-1]))) <= tol_a
        np.testing.assert_array_equal(s.buffer.cpu().numpy()[:, -1], new_o[:, -1].astype(np.float32))
        np.testing.assert_array_equal(s.counters(), cnt_o)
    s.close()


def test_schedule_per_robot_denoise_chunk():
    # the full-horizon baseline ignores the schedules (one flow time per pass)
    # and must give the same chunk as the oracle's
    cfg = _cfg("bf16")
    case = Case(cfg)
    s = _session(case)
    cnt0 = s.counters()
    got = s.denoise_chunk(4, case.fop, case.delta).cpu().numpy()
    want, cnt1 = expert.denoise_chunk(cfg, case.W, case.seeds, cnt0, 4, case.k, case.v, case.P, case.fop, case.delta)
    assert float(np.max(np.abs(got - want))) <= TOL["bf16"][0]
    np.testing.assert_array_equal(s.counters(), cnt1)
    s.close()
