"""GPU parity of the rolling step in relative coordinates (ravel_roll_step_rel).

The expert predicts actions relative to the latest robot state while the
buffer keeps absolute targets (App. "LIBERO and RoboTwin 2.0", and the same
conversion for DynamicVLA's relative pose / absolute gripper actions): the
step converts each slot to relative coordinates at its flow time, runs the
expert and the Euler update there, and converts back at the slot's new time.
Checked teacher-forced against the oracle with a different robot state at
every step, a mask with an absolute (gripper) dimension, and h = 2 actions per
slot (the slot vector is two robot actions, the mask repeated).
"""
import numpy as np
import pytest

import synth
from oracle import expert
from tests._harness import TOL, Case, gpu_session, rel_l2

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34170_gb300 import build, load
    build.build()
    load()


@pytest.mark.parametrize("dtype,h", [("fp32", 1), ("bf16", 1), ("bf16", 2)])
def test_relative_step_matches_oracle(dtype, h):
    a_robot = 3
    cfg = synth.ExpertConfig(layers=2, width=192, n_q_heads=6, n_kv_heads=2, head_dim=40, mlp_dim=320, slots=7,
                             action_dim=a_robot * h, prefix=45, fop_tokens=3, batch=3, dtype=dtype)
    case = Case(cfg)
    s = gpu_session(case)
    mask = np.tile(np.array([1.0, 1.0, 0.0], np.float32), h)      # two relative dims, an absolute gripper
    s.set_relative_dims(mask)
    rng = np.random.default_rng(5)
    tol_a, tol_v = TOL[dtype]
    for step in range(4):
        state = (rng.standard_normal((cfg.batch, cfg.action_dim)) * 2.0).astype(np.float32)
        buf0, cnt0 = s.buffer.cpu().numpy().copy(), s.counters()
        s.step(case.t, case.fop, case.delta, want_velocity=True, state=state)
        torch.cuda.synchronize()
        rel, new, cnt, vel = expert.roll_step(cfg, case.W, buf0, case.t, case.k, case.v, case.P, case.fop, case.delta,
                                              case.seeds, cnt0, state=state, rel_mask=mask)
        err_a = float(np.max(np.abs(s.released.cpu().numpy() - rel)))
        assert err_a <= tol_a, f"step {step}: released max-abs {err_a:.3e}"
        assert rel_l2(s.velocity.cpu().numpy(), vel) <= tol_v
        got = s.buffer.cpu().numpy()
        assert float(np.max(np.abs(got[:, :-1] - new[:, :-1]))) <= tol_a
        np.testing.assert_array_equal(got[:, -1], new[:, -1].astype(np.float32))
        np.testing.assert_array_equal(s.counters(), cnt)
    s.close()
