"""GPU parity of the full-horizon (synchronous) denoising baseline against the
fp64 oracle, through the C ABI (ravel_denoise_chunk).

The paper compares rolling inference with ten full-horizon denoising steps
per policy query (Experiments, synchronous simulation; Table 1).  The chunk
is the result of n_steps dependent expert passes, so it is held to the
released-action tolerance of the step (max-abs 1e-4 fp32, 5e-2 bf16); the
fresh chunk noise (before any pass) is bit-exact.
"""
import numpy as np
import pytest

import synth
from oracle import expert, noise
from tests._harness import TOL, Case

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34170_gb300 import build, load
    build.build()
    load()


def _session(case):
    from paper_2609_34170_gb300 import RollingSession
    s = RollingSession(case.cfg, case.W, 0)
    s.reset(case.seeds)
    s.set_context(case.k, case.v, case.P)
    return s


def _check_chunk(case, s, n_steps, robots=None, label=""):
    cnt0 = s.counters()
    got = s.denoise_chunk(n_steps, case.fop, case.delta).cpu().numpy()
    rob = np.arange(case.B) if robots is None else np.asarray(robots)
    want, cnt1 = expert.denoise_chunk(case.cfg, case.W, case.seeds[rob], cnt0[rob], n_steps, case.k[:, rob],
                                      case.v[:, rob], case.P, case.fop[rob], case.delta[rob])
    err = float(np.max(np.abs(got[rob] - want)))
    assert err <= TOL[case.cfg.dtype][0], f"{label} chunk max-abs {err:.3e}"
    np.testing.assert_array_equal(s.counters()[rob], cnt1)
    return err


@pytest.mark.parametrize("name,kw", [("tiny_fp32_b1", {}),
                                     ("ragged_bf16", dict(layers=2, width=192, n_q_heads=6, n_kv_heads=2, head_dim=40,
                                                          mlp_dim=320, slots=7, action_dim=5, prefix=45, fop_tokens=3,
                                                          batch=3, dtype="bf16"))])
def test_denoise_chunk_matches_oracle(name, kw):
    cfg = synth.PRESETS[name] if name in synth.PRESETS else synth.ExpertConfig(**kw)
    case = Case(cfg)
    s = _session(case)
    for n_steps in (1, 10):
        _check_chunk(case, s, n_steps, label=f"{name} n={n_steps}")
    # rolling steps continue from the advanced counters
    from tests._harness import check_step
    check_step(case, s, label="roll after chunks")
    s.close()


def test_denoise_chunk_noise_is_the_next_h_actions():
    # zero velocity head (out_w = out_b = 0): the chunk stays its fresh noise
    cfg = synth.ExpertConfig(layers=1, width=64, n_q_heads=2, n_kv_heads=1, head_dim=32, mlp_dim=128, slots=6,
                             action_dim=9, prefix=10, fop_tokens=2, batch=2, dtype="bf16")
    case = Case(cfg)
    case.W = dict(case.W, out_w=np.zeros_like(case.W["out_w"]), out_b=np.zeros_like(case.W["out_b"]))
    s = _session(case)
    cnt0 = s.counters()
    got = s.denoise_chunk(10, case.fop, case.delta).cpu().numpy()
    for b in range(2):
        want = noise.action_noise(int(case.seeds[b]), cnt0[b] + np.arange(cfg.slots, dtype=np.uint64), cfg.action_dim)
        np.testing.assert_array_equal(got[b], want)
    s.close()


def test_denoise_chunk_pi05_b1():
    case = Case(synth.PRESETS["pi05_bf16_b1"])
    s = _session(case)
    _check_chunk(case, s, 10, label="pi05 b1 n=10")
    s.close()
