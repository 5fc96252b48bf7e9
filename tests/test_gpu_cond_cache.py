"""The steady-state conditioning cache, through the C ABI.

In the paper's rolling schedule the slot flow times are the same every step
and the context age delta = p/K takes a handful of values (Sec. 3.1, App. A.1),
so the modulation rows of the conditioning are usually computed already; the
step then skips the embedding, the conditioning MLPs and the modulation GEMM
and reads cached rows.  The cache must be invisible in the results:

* a step served from the cache is bit-identical to the same step computed
  from scratch on a fresh handle;
* more distinct offsets than the cache holds, and changing slot times, stay
  within the step tolerances of the oracle at every step.
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


def _ragged(dtype, **kw):
    base = dict(layers=2, width=192, n_q_heads=6, n_kv_heads=2, head_dim=40, mlp_dim=320, slots=7,
                action_dim=5, prefix=45, fop_tokens=3, batch=3, dtype=dtype)
    base.update(kw)
    return synth.ExpertConfig(**base)


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_cached_step_is_bit_identical_to_a_cold_step(dtype):
    case = Case(_ragged(dtype))
    warm = gpu_session(case)
    for _ in range(3):                      # the conditioning rows are cached after the first step
        warm.step(case.t, case.fop, case.delta)
    buf = warm.buffer.clone()
    cnt = warm.counters()
    warm.step(case.t, case.fop, case.delta, want_velocity=True)
    torch.cuda.synchronize()
    cold = gpu_session(case)                # a fresh handle: nothing cached
    cold.buffer.copy_(buf)
    cold.set_counters(cnt)
    cold.step(case.t, case.fop, case.delta, want_velocity=True)
    torch.cuda.synchronize()
    assert torch.equal(warm.velocity, cold.velocity)
    assert torch.equal(warm.released, cold.released)
    assert torch.equal(warm.buffer, cold.buffer)
    warm.close()
    cold.close()


def test_many_offsets_and_changing_times_stay_exact():
    cfg = _ragged("bf16", batch=2)
    case = Case(cfg)
    s = gpu_session(case)
    rng = np.random.default_rng(3)
    for step in range(24):
        # 24 steps over 20 distinct ages per robot (more than the 16 cached
        # offsets), robots of different ages, and a different slot-time
        # schedule every 8 steps
        case.delta = synth.make_delta(cfg.batch, [step % 20, (step * 7) % 20], cfg.slots)
        if step % 8 == 0:
            t = np.sort(rng.uniform(0.05, 1.0, cfg.slots)).astype(np.float32)
            t[-1] = 1.0
            case.t = t
        check_step(case, s, label=f"step {step}")
    s.close()
