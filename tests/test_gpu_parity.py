"""GPU parity of the rolling step against the fp64 oracle, through the C ABI.

Tolerances (fixed for the step): fp32 mode released max-abs <= 1e-4 and
velocity relative L2 <= 1e-4; bf16 mode 5e-2 and 2e-2; the appended Gaussian
slot bit-exact in both modes.
"""
import numpy as np
import pytest

import synth
from oracle import expert, noise
from tests._harness import TOL, Case, check_step, gpu_session, oracle_step, rel_l2

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


def test_reset_noise_bit_exact_over_a_million_draws():
    cfg = synth.ExpertConfig(layers=1, width=64, n_q_heads=1, n_kv_heads=1, head_dim=64, mlp_dim=64, slots=50,
                             action_dim=31, prefix=1, fop_tokens=0, batch=700, dtype="fp32")
    seeds = np.array([(b * 0x9E3779B97F4A7C15 + 17) % 2 ** 64 for b in range(cfg.batch)], dtype=np.uint64)
    from paper_2609_34170_gb300 import RollingSession
    s = RollingSession(cfg, synth.make_weights(cfg), 0)
    s.reset(seeds)
    got = s.buffer.cpu().numpy()
    want, cnt = expert.reset(cfg, seeds)
    assert got.size >= 10 ** 6
    np.testing.assert_array_equal(got, want)
    np.testing.assert_array_equal(s.counters(), cnt)
    s.close()


def test_tiny_fp32_single_step_and_rollout():
    cfg = synth.PRESETS["tiny_fp32_b1"]
    case = Case(cfg)
    s = gpu_session(case)
    for i in range(21):   # one step plus a 20-step rollout, teacher-forced
        check_step(case, s, label=f"step {i}")
    s.close()


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_ragged_shapes(dtype):
    cfg = _ragged(dtype)
    case = Case(cfg, prefix_len=37)           # prefix shorter than the slot capacity
    s = gpu_session(case, max_batch=4, max_prefix=cfg.prefix)
    for i in range(3):
        check_step(case, s, label=f"{dtype} step {i}")
    s.close()


# Key chunks split over a thread-block cluster (2, 4, 16 splits; one and two
# query tiles; two robots), with a partial last prefix chunk, and a prefix
# shorter than the slot capacity so that some splits get no key at all; and
# head dims that are not a multiple of 64.
SPLIT_KV = [
    (dict(layers=2, width=256, n_q_heads=4, n_kv_heads=1, head_dim=64, mlp_dim=512, slots=20, action_dim=7,
          prefix=300, fop_tokens=5, batch=1), None),
    (dict(layers=2, width=256, n_q_heads=4, n_kv_heads=2, head_dim=128, mlp_dim=512, slots=12, action_dim=5,
          prefix=700, fop_tokens=4, batch=1), None),
    (dict(layers=1, width=256, n_q_heads=2, n_kv_heads=1, head_dim=128, mlp_dim=256, slots=12, action_dim=5,
          prefix=2000, fop_tokens=3, batch=1), 1500),
    (dict(layers=1, width=256, n_q_heads=8, n_kv_heads=2, head_dim=64, mlp_dim=256, slots=40, action_dim=6,
          prefix=500, fop_tokens=8, batch=2), None),
    # head dims that end inside a 64-wide block: P V reads V as an MN-major
    # operand whose second block is partial (96 = 64 + 32 split, 80 = 64 + 16
    # over 64 robots, whose query tiles are not split)
    (dict(layers=1, width=192, n_q_heads=4, n_kv_heads=2, head_dim=96, mlp_dim=256, slots=10, action_dim=5,
          prefix=260, fop_tokens=3, batch=1), None),
    (dict(layers=1, width=160, n_q_heads=2, n_kv_heads=1, head_dim=80, mlp_dim=256, slots=9, action_dim=4,
          prefix=130, fop_tokens=2, batch=64), None),
]


@pytest.mark.parametrize("kw,prefix_len", SPLIT_KV)
def test_split_kv_attention(kw, prefix_len):
    cfg = synth.ExpertConfig(**kw, dtype="bf16")
    case = Case(cfg, prefix_len=prefix_len)
    s = gpu_session(case)
    for i in range(2):
        check_step(case, s, label=f"split-kv step {i}")
    s.close()


def test_slot_isolated_mask():
    cfg = _ragged("fp32", batch=2)
    case = Case(cfg)
    s = gpu_session(case, mask_mode=1)
    check_step(case, s, mask="slot_isolated")
    s.close()


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_no_fop_tokens(dtype):
    cfg = _ragged(dtype, fop_tokens=0, batch=2)
    case = Case(cfg)
    s = gpu_session(case)
    check_step(case, s)
    s.close()


def test_context_swap_and_errors():
    from paper_2609_34170_gb300 import RavelError, RollingSession
    cfg = _ragged("fp32", batch=2)
    a = Case(cfg)
    b = Case(cfg, ctx_seed=555, prefix_len=20)
    s = RollingSession(cfg, a.W, 0, 2, cfg.prefix)
    s.reset(a.seeds)
    with pytest.raises(RavelError) as ei:
        s.step(a.t, a.fop, a.delta)
    assert ei.value.status == 5                   # no context yet
    with pytest.raises(RavelError) as ei:
        s.set_context(a.k, a.v, cfg.prefix + 1)
    assert ei.value.status == 2                   # prefix too long
    s.set_context(a.k, a.v, a.P)
    with pytest.raises(RavelError) as ei:
        s.set_context(b.k, b.v, b.P)
    assert ei.value.status == 6                   # previous swap still pending
    check_step(a, s, label="context A")
    side = torch.cuda.Stream()
    s.set_context(b.k, b.v, b.P, side_stream=side)   # swapped in from a side stream
    check_step(b, s, label="context B")
    check_step(b, s, label="context B reused")
    s.close()


def test_state_resume_is_bit_exact():
    cfg = _ragged("bf16", batch=2)
    case = Case(cfg)
    s = gpu_session(case)
    for _ in range(3):
        s.step(case.t, case.fop, case.delta)
    saved_buf, saved_cnt = s.buffer.clone(), s.counters()
    outs = [s.step(case.t, case.fop, case.delta).clone() for _ in range(4)]
    s.buffer.copy_(saved_buf)
    s.set_counters(saved_cnt)
    again = [s.step(case.t, case.fop, case.delta).clone() for _ in range(4)]
    for x, y in zip(outs, again):
        assert torch.equal(x, y)
    s.close()


@pytest.mark.parametrize("name,robots", [("pi05_bf16_b1", [0]), ("pi05_bf16_b64", [0, 37, 63]),
                                         ("wide_bf16_b8", [0, 5, 7])])
def test_full_size_configs_sampled(name, robots):
    cfg = synth.PRESETS[name]
    case = Case(cfg)
    s = gpu_session(case)
    check_step(case, s, robots=robots, label=name)
    s.close()
