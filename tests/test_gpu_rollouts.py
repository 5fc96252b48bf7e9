"""GPU parity at the stress-grid corners and over rollouts, through the C ABI.

* Three corners of the batch x prefix x slots grid at the full pi0.5 width
  (B=256 P=2048 H=50; B=16 P=256 H=16; B=1 P=2048 H=16): one step, checked on
  sampled robots against the fp64 oracle (the step is independent per robot,
  so the other robots' prefixes are random values drawn on the device).
* The pi0.5-shaped batch-1 rollout with a new VLM context every 10 steps
  (Sec. 3.2: the latest context is reused until a new one arrives), 100 steps,
  teacher-forced against the oracle on the first step after each swap.
* Torn reads: two constant-valued contexts alternate, swapped in from a side
  stream while earlier steps are still queued; every step's released action
  must be the oracle's for the context set before it, never the other's.

Tolerances: released max-abs 5e-2 and velocity relative L2 2e-2 (bf16), the
appended Gaussian slot bit-exact.
"""
import numpy as np
import pytest

import synth
from oracle import expert
from tests._harness import TOL, rel_l2

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34170_gb300 import build, load
    build.build()
    load()


def _compare(cfg, W, buf0, cnt0, t, k, v, z, d, seeds, robots, rel, vel, buf1, label):
    tol_a, tol_v = TOL[cfg.dtype]
    for b in robots:
        rel_o, new_o, cnt_o, vel_o = expert.roll_step(cfg, W, buf0[b:b + 1], t, k[b], v[b], k[b].shape[3],
                                                      z[b:b + 1], d[b:b + 1], seeds[b:b + 1], cnt0[b:b + 1])
        err_a = float(np.max(np.abs(rel[b] - rel_o[0])))
        err_v = rel_l2(vel[b], vel_o[0])
        assert err_a <= tol_a, f"{label} robot {b}: released max-abs {err_a:.3e}"
        assert err_v <= tol_v, f"{label} robot {b}: velocity rel-L2 {err_v:.3e}"
        assert float(np.max(np.abs(buf1[b, :-1] - new_o[0, :-1]))) <= tol_a, label
        np.testing.assert_array_equal(buf1[b, -1], new_o[0, -1].astype(np.float32), err_msg=label)


@pytest.mark.parametrize("batch,prefix,slots,robots", [(256, 2048, 50, [0, 131, 255]), (16, 256, 16, [0, 9, 15]),
                                                       (1, 2048, 16, [0])])
def test_stress_grid_corner_sampled(batch, prefix, slots, robots):
    from paper_2609_34170_gb300 import RollingSession
    cfg = synth.PRESETS["pi05_bf16_b1"].replace(batch=batch, prefix=prefix, slots=slots)
    W = synth.make_weights(cfg, 0)
    s = RollingSession(cfg, W, 0)
    seeds = synth.robot_seeds(7, batch)
    s.reset(seeds)
    shape = (cfg.layers, batch, cfg.n_kv_heads, prefix, cfg.head_dim)
    gen = torch.Generator(device="cuda").manual_seed(5)
    kd = torch.randn(shape, generator=gen, device="cuda", dtype=torch.bfloat16)
    vd = torch.randn(shape, generator=gen, device="cuda", dtype=torch.bfloat16)
    k, v = {}, {}
    for b in robots:   # the sampled robots' prefixes come from the seeded host generator
        kb, vb = synth.make_context(cfg, 1000 + b, batch=1)
        kd[:, b] = torch.from_numpy(kb[:, 0]).to("cuda", torch.bfloat16)
        vd[:, b] = torch.from_numpy(vb[:, 0]).to("cuda", torch.bfloat16)
        k[b], v[b] = kb, vb
    s.set_context(kd, vd, prefix)
    z = synth.make_fop(cfg, 2000)
    t = synth.staggered_times(slots)
    d = synth.make_delta(batch, 2, slots)
    buf0 = s.buffer.cpu().numpy().copy()
    cnt0 = s.counters()
    s.step(t, z, d, want_velocity=True)
    torch.cuda.synchronize()
    _compare(cfg, W, buf0, cnt0, t, k, v, z, d, seeds, robots, s.released.cpu().numpy(), s.velocity.cpu().numpy(),
             s.buffer.cpu().numpy(), f"B{batch} P{prefix} H{slots}")
    s.close()
    del kd, vd
    torch.cuda.empty_cache()


def test_pi05_rollout_with_context_swaps_teacher_forced():
    from paper_2609_34170_gb300 import RollingSession
    cfg = synth.PRESETS["pi05_bf16_b1"]
    W = synth.make_weights(cfg, 0)
    s = RollingSession(cfg, W, 0)
    seeds = synth.robot_seeds(7, 1)
    s.reset(seeds)
    ctxs = [synth.make_context(cfg, cs) for cs in (1000, 5000, 9000)]
    dev = [(torch.from_numpy(a).to("cuda", torch.bfloat16), torch.from_numpy(b).to("cuda", torch.bfloat16))
           for a, b in ctxs]
    z = synth.make_fop(cfg, 2000)
    t = synth.staggered_times(cfg.slots)
    side = torch.cuda.Stream()
    s.set_context(*dev[0], cfg.prefix)
    checked = 0
    for step in range(100):
        age = 2 + step % 10
        d = synth.make_delta(1, age, cfg.slots)
        c = (step // 10) % 3
        if step % 10 == 0 and step > 0:
            s.set_context(*dev[c], cfg.prefix, side_stream=side)
        if step % 10 == 0 and step > 0 and checked < 4:   # the first step after each of the first swaps
            torch.cuda.synchronize()
            buf0, cnt0 = s.buffer.cpu().numpy().copy(), s.counters()
            s.step(t, z, d, want_velocity=True)
            torch.cuda.synchronize()
            _compare(cfg, W, buf0, cnt0, t, {0: ctxs[c][0]}, {0: ctxs[c][1]}, z, d, seeds, [0],
                     s.released.cpu().numpy(), s.velocity.cpu().numpy(), s.buffer.cpu().numpy(),
                     f"step {step} (context {c})")
            checked += 1
        else:
            s.step(t, z, d, want_velocity=True)
    torch.cuda.synchronize()
    assert checked == 4
    assert np.all(np.isfinite(s.buffer.cpu().numpy()))
    s.close()


def test_context_swaps_never_tear():
    from paper_2609_34170_gb300 import RollingSession, ravel_roll_step
    cfg = synth.ExpertConfig(layers=2, width=192, n_q_heads=6, n_kv_heads=2, head_dim=40, mlp_dim=320, slots=7,
                             action_dim=5, prefix=600, fop_tokens=3, batch=2, dtype="bf16")
    W = synth.make_weights(cfg, 0)
    s = RollingSession(cfg, W, 0)
    seeds = synth.robot_seeds(7, cfg.batch)
    s.reset(seeds)
    shape = (cfg.layers, cfg.batch, cfg.n_kv_heads, cfg.prefix, cfg.head_dim)
    # two constant-valued contexts: a step that read part of one and part of
    # the other would match neither oracle result
    consts = [(np.full(shape, 0.75, np.float32), np.full(shape, -1.5, np.float32)),
              (np.full(shape, -0.5, np.float32), np.full(shape, 2.0, np.float32))]
    dev = [(torch.from_numpy(a).to("cuda", torch.bfloat16), torch.from_numpy(b).to("cuda", torch.bfloat16))
           for a, b in consts]
    z = synth.make_fop(cfg, 2000)
    t = synth.staggered_times(cfg.slots)
    d = synth.make_delta(cfg.batch, 3, cfg.slots)
    zt, tt, dt = (torch.from_numpy(z).to("cuda", torch.bfloat16), torch.from_numpy(t).cuda(),
                  torch.from_numpy(d).cuda())
    side = torch.cuda.Stream()
    st = torch.cuda.current_stream()
    n = 24
    buf_hist = torch.empty((n,) + tuple(s.buffer.shape), device="cuda")
    rel_hist = torch.empty((n,) + tuple(s.released.shape), device="cuda")
    expect = []
    s.set_context(*dev[0], cfg.prefix)
    cur = 0
    for step in range(n):   # nothing synchronises the host inside this loop
        if step % 2 == 0 and step > 0:
            cur = 1 - cur
            s.set_context(*dev[cur], cfg.prefix, side_stream=side)
        expect.append(cur)
        buf_hist[step].copy_(s.buffer)
        ravel_roll_step(s.handle, s.buffer, tt, zt, dt, s.released, None, st)
        rel_hist[step].copy_(s.released)
    torch.cuda.synchronize()
    bh, rh = buf_hist.cpu().numpy(), rel_hist.cpu().numpy()
    cnt = np.full(cfg.batch, cfg.slots, np.uint64)
    tol = TOL["bf16"][0]
    for step in range(n):
        outs = []
        for c in (0, 1):
            k, v = consts[c]
            rel_o, _, _, _ = expert.roll_step(cfg, W, bh[step], t, k, v, cfg.prefix, z, d, seeds, cnt + step)
            outs.append(float(np.max(np.abs(rh[step] - rel_o))))
        want, other = outs[expect[step]], outs[1 - expect[step]]
        assert want <= tol, f"step {step}: {want:.3e} from the context it should have read"
        # ... and far from the other context's result (a torn read would sit
        # between the two, or away from both)
        assert other > 8 * want, f"step {step}: {other:.3e} from the other context vs {want:.3e}"
    s.close()
