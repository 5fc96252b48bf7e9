"""Shared test helpers: run the CUDA path (through the C ABI) and the fp64
oracle on the same seeded inputs and compare them."""
from __future__ import annotations

import numpy as np

import synth
from oracle import expert

# tolerances of the rolling step (released actions max-abs, velocity relative L2)
TOL = {"fp32": (1e-4, 1e-4), "bf16": (5e-2, 2e-2)}


def rel_l2(a, b) -> float:
    a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))


class Case:
    """Seeded inputs of one configuration."""

    def __init__(self, cfg, weight_seed=0, ctx_seed=1000, fop_seed=2000, noise_seed=7, prefix_len=None,
                 age=2, batch=None):
        self.cfg = cfg
        self.B = cfg.batch if batch is None else batch
        self.W = synth.make_weights(cfg, weight_seed)
        self.P = cfg.prefix if prefix_len is None else prefix_len
        self.k, self.v = synth.make_context(cfg, ctx_seed, self.B, self.P)
        self.fop = synth.make_fop(cfg, fop_seed, self.B)
        self.t = synth.staggered_times(cfg.slots)
        self.delta = synth.make_delta(self.B, age, cfg.slots)
        self.seeds = synth.robot_seeds(noise_seed, self.B)


def oracle_step(case: Case, buffer, counters, robots=None, mask="full", k=None, v=None, fop=None, delta=None):
    """Oracle roll step on the given (GPU-produced) buffer; optionally only for
    a subset of robots (the step is independent per robot)."""
    robots = np.arange(case.B) if robots is None else np.asarray(robots)
    k = case.k if k is None else k
    v = case.v if v is None else v
    fop = case.fop if fop is None else fop
    delta = case.delta if delta is None else delta
    return expert.roll_step(case.cfg, case.W, np.asarray(buffer)[robots], case.t, k[:, robots], v[:, robots],
                            k.shape[3], fop[robots], delta[robots], case.seeds[robots],
                            np.asarray(counters, np.uint64)[robots], mask=mask)


def gpu_session(case: Case, mask_mode=0, max_batch=None, max_prefix=None):
    from paper_2609_34170_gb300 import RollingSession
    s = RollingSession(case.cfg, case.W, 0, max_batch or case.B, max_prefix or case.cfg.prefix, mask_mode)
    s.reset(case.seeds)
    s.set_context(case.k, case.v, case.P)
    return s


def check_step(case: Case, sess, mask="full", robots=None, label=""):
    """One GPU step vs the oracle on the same buffer; returns (max-abs, relL2)."""
    import torch
    buf0 = sess.buffer.cpu().numpy().copy()
    cnt0 = np.full(case.B, 0, np.uint64)
    cnt0[:] = sess.counters()
    sess.step(case.t, case.fop, case.delta, want_velocity=True)
    torch.cuda.synchronize()
    rel_gpu = sess.released.cpu().numpy()
    vel_gpu = sess.velocity.cpu().numpy()
    buf_gpu = sess.buffer.cpu().numpy()
    rob = np.arange(case.B) if robots is None else np.asarray(robots)
    rel_o, new_o, cnt_o, vel_o = oracle_step(case, buf0, cnt0, rob, mask)
    tol_a, tol_v = TOL[case.cfg.dtype]
    err_a = float(np.max(np.abs(rel_gpu[rob] - rel_o)))
    err_v = rel_l2(vel_gpu[rob], vel_o)
    assert err_a <= tol_a, f"{label} released max-abs {err_a:.3e} > {tol_a}"
    assert err_v <= tol_v, f"{label} velocity rel-L2 {err_v:.3e} > {tol_v}"
    # kept slots: within tolerance; appended slot: bit-exact noise
    assert float(np.max(np.abs(buf_gpu[rob, :-1] - new_o[:, :-1]))) <= tol_a
    np.testing.assert_array_equal(buf_gpu[rob, -1], new_o[:, -1].astype(np.float32))
    np.testing.assert_array_equal(sess.counters()[rob], cnt_o)
    return err_a, err_v
