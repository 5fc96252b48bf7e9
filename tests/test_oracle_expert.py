"""Pins of the fp64 oracle of the rolling step (Eq. 1, Eq. 3, Sec. 3.1, App. A.1).

Nothing here re-types the oracle's formulas: each test checks it against a
library routine, a brute-force loop, a closed form of Euler integration, or a
structural law the step must obey (equivariance, batch independence, slot
isolation, GQA expansion, residual identity).
"""
import numpy as np
import pytest
import torch

import synth
from oracle import expert, noise

TINY = synth.ExpertConfig(layers=2, width=32, n_q_heads=4, n_kv_heads=2, head_dim=8, mlp_dim=48,
                          slots=5, action_dim=3, prefix=7, fop_tokens=2, batch=2, dtype="fp32")


def _inputs(cfg, seed=0, prefix_len=None, std=0.2):
    W = synth.make_weights(cfg, seed, std=std)
    k, v = synth.make_context(cfg, 100)
    z = synth.make_fop(cfg, 200)
    t = synth.staggered_times(cfg.slots)
    d = synth.make_delta(cfg.batch, [2, 5][:cfg.batch] + [1] * max(0, cfg.batch - 2), cfg.slots)
    buf, cnt = expert.reset(cfg, synth.robot_seeds(7, cfg.batch))
    return W, buf, t, k, v, cfg.prefix if prefix_len is None else prefix_len, z, d, cnt


# ----------------------------------------------------------------------------- parts

@pytest.mark.parametrize("nq,nk,hd", [(1, 1, 4), (3, 7, 8), (6, 12, 5)])
def test_attention_vs_bruteforce_and_sdpa(nq, nk, hd):
    rng = np.random.default_rng(nq * 100 + nk)
    q, k, v = rng.standard_normal((nq, hd)), rng.standard_normal((nk, hd)), rng.standard_normal((nk, hd))
    valid = rng.random((nq, nk)) < 0.7
    valid[:, 0] = True
    got = expert.attention(q, k, v, valid)
    for i in range(nq):   # brute force, one query at a time
        s = [sum(q[i, c] * k[j, c] for c in range(hd)) / np.sqrt(hd) for j in range(nk) if valid[i, j]]
        vv = [v[j] for j in range(nk) if valid[i, j]]
        w = np.exp(np.array(s) - max(s))
        np.testing.assert_allclose(got[i], (w[:, None] * np.array(vv)).sum(0) / w.sum(), rtol=1e-12)
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.tensor(q)[None], torch.tensor(k)[None], torch.tensor(v)[None],
        attn_mask=torch.tensor(valid)[None])[0].numpy()
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_attention_single_key_returns_value():
    v = np.array([[1.5, -2.0, 3.0]])
    out = expert.attention(np.ones((4, 3)), np.array([[0.3, 0.1, -9.0]]), v)
    np.testing.assert_array_equal(out, np.repeat(v, 4, axis=0))


def test_ada_rmsnorm_of_constant_row():
    sc = np.linspace(-0.5, 0.5, 16)
    sh = np.linspace(1.0, 2.0, 16)
    for c in (3.0, -40.0):   # eps = 1e-6 is negligible next to c^2
        y = expert.ada_rmsnorm(np.full(16, c), sc, sh)
        np.testing.assert_allclose(y, np.sign(c) * (1 + sc) + sh, rtol=1e-6)


def test_activations_vs_torch():
    x = np.linspace(-6, 6, 101)
    tx = torch.tensor(x)
    np.testing.assert_allclose(expert.gelu_tanh(x), torch.nn.functional.gelu(tx, approximate="tanh").numpy(),
                               rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(expert.silu(x), torch.nn.functional.silu(tx).numpy(), rtol=1e-13, atol=1e-15)


def test_sinusoidal_embedding_frequencies():
    D = 64
    e0 = expert.sinusoidal(np.array([0.0]), D)[0]
    np.testing.assert_array_equal(e0, np.r_[np.zeros(D // 2), np.ones(D // 2)])
    # component i completes a full period at x = p_i; p_0 = 4e-3, p_last = 4
    for i, p in ((0, 4e-3), (D // 2 - 1, 4.0)):
        e = expert.sinusoidal(np.array([p, p / 4]), D)
        assert abs(e[0, i]) < 1e-12 and abs(e[0, D // 2 + i] - 1) < 1e-12
        assert abs(e[1, i] - 1) < 1e-12 and abs(e[1, D // 2 + i]) < 1e-12


# ----------------------------------------------------------------------------- Euler / roll


def _rollout(cfg, steps, slot_times, field, seeds):
    """Run ``steps`` rolls from the reset buffer with an externally given
    velocity field(step, buffer) -> [B, H, A]; returns released [steps, B, A]."""
    buf, cnt = expert.reset(cfg, seeds)
    buf = buf.astype(np.float64)
    out = []
    for s in range(steps):
        rel, buf, cnt = expert.euler_roll(buf, field(s, buf), slot_times, seeds, cnt)
        out.append(rel)
    return np.array(out)


def _received_time(n, t):
    """Sum of dt an action with index n has received when released: t_min(n, H-1)."""
    return t[min(n, len(t) - 1)]


@pytest.mark.parametrize("schedule", ["staggered", "quadratic"])
def test_euler_constant_field_closed_form(schedule):
    cfg = TINY.replace(batch=2, slots=6, action_dim=5)
    H = cfg.slots
    t = synth.staggered_times(H) if schedule == "staggered" else (((np.arange(H) + 1) / H) ** 2).astype(np.float32)
    seeds = synth.robot_seeds(11, 2)
    c = np.array([0.5, -1.0, 2.0, 0.0, 3.0])
    rel = _rollout(cfg, 3 * H, t, lambda s, b: np.broadcast_to(c, b.shape), seeds)
    for n in range(3 * H):
        for b in range(2):
            a0 = noise.action_noise(int(seeds[b]), n, cfg.action_dim).astype(np.float64)
            np.testing.assert_allclose(rel[n, b], a0 + c * float(_received_time(n, t)), rtol=0, atol=1e-12)


def test_euler_dt_invariant_each_action_integrates_time_once():
    # unit field: released - initial noise = total flow time integrated = 1 after warm start
    cfg = TINY.replace(batch=1, slots=7, action_dim=2)
    t = synth.staggered_times(cfg.slots)
    seeds = synth.robot_seeds(3, 1)
    rel = _rollout(cfg, 4 * cfg.slots, t, lambda s, b: np.ones_like(b), seeds)
    for n in range(4 * cfg.slots):
        a0 = noise.action_noise(int(seeds[0]), n, 2).astype(np.float64)
        want = 1.0 if n >= cfg.slots - 1 else (n + 1) / cfg.slots
        np.testing.assert_allclose(rel[n, 0] - a0, want, rtol=0, atol=1e-7)


def test_euler_linear_and_time_fields_closed_form():
    cfg = TINY.replace(batch=1, slots=5, action_dim=3)
    H = cfg.slots
    t = synth.staggered_times(H)
    dt = np.diff(np.r_[0.0, t.astype(np.float64)])
    seeds = synth.robot_seeds(4, 1)
    alpha = -0.7
    rel = _rollout(cfg, 3 * H, t, lambda s, b: alpha * b, seeds)
    f = lambda tt: np.sin(3 * tt) + tt ** 2   # noqa: E731
    rel_t = _rollout(cfg, 3 * H, t, lambda s, b: np.broadcast_to(f(t.astype(np.float64))[None, :, None], b.shape), seeds)
    for n in range(3 * H):
        a0 = noise.action_noise(int(seeds[0]), n, 3).astype(np.float64)
        k = min(n, H - 1)
        np.testing.assert_allclose(rel[n, 0], a0 * np.prod(1 + alpha * dt[:k + 1]), rtol=1e-12)
        np.testing.assert_allclose(rel_t[n, 0], a0 + np.sum(f(t[:k + 1].astype(np.float64)) * dt[:k + 1]),
                                   rtol=1e-12, atol=1e-12)


def test_ideal_single_target_field_releases_targets_in_order():
    # v*(a, t) = (target - a) / t is the flow-matching field of one data point
    # (Eq. 5: a^tau = (1 - tau) eps + tau a_hat, velocity a_hat - eps); Euler is
    # exact on it, so every released action equals its own target, from the
    # very first (warm-start) step on.
    cfg = TINY.replace(batch=2, slots=6, action_dim=4)
    H = cfg.slots
    t = synth.staggered_times(H).astype(np.float64)
    steps = 4 * H
    targets = np.random.default_rng(9).standard_normal((steps + H, 2, 4))
    seeds = synth.robot_seeds(21, 2)

    def field(s, buf):
        tgt = np.stack([targets[s + j] for j in range(H)], axis=1)   # slot j holds action s + j
        return (tgt - buf) / t[None, :, None]

    rel = _rollout(cfg, steps, t.astype(np.float32), field, seeds)
    np.testing.assert_allclose(rel, targets[:steps], rtol=0, atol=1e-12)


def test_ideal_field_with_a_schedule_per_robot():
    # robots running their own slot-time schedules ([B, H] slot times): the
    # single-target field is still integrated exactly, so each robot releases
    # its targets in order (fails if a robot's dt comes from another robot's
    # schedule, or if dt is taken along the robot axis)
    cfg = TINY.replace(batch=2, slots=6, action_dim=4)
    H = cfg.slots
    t = np.stack([synth.staggered_times(H), ((np.arange(H) + 1) / H) ** 2]).astype(np.float32).astype(np.float64)
    steps = 3 * H
    targets = np.random.default_rng(19).standard_normal((steps + H, 2, 4))
    seeds = synth.robot_seeds(23, 2)

    def field(s, buf):
        tgt = np.stack([targets[s + j] for j in range(H)], axis=1)
        return (tgt - buf) / t[:, :, None]

    rel = _rollout(cfg, steps, t.astype(np.float32), field, seeds)
    np.testing.assert_allclose(rel, targets[:steps], rtol=0, atol=1e-12)


def test_per_robot_slot_times_are_independent_robots():
    # a step with one schedule per robot equals one-robot steps with each
    # robot's own schedule; with equal rows it equals the shared-times step
    cfg = TINY.replace(batch=3)
    W, buf, t, k, v, P, z, d, cnt = _inputs(cfg)
    H = cfg.slots
    tb = np.stack([t, ((np.arange(H) + 1) / H) ** 2, np.sqrt((np.arange(H) + 1) / H)]).astype(np.float32)
    seeds = synth.robot_seeds(7, 3)
    full = expert.roll_step(cfg, W, buf, tb, k, v, P, z, d, seeds, cnt)
    for b in range(3):
        one = expert.roll_step(cfg.replace(batch=1), W, buf[b:b + 1], tb[b], k[:, b:b + 1], v[:, b:b + 1], P,
                               z[b:b + 1], d[b:b + 1], seeds[b:b + 1], cnt[b:b + 1])
        for x, y in zip(full, one):
            np.testing.assert_allclose(np.asarray(x)[b], np.asarray(y)[0], rtol=1e-12, atol=1e-13)
    same = expert.roll_step(cfg, W, buf, np.stack([t] * 3), k, v, P, z, d, seeds, cnt)
    shared = expert.roll_step(cfg, W, buf, t, k, v, P, z, d, seeds, cnt)
    for x, y in zip(same, shared):
        np.testing.assert_allclose(np.asarray(x), np.asarray(y), rtol=1e-13, atol=1e-14)
    # relative coordinates follow each robot's own schedule too
    state = np.random.default_rng(4).standard_normal((3, cfg.action_dim))
    mask = np.array([1.0, 0.0, 1.0][:cfg.action_dim] + [1.0] * max(0, cfg.action_dim - 3))
    full = expert.roll_step(cfg, W, buf, tb, k, v, P, z, d, seeds, cnt, state=state, rel_mask=mask)
    for b in range(3):
        one = expert.roll_step(cfg.replace(batch=1), W, buf[b:b + 1], tb[b], k[:, b:b + 1], v[:, b:b + 1], P,
                               z[b:b + 1], d[b:b + 1], seeds[b:b + 1], cnt[b:b + 1], state=state[b:b + 1],
                               rel_mask=mask)
        for x, y in zip(full, one):
            np.testing.assert_allclose(np.asarray(x)[b], np.asarray(y)[0], rtol=1e-12, atol=1e-13)


def test_reset_and_append_bookkeeping():
    cfg = TINY.replace(batch=3, slots=4, action_dim=6)
    seeds = synth.robot_seeds(1 << 40, 3)
    buf, cnt = expert.reset(cfg, seeds)
    for b in range(3):
        for j in range(4):
            np.testing.assert_array_equal(buf[b, j], noise.action_noise(int(seeds[b]), j, 6))
    assert list(cnt) == [4, 4, 4]
    rel, new, cnt2 = expert.euler_roll(buf, np.zeros_like(buf), synth.staggered_times(4), seeds, cnt)
    np.testing.assert_array_equal(rel, buf[:, 0])
    np.testing.assert_array_equal(new[:, :3], buf[:, 1:])
    for b in range(3):
        np.testing.assert_array_equal(new[b, 3], noise.action_noise(int(seeds[b]), 4, 6))
    assert list(cnt2) == [5, 5, 5]


# ----------------------------------------------------------------------------- the network


def test_batch_independence():
    cfg = TINY.replace(batch=3)
    W, buf, t, k, v, P, z, d, _ = _inputs(cfg)
    full = expert.expert_velocity(cfg, W, buf, t, k, v, P, z, d)
    for b in range(3):
        one = expert.expert_velocity(cfg.replace(batch=1), W, buf[b:b + 1], t, k[:, b:b + 1], v[:, b:b + 1], P,
                                     z[b:b + 1], d[b:b + 1])
        np.testing.assert_allclose(full[b], one[0], rtol=1e-12, atol=1e-14)


def test_per_robot_prefix_lengths_are_independent_robots():
    # robots whose contexts arrived at different times attend to prefixes of
    # their own lengths (Sec. 3.2); each robot must equal a one-robot call with
    # its own length (fails if one robot's length is applied to all, or if a
    # robot's keys beyond its length leak in)
    cfg = TINY.replace(batch=3)
    W, buf, t, k, v, P, z, d, _ = _inputs(cfg)
    lens = np.array([P, 3, 1])
    full = expert.expert_velocity(cfg, W, buf, t, k, v, lens, z, d)
    for b in range(3):
        one = expert.expert_velocity(cfg.replace(batch=1), W, buf[b:b + 1], t, k[:, b:b + 1], v[:, b:b + 1],
                                     int(lens[b]), z[b:b + 1], d[b:b + 1])
        np.testing.assert_allclose(full[b], one[0], rtol=1e-12, atol=1e-14)
    assert np.abs(full[1] - expert.expert_velocity(cfg, W, buf, t, k, v, P, z, d)[1]).max() > 1e-6


def test_slot_permutation_equivariance():
    # full mask, no positional encoding: slots are told apart only by their times
    cfg = TINY
    W, buf, t, k, v, P, z, d, _ = _inputs(cfg)
    perm = np.array([3, 0, 4, 1, 2])
    a = expert.expert_velocity(cfg, W, buf, t, k, v, P, z, d)
    b = expert.expert_velocity(cfg, W, buf[:, perm], t[perm], k, v, P, z, d)
    np.testing.assert_allclose(b, a[:, perm], rtol=1e-11, atol=1e-13)


def test_prefix_permutation_and_padding_are_ignored():
    cfg = TINY
    W, buf, t, k, v, P, z, d, _ = _inputs(cfg, prefix_len=5)
    a = expert.expert_velocity(cfg, W, buf, t, k, v, 5, z, d)
    perm = np.r_[np.random.default_rng(2).permutation(5), 5, 6]
    k2, v2 = k[:, :, :, perm].copy(), v[:, :, :, perm].copy()
    k2[:, :, :, 5:] = 1e3
    v2[:, :, :, 5:] = -1e3
    b = expert.expert_velocity(cfg, W, buf, t, k2, v2, 5, z, d)
    np.testing.assert_allclose(b, a, rtol=1e-11, atol=1e-13)


def test_gqa_equals_mha_with_repeat_interleaved_kv():
    cfg = TINY            # Hq 4, Hkv 2: heads 0,1 read KV head 0; heads 2,3 read KV head 1
    W, buf, t, k, v, P, z, d, _ = _inputs(cfg)
    hd, Hq, Hkv = cfg.head_dim, cfg.n_q_heads, cfg.n_kv_heads
    G = Hq // Hkv
    mha = cfg.replace(n_kv_heads=Hq)
    W2 = dict(W)
    wq = W["w_qkv"][:, :, :Hq * hd]
    wk = W["w_qkv"][:, :, Hq * hd:(Hq + Hkv) * hd].reshape(cfg.layers, cfg.width, Hkv, hd)
    wv = W["w_qkv"][:, :, (Hq + Hkv) * hd:].reshape(cfg.layers, cfg.width, Hkv, hd)
    rep = lambda w: np.repeat(w, G, axis=2).reshape(cfg.layers, cfg.width, Hq * hd)  # noqa: E731
    W2["w_qkv"] = np.concatenate([wq, rep(wk), rep(wv)], axis=2)
    a = expert.expert_velocity(cfg, W, buf, t, k, v, P, z, d)
    b = expert.expert_velocity(mha, W2, buf, t, np.repeat(k, G, axis=2), np.repeat(v, G, axis=2), P, z, d)
    np.testing.assert_allclose(b, a, rtol=1e-11, atol=1e-13)


def test_slot_isolated_step_equals_independent_single_slot_calls():
    cfg = TINY
    W, buf, t, k, v, P, z, d, _ = _inputs(cfg)
    whole = expert.expert_velocity(cfg, W, buf, t, k, v, P, z, d, mask="slot_isolated")
    for j in range(cfg.slots):
        one = expert.expert_velocity(cfg.replace(slots=1), W, buf[:, j:j + 1], t[j:j + 1], k, v, P, z, d)
        np.testing.assert_allclose(whole[:, j], one[:, 0], rtol=1e-11, atol=1e-13)
    full = expert.expert_velocity(cfg, W, buf, t, k, v, P, z, d)
    assert np.max(np.abs(full - whole)) > 1e-6      # the masks really differ


def test_zero_output_projections_make_layers_identity():
    # x <- x + attn(...) W_o and x <- x + mlp(...) W_down: with both W zero the
    # layers are the identity and the expert reduces to its zero-layer form
    cfg = TINY
    W, buf, t, k, v, P, z, d, _ = _inputs(cfg)
    W0 = dict(W, w_o=np.zeros_like(W["w_o"]), w_down=np.zeros_like(W["w_down"]))
    a = expert.expert_velocity(cfg, W0, buf, t, k, v, P, z, d)
    c0 = cfg.replace(layers=0)
    Wz = {n: (W[n][:0] if n in ("fop_gamma", "w_qkv", "w_o", "w_gate", "w_up", "w_down") else W[n]) for n in W}
    Wz["mod_w"], Wz["mod_b"] = W["mod_w"][:, -2 * cfg.width:], W["mod_b"][-2 * cfg.width:]
    b = expert.expert_velocity(c0, Wz, buf, t, k, v, P, z, d)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-14)
    # ... while the full network differs from it
    assert np.max(np.abs(expert.expert_velocity(cfg, W, buf, t, k, v, P, z, d) - b)) > 1e-3


def test_uniform_queries_average_prefix_values_over_all_keys():
    # W_q = 0 makes every score 0 (uniform softmax over the P + F + H visible
    # keys); zero K/V projections make FOP and action values 0, so the first
    # layer's attention output is sum(prefix V) / (P + F + H) per head.
    cfg = TINY.replace(layers=1)
    Hq, Hkv, hd = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim
    W, buf, t, k, v, _, z, d, _ = _inputs(cfg)
    P = 5
    W1 = dict(W, w_qkv=np.zeros_like(W["w_qkv"]), w_gate=np.zeros_like(W["w_gate"]))
    tr = {}
    expert.expert_velocity(cfg, W1, buf, t, k, v, P, z, d, trace=tr)
    x0 = buf.astype(np.float64) @ W["in_w"] + W["in_b"]
    G = Hq // Hkv
    o = np.zeros((cfg.batch, Hq * hd))
    for b in range(cfg.batch):
        for h in range(Hq):
            o[b, h * hd:(h + 1) * hd] = v[0, b, h // G, :P].astype(np.float64).sum(0) / (P + cfg.fop_tokens + cfg.slots)
    want = x0 + (o @ W["w_o"][0].astype(np.float64))[:, None, :]
    np.testing.assert_allclose(tr["x"][0], want, rtol=1e-11, atol=1e-13)


def test_roll_step_composes_velocity_and_roll():
    cfg = TINY
    W, buf, t, k, v, P, z, d, cnt = _inputs(cfg)
    seeds = synth.robot_seeds(7, cfg.batch)
    rel, new, cnt2, vel = expert.roll_step(cfg, W, buf, t, k, v, P, z, d, seeds, cnt)
    np.testing.assert_allclose(rel, buf[:, 0] + t[0] * vel[:, 0], rtol=1e-12)
    assert np.all(cnt2 == cnt + 1)
    np.testing.assert_allclose(new[:, :-1], buf[:, 1:] + np.diff(np.r_[0, t.astype(np.float64)])[None, 1:, None]
                               * vel[:, 1:], rtol=1e-12)


def test_conditioning_with_permutation_weights_vs_torch_silu():
    # W1 a permutation, W2 diagonal: cond = silu(emb(t) permuted + b1) * s + b2
    # for the time MLP, plus the same for the offset MLP (App. A.1: the offset
    # embedding is added to the flow-timestep embedding).  A transposed or
    # misplaced operand moves entries and fails this.
    cfg = TINY.replace(width=16)
    D = cfg.width
    rng = np.random.default_rng(3)
    W = {}
    want = {}
    x = {"t": np.array([0.2, 0.6, 1.0]), "d": np.array([0.0, 0.35])}
    for m in ("t", "d"):
        pi = rng.permutation(D)
        P = np.zeros((D, D))
        P[np.arange(D), pi] = 1.0
        b1, s, b2 = rng.standard_normal(D), rng.standard_normal(D), rng.standard_normal(D)
        W.update({f"{m}_w1": P, f"{m}_b1": b1, f"{m}_w2": np.diag(s), f"{m}_b2": b2})
        e = expert.sinusoidal(x[m], D)
        moved = np.empty_like(e)
        moved[:, pi] = e
        want[m] = torch.nn.functional.silu(torch.tensor(moved + b1)).numpy() * s + b2
    cond = expert.conditioning(cfg, W, x["t"], x["d"])
    np.testing.assert_allclose(cond, want["d"][:, None, :] + want["t"][None, :, :], rtol=1e-12, atol=1e-13)


# ----------------------------------------------------------------------------- the FOP branch (Eq. 4)
# FOP tokens z enter every layer as extra keys / values: that layer's K / V
# projection of RMSNorm(z) * (1 + gamma_l) (the FOP-as-keys reading of Eq. 4).
# The two pins below fail on the plausible slips of that branch: a dropped
# RMSNorm on z, gamma used in place of 1 + gamma, the action rows' modulation
# applied to the FOP rows, the K columns used as values, or a wrong key count.


def test_fop_tokens_enter_through_a_scale_free_norm():
    # RMSNorm(c z) = RMSNorm(z) for c > 0 (eps negligible: |z| ~ 100), so the
    # velocity must not change when the tokens are rescaled -- and it must
    # change when they are replaced.
    cfg = TINY
    W, buf, t, k, v, P, z, d, _ = _inputs(cfg)
    z = z.astype(np.float64) * 100.0
    a = expert.expert_velocity(cfg, W, buf, t, k, v, P, z, d)
    for c in (0.1, 7.3):
        b = expert.expert_velocity(cfg, W, buf, t, k, v, P, c * z, d)
        # eps shifts RMSNorm(c z) by ~eps (1/c^2 - 1) / (2 mean(z^2)) ~ 5e-9
        np.testing.assert_allclose(b, a, rtol=1e-6, atol=1e-10)
    other = synth.make_fop(cfg, 999) * 100.0
    assert np.max(np.abs(expert.expert_velocity(cfg, W, buf, t, k, v, P, other, d) - a)) > 1e-3


def test_fop_values_closed_form_first_layer():
    # W_q = 0 makes every score 0, so each head's first-layer attention output
    # is the plain mean of the P prefix, F FOP and H action values of its KV
    # head.  With W_gate = 0 the MLP adds nothing, with W_mod = 0 every row's
    # modulation is the bias, and with in_w = 0 every action row is the bias
    # in_b (large, so eps is negligible).  The values are written out here
    # from the definitions: FOP  sqrt(D) z / |z| * (1 + gamma_0) @ W_v,
    # action  (sqrt(D) x0 / |x0| * (1 + scale) + shift) @ W_v.
    cfg = TINY.replace(layers=1)
    D, Hq, Hkv, hd, H, F = cfg.width, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.slots, cfg.fop_tokens
    G = Hq // Hkv
    W, buf, t, k, v, _, z, d, _ = _inputs(cfg)
    P = 6
    z = z.astype(np.float64) * 100.0
    W1 = dict(W)
    wqkv = W["w_qkv"].astype(np.float64).copy()
    wqkv[:, :, :(Hq + Hkv) * hd] = 0.0                 # Q and K columns
    W1.update(w_qkv=wqkv, w_gate=np.zeros_like(W["w_gate"]), mod_w=np.zeros_like(W["mod_w"]),
              in_w=np.zeros_like(W["in_w"]), in_b=W["in_b"].astype(np.float64) * 1000.0)
    W1["fop_gamma"] = W["fop_gamma"].astype(np.float64) * 20.0   # far from 0, so gamma vs 1 + gamma differs
    tr = {}
    expert.expert_velocity(cfg, W1, buf, t, k, v, P, z, d, trace=tr)
    wv = wqkv[0][:, (Hq + Hkv) * hd:]                  # [D, Hkv hd]
    x0 = W1["in_b"]
    sc, sh = W["mod_b"][:D].astype(np.float64), W["mod_b"][D:2 * D].astype(np.float64)
    ya = np.sqrt(D) * x0 / np.linalg.norm(x0) * (1.0 + sc) + sh
    va = ya @ wv                                        # the same for every slot
    o = np.zeros((cfg.batch, Hq * hd))
    for b in range(cfg.batch):
        yf = np.sqrt(D) * z[b] / np.linalg.norm(z[b], axis=1, keepdims=True) * (1.0 + W1["fop_gamma"][0])
        vf = yf @ wv                                    # [F, Hkv hd]
        for h in range(Hq):
            g = h // G
            tot = v[0, b, g, :P].astype(np.float64).sum(0) + vf[:, g * hd:(g + 1) * hd].sum(0) \
                + H * va[g * hd:(g + 1) * hd]
            o[b, h * hd:(h + 1) * hd] = tot / (P + F + H)
    want = x0[None, None, :] + (o @ W["w_o"][0].astype(np.float64))[:, None, :]
    np.testing.assert_allclose(tr["x"][0], np.broadcast_to(want, tr["x"][0].shape), rtol=1e-9, atol=1e-9)


# ----------------------------------------------------------------------------- full-chunk denoising baseline


def test_denoise_chunk_constant_field_and_noise_indices():
    # c = 0 leaves the chunk at its fresh noise: actions counters .. counters + H - 1;
    # a constant field c moves every action by c * sum(dt) = c
    cfg = TINY.replace(batch=2, slots=5, action_dim=3)
    seeds = synth.robot_seeds(13, 2)
    cnt = np.array([5, 40], np.uint64)
    for c in (0.0, 1.75):
        for n_steps in (1, 4, 10):
            chunk, cnt2 = expert.denoise_chunk(cfg, None, seeds, cnt, n_steps, None, None, 0, None, None,
                                               field=lambda n, a, tt: np.full_like(a, c))
            assert list(cnt2) == [10, 45]
            for b in range(2):
                for j in range(5):
                    a0 = noise.action_noise(int(seeds[b]), int(cnt[b]) + j, 3).astype(np.float64)
                    np.testing.assert_allclose(chunk[b, j], a0 + c, rtol=0, atol=1e-12)


def test_denoise_chunk_is_exact_on_the_single_target_field():
    # v*(a, t) = (target - a) / t is the flow-matching field of one data point
    # (Eq. 5); Euler is exact on its straight path, so ten (or any number of)
    # synchronous steps from t = 1 land every slot on its own target
    cfg = TINY.replace(batch=2, slots=6, action_dim=4)
    seeds = synth.robot_seeds(17, 2)
    targets = np.random.default_rng(4).standard_normal((2, 6, 4))
    seen = []

    def field(n, a, times):
        seen.append(float(times[0]))
        assert np.all(times == times[0])               # one flow time for the whole chunk
        return (targets - a) / float(times[0])

    for n_steps in (1, 3, 10):
        seen.clear()
        chunk, _ = expert.denoise_chunk(cfg, None, seeds, np.zeros(2, np.uint64), n_steps, None, None, 0, None,
                                        None, field=field)
        np.testing.assert_allclose(chunk, targets, rtol=0, atol=1e-12)
        np.testing.assert_allclose(seen, 1.0 - np.arange(n_steps) / n_steps, rtol=1e-7)


def test_denoise_chunk_one_step_is_one_expert_pass_at_t1():
    cfg = TINY
    W, _, _, k, v, P, z, d, _ = _inputs(cfg)
    seeds = synth.robot_seeds(7, cfg.batch)
    cnt = np.full(cfg.batch, 9, np.uint64)
    chunk, _ = expert.denoise_chunk(cfg, W, seeds, cnt, 1, k, v, P, z, d)
    a0 = np.stack([noise.action_noise(int(seeds[b]), 9 + np.arange(cfg.slots, dtype=np.uint64), cfg.action_dim)
                   for b in range(cfg.batch)]).astype(np.float64)
    vel = expert.expert_velocity(cfg, W, a0, np.ones(cfg.slots, np.float32), k, v, P, z, d)
    np.testing.assert_allclose(chunk, a0 + vel, rtol=1e-12, atol=1e-14)


# ----------------------------------------------------------------------------- relative <-> absolute buffer


def test_relative_coordinates_keep_absolute_targets_while_the_state_moves():
    # The expert predicts relative to the latest robot state (App. "LIBERO and
    # RoboTwin 2.0"); the buffer stores absolute targets.  With the ideal
    # single-target field written in relative coordinates -- the target
    # relative to THIS step's state -- every released action must be its
    # absolute target, although the state changes at every step; the gripper
    # dimension (rel_mask 0) is absolute throughout.
    cfg = TINY.replace(batch=2, slots=6, action_dim=4)
    H = cfg.slots
    t = synth.staggered_times(H).astype(np.float64)
    rng = np.random.default_rng(11)
    steps = 4 * H
    targets = rng.standard_normal((steps + H, 2, 4))       # absolute targets of action n
    states = rng.standard_normal((steps, 2, 4)) * 3.0       # a different robot state every step
    rel_mask = np.array([1.0, 1.0, 1.0, 0.0])
    seeds = synth.robot_seeds(31, 2)
    buf, cnt = expert.reset(cfg, seeds)
    buf = buf.astype(np.float64)
    out = []
    for s in range(steps):
        rel = expert.to_relative(buf, t.astype(np.float32), states[s], rel_mask)
        tgt_rel = np.stack([targets[s + j] for j in range(H)], axis=1) - rel_mask * states[s][:, None, :]
        v = (tgt_rel - rel) / t[None, :, None]
        released, buf, cnt = expert.roll_relative(rel, v, t.astype(np.float32), seeds, cnt, states[s], rel_mask)
        out.append(released)
    np.testing.assert_allclose(np.array(out), targets[:steps], rtol=0, atol=1e-10)
    # ... while keeping the stored targets relative (no conversion) breaks it
    buf, cnt = expert.reset(cfg, seeds)
    buf = buf.astype(np.float64)
    for s in range(H + 2):
        tgt_rel = np.stack([targets[s + j] for j in range(H)], axis=1) - rel_mask * states[s][:, None, :]
        released, buf, cnt = expert.euler_roll(buf, (tgt_rel - buf) / t[None, :, None], t.astype(np.float32), seeds, cnt)
    assert np.max(np.abs(released - targets[H + 1])) > 0.1


def test_relative_step_with_zero_mask_is_the_absolute_step():
    cfg = TINY
    W, buf, t, k, v, P, z, d, cnt = _inputs(cfg)
    seeds = synth.robot_seeds(7, cfg.batch)
    state = np.random.default_rng(2).standard_normal((cfg.batch, cfg.action_dim))
    a = expert.roll_step(cfg, W, buf, t, k, v, P, z, d, seeds, cnt)
    b = expert.roll_step(cfg, W, buf, t, k, v, P, z, d, seeds, cnt, state=state, rel_mask=np.zeros(cfg.action_dim))
    for x, y in zip(a, b):
        np.testing.assert_allclose(np.asarray(x, np.float64), np.asarray(y, np.float64), rtol=1e-13, atol=1e-14)
    # with a mask, the expert sees the buffer shifted by (1 - t_j) s on those dimensions
    m = np.array([1.0] * (cfg.action_dim - 1) + [0.0])
    rel, new, _, vel = expert.roll_step(cfg, W, buf, t, k, v, P, z, d, seeds, cnt, state=state, rel_mask=m)
    want_v = expert.expert_velocity(cfg, W, buf - (1 - t.astype(np.float64))[None, :, None] * (m * state)[:, None, :],
                                    t, k, v, P, z, d)
    np.testing.assert_allclose(vel, want_v, rtol=1e-12, atol=1e-14)
    # slot 0 moves from t_0 to 0: a' = a + dt (v + m s), dt = t_0
    np.testing.assert_allclose(rel, buf[:, 0] + t[0] * (vel[:, 0] + m * state), rtol=1e-12, atol=1e-13)


# ----------------------------------------------------------------------------- gated cross-attention FOP adapters


ADAPT = TINY.replace(layers=4, fop_adapter_every=2)      # adapters in layers 1 and 3


def test_adapter_with_closed_gates_is_the_network_without_fop():
    # tanh(0) = 0: every adapter adds nothing, and in adapter mode the FOP
    # tokens are no keys of the self-attention -- so the expert is the one
    # that never sees them
    W, buf, t, k, v, P, z, d, _ = _inputs(ADAPT)
    W0 = dict(W, a_gate=np.zeros_like(W["a_gate"]))
    a = expert.expert_velocity(ADAPT, W0, buf, t, k, v, P, z, d)
    nofop = ADAPT.replace(fop_adapter_every=0, fop_tokens=0)
    Wn = {n: W[n] for n in synth.weight_names(nofop)}
    b = expert.expert_velocity(nofop, Wn, buf, t, k, v, P, z[:, :0], d)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-14)
    # open gates change the result, and do not depend on the order of the FOP tokens
    W1 = dict(W, a_gate=np.full_like(W["a_gate"], 0.8))
    c = expert.expert_velocity(ADAPT, W1, buf, t, k, v, P, z, d)
    assert np.max(np.abs(c - a)) > 1e-4
    perm = np.random.default_rng(1).permutation(ADAPT.fop_tokens)
    np.testing.assert_allclose(expert.expert_velocity(ADAPT, W1, buf, t, k, v, P, z[:, perm], d), c,
                               rtol=1e-11, atol=1e-13)


def test_adapter_closed_form_one_layer():
    # one layer with its adapter; W_q^a = 0 makes the cross-attention uniform
    # over the F FOP tokens, and zero self-attention / MLP outputs leave
    #   x1 = x0 + tanh(g) * (mean_f (sqrt(D) z_f / |z_f| (1 + a_zgamma)) W_v^a) W_o^a
    # per head (|z| ~ 100: eps negligible), written out here from the definition
    cfg = TINY.replace(layers=1, fop_adapter_every=1)
    D, Hq, Hkv, hd, F = cfg.width, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.fop_tokens
    G = Hq // Hkv
    W, buf, t, k, v, P, z, d, _ = _inputs(cfg)
    z = z.astype(np.float64) * 100.0
    g = 2.0     # tanh(2) = 0.964, unlike sigmoid(2) or 2 itself
    W1 = dict(W, a_wq=np.zeros_like(W["a_wq"]), w_o=np.zeros_like(W["w_o"]), w_gate=np.zeros_like(W["w_gate"]),
              a_gate=np.array([g]), a_zgamma=W["a_zgamma"].astype(np.float64) * 20.0)
    tr = {}
    expert.expert_velocity(cfg, W1, buf, t, k, v, P, z, d, trace=tr)
    x0 = buf.astype(np.float64) @ W["in_w"] + W["in_b"]
    wv = W["a_wkv"][0].astype(np.float64)[:, Hkv * hd:]
    o = np.zeros((cfg.batch, Hq * hd))
    for b in range(cfg.batch):
        yz = np.sqrt(D) * z[b] / np.linalg.norm(z[b], axis=1, keepdims=True) * (1.0 + W1["a_zgamma"][0])
        vf = yz @ wv
        for h in range(Hq):
            o[b, h * hd:(h + 1) * hd] = vf[:, (h // G) * hd:(h // G + 1) * hd].mean(0)
    want = x0 + np.tanh(g) * (o @ W["a_wo"][0].astype(np.float64))[:, None, :]
    np.testing.assert_allclose(tr["x"][0], want, rtol=1e-9, atol=1e-9)
