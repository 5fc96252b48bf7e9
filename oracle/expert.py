"""Oracle: one rolling action-expert step in fp64 (test infrastructure).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg
may import this module; the CUDA library never does, and nothing here imports
the library.  Plain numpy, float64 throughout (the appended noise is the
float32 sequence of ``oracle.noise``).  No blocking, fusion or reordering:
each function is the definition it cites, in the order the paper states it.

The paper (Sec. 3.1, Eq. 1 and Eq. 3) defines the step as: one forward pass of
the flow-matching action expert v_theta(A, tau, c, delta_p) over the K-slot
buffer, a per-slot Euler update by the slot's flow-time step, release of the
first slot, a shift, and the append of a Gaussian slot.  The expert's
internals are not printed in the paper; the readings used here are:

* time convention t = 1 - tau (t = 1 pure noise); slot j (0-based, j = 0 is
  released next) carries t_j, staggered t_j = (j+1)/H;  dt_j = t_j - t_{j-1},
  t_{-1} = 0 (Eq. 3 uses the uniform 1/K);
* conditioning (App. A.1, pi0.5): cond = MLP_t(emb(t_j)) + MLP_d(emb(delta_b)),
  MLP = Linear -> SiLU -> Linear, emb = sinusoidal with periods geometric from
  4e-3 to 4;
* adaRMSNorm: x / sqrt(mean(x^2) + 1e-6) * (1 + scale) + shift, with
  (scale, shift) a slice of mod = cond @ W_mod + b_mod (two norms per layer and
  one final norm);
* VLM context (Eq. 2) = a per-layer prefix K/V cache; FOP tokens z (Eq. 4)
  enter every layer as extra keys/values through that layer's own K/V
  projection of RMSNorm(z) * (1 + gamma_l);
* attention: grouped-query, query head h reads KV head h // (Hq/Hkv); keys are
  [valid prefix | FOP | the H action slots]; full bidirectional mask (a
  ``slot_isolated`` test mask lets action query j see only action key j);
  no positional encoding; scale 1/sqrt(hd);
* MLP: GeGLU with the tanh form of GELU; no biases in QKV / O / MLP.
"""
from __future__ import annotations

import numpy as np

from .noise import action_noise

EPS = 1e-6


def _f64(a):
    return np.asarray(a, dtype=np.float64)


def sinusoidal(x, width: int) -> np.ndarray:
    """Sinusoidal embedding [..., width] of scalars x [...]: first half
    sin(x w_i), second half cos(x w_i), w_i = 2 pi / p_i, periods p_i
    geometric from 4e-3 (i = 0) to 4.0 (i = width/2 - 1)."""
    half = width // 2
    i = np.arange(half, dtype=np.float64)
    period = 4e-3 * (4.0 / 4e-3) ** (i / (half - 1))
    ang = _f64(x)[..., None] * (2.0 * np.pi / period)
    return np.concatenate([np.sin(ang), np.cos(ang)], axis=-1)


def per_slot(slot_times):
    """Slot times [H] (shared by every robot) or [B, H] (one schedule per
    robot) as a [1 or B, H, 1] array for per-slot arithmetic."""
    t = _f64(slot_times)
    return t[None, :, None] if t.ndim == 1 else t[:, :, None]


def silu(x):
    return x / (1.0 + np.exp(-x))


def gelu_tanh(x):
    """0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3))) (Hendrycks & Gimpel)."""
    return 0.5 * x * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (x + 0.044715 * x ** 3)))


def rmsnorm(x):
    """x / sqrt(mean(x^2) + eps) over the last axis."""
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + EPS)


def ada_rmsnorm(x, scale, shift):
    """adaRMSNorm with per-row modulation: rmsnorm(x) * (1 + scale) + shift."""
    return rmsnorm(x) * (1.0 + scale) + shift


def mlp2(e, w1, b1, w2, b2):
    """Linear -> SiLU -> Linear."""
    return silu(e @ _f64(w1) + _f64(b1)) @ _f64(w2) + _f64(b2)


def conditioning(cfg, W, slot_times, delta):
    """cond[b, j] = MLP_t(emb(t_j)) + MLP_d(emb(delta_b))  (App. A.1: the offset
    MLP's embedding is added to the flow-timestep embedding; every slot keeps
    its own t_j and all slots share delta_b).  slot_times [H], or [B, H] when
    every robot runs its own schedule (t_bj).  Returns [B, H, D]."""
    D = cfg.width
    ht = mlp2(sinusoidal(slot_times, D), W["t_w1"], W["t_b1"], W["t_w2"], W["t_b2"])   # [H, D] or [B, H, D]
    hd = mlp2(sinusoidal(delta, D), W["d_w1"], W["d_b1"], W["d_w2"], W["d_b2"])        # [B, D]
    return hd[:, None, :] + (ht[None, :, :] if ht.ndim == 2 else ht)


def modulation(cfg, W, cond):
    """mod = cond @ W_mod + b_mod: [B, H, 4 L D + 2 D]."""
    return cond @ _f64(W["mod_w"]) + _f64(W["mod_b"])


def mod_slice(cfg, mod, layer: int, which: int):
    """(scale, shift) of norm ``which`` (0: before attention, 1: before the MLP)
    of ``layer``; layer == cfg.layers selects the final norm."""
    D = cfg.width
    base = 4 * D * layer + 2 * D * which
    return mod[..., base:base + D], mod[..., base + D:base + 2 * D]


def attention(q, k, v, valid=None):
    """Softmax attention of one KV head.

    q [Nq, hd], k/v [Nk, hd], valid: optional bool [Nq, Nk] (True = visible).
    Returns [Nq, hd].  Masked keys are excluded from the softmax."""
    s = (q @ k.T) / np.sqrt(q.shape[-1])
    if valid is not None:
        s = np.where(valid, s, -np.inf)
    s = s - s.max(axis=-1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=-1, keepdims=True)
    return p @ v


def adapter_of_layer(cfg, layer: int) -> int:
    """Index of the FOP adapter in ``layer``, or -1: with adapters every k
    layers, layers k-1, 2k-1, ... carry one."""
    k = getattr(cfg, "fop_adapter_every", 0)
    return (layer + 1) // k - 1 if k and (layer + 1) % k == 0 else -1


def gated_cross_attention(cfg, W, i, x, fop):
    """FOP adapter i (Sec. 3.2: the FOP tokens are injected into selected
    expert layers through gated cross-attention adapters): the action rows
    attend to the FOP tokens only,
        q = (RMSNorm(x) (1 + a_gamma_i)) W_q,  [k | v] = (RMSNorm(z) (1 + a_zgamma_i)) W_kv,
    grouped-query heads as in the self-attention, and the result enters the
    residual stream through a tanh gate:  tanh(a_gate_i) * attn W_o.
    Returns that increment [B, H, D]."""
    B, H, D = x.shape
    F = fop.shape[1]
    Hq, Hkv, hd = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim
    G = Hq // Hkv
    q = ((rmsnorm(x) * (1.0 + _f64(W["a_gamma"][i]))) @ _f64(W["a_wq"][i])).reshape(B, H, Hq, hd)
    kv = (rmsnorm(_f64(fop)) * (1.0 + _f64(W["a_zgamma"][i]))) @ _f64(W["a_wkv"][i])
    k = kv[..., :Hkv * hd].reshape(B, F, Hkv, hd)
    v = kv[..., Hkv * hd:].reshape(B, F, Hkv, hd)
    o = np.empty((B, H, Hq, hd))
    for b in range(B):
        for h in range(Hq):
            o[b, :, h] = attention(q[b, :, h], k[b, :, h // G], v[b, :, h // G])
    return np.tanh(float(W["a_gate"][i])) * (o.reshape(B, H, Hq * hd) @ _f64(W["a_wo"][i]))


def expert_velocity(cfg, W, buffer, slot_times, ctx_k, ctx_v, prefix_len, fop, delta,
                    mask: str = "full", trace: dict | None = None):
    """v_theta(A, t, c, delta) for B robots: [B, H, A] float64 (Eq. 3's velocity).

    buffer [B, H, A]; slot_times [H] or [B, H]; ctx_k / ctx_v [L, B, Hkv, >=prefix_len, hd];
    fop [B, F, D]; delta [B].  prefix_len: one valid prefix length for every
    robot, or one per robot ([B]: robots whose contexts arrived at different
    times, Sec. 3.2).  ``trace`` (optional dict) receives intermediates.
    """
    B, H, A = buffer.shape
    D, L = cfg.width, cfg.layers
    Hq, Hkv, hd = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim
    G = Hq // Hkv
    adapters = getattr(cfg, "fop_adapter_every", 0) > 0
    F = 0 if adapters else fop.shape[1]   # FOP keys of the self-attention
    Pb = np.broadcast_to(np.asarray(prefix_len, dtype=np.int64), (B,))

    cond = conditioning(cfg, W, _f64(slot_times), _f64(delta))
    mod = modulation(cfg, W, cond)
    x = _f64(buffer) @ _f64(W["in_w"]) + _f64(W["in_b"])         # residual stream [B, H, D]
    zn = rmsnorm(_f64(fop))                                        # [B, F, D]

    if mask not in ("full", "slot_isolated"):
        raise ValueError(mask)

    def valid_of(P):   # [H, P + F + H]: which keys each slot sees
        valid = np.ones((H, P + F + H), dtype=bool)
        if mask == "slot_isolated":
            valid[:, P + F:] = np.eye(H, dtype=bool)
        return valid

    for l in range(L):
        wqkv = _f64(W["w_qkv"][l])
        sc, sh = mod_slice(cfg, mod, l, 0)
        y = ada_rmsnorm(x, sc, sh)                                  # [B, H, D]
        yf = (zn * (1.0 + _f64(W["fop_gamma"][l])))[:, :F]         # [B, F, D]
        qkv = y @ wqkv                                              # [B, H, NQKV]
        kvf = yf @ wqkv[:, Hq * hd:]                                # [B, F, 2 Hkv hd]
        q = qkv[..., :Hq * hd].reshape(B, H, Hq, hd)
        ka = qkv[..., Hq * hd:(Hq + Hkv) * hd].reshape(B, H, Hkv, hd)
        va = qkv[..., (Hq + Hkv) * hd:].reshape(B, H, Hkv, hd)
        kf = kvf[..., :Hkv * hd].reshape(B, F, Hkv, hd)
        vf = kvf[..., Hkv * hd:].reshape(B, F, Hkv, hd)
        o = np.empty((B, H, Hq, hd))
        for b in range(B):
            P = int(Pb[b])
            valid = valid_of(P)
            for g in range(Hkv):
                keys = np.concatenate([_f64(ctx_k[l, b, g, :P]), kf[b, :, g], ka[b, :, g]])
                vals = np.concatenate([_f64(ctx_v[l, b, g, :P]), vf[b, :, g], va[b, :, g]])
                for h in range(g * G, (g + 1) * G):
                    o[b, :, h] = attention(q[b, :, h], keys, vals, valid)
        x = x + o.reshape(B, H, Hq * hd) @ _f64(W["w_o"][l])
        if adapter_of_layer(cfg, l) >= 0:
            x = x + gated_cross_attention(cfg, W, adapter_of_layer(cfg, l), x, fop)
        sc2, sh2 = mod_slice(cfg, mod, l, 1)
        y2 = ada_rmsnorm(x, sc2, sh2)
        hmid = gelu_tanh(y2 @ _f64(W["w_gate"][l])) * (y2 @ _f64(W["w_up"][l]))
        x = x + hmid @ _f64(W["w_down"][l])
        if trace is not None:
            trace.setdefault("x", []).append(x.copy())

    scf, shf = mod_slice(cfg, mod, L, 0)
    v = ada_rmsnorm(x, scf, shf) @ _f64(W["out_w"]) + _f64(W["out_b"])
    if trace is not None:
        trace.update(cond=cond, mod=mod)
    return v


def slot_dt(slot_times):
    """dt_j = t_j - t_{j-1} with t_{-1} = 0 (Eq. 3's Delta tau per slot), per
    robot for [B, H] slot times."""
    t = _f64(slot_times)
    return np.diff(t, axis=-1, prepend=0.0)


def euler_roll(buffer, velocity, slot_times, seeds, counters):
    """Eq. 3 then the release / shift / append that follows it.

    a'_j = a_j + dt_j v_j for every slot; slot 0 (now at t = 0) is released; the
    remaining H-1 slots move forward; the new last slot is the Gaussian action
    of index n_b (the robot's counter), which then advances by one.
    Returns (released [B, A], new buffer [B, H, A], new counters [B]).
    """
    a = _f64(buffer) + per_slot(slot_dt(slot_times)) * _f64(velocity)
    released = a[:, 0].copy()
    B, H, A = a.shape
    counters = np.asarray(counters, dtype=np.uint64)
    fresh = np.stack([action_noise(int(seeds[b]), counters[b], A) for b in range(B)]) \
        if B else np.zeros((0, A), np.float32)
    new = np.concatenate([a[:, 1:], _f64(fresh)[:, None, :]], axis=1)
    return released, new, counters + np.uint64(1)


def to_relative(buffer, slot_times, state, rel_mask):
    """Absolute buffer -> the expert's relative coordinates (App. "LIBERO and
    RoboTwin 2.0": absolute targets are stored, and converted to actions
    relative to the latest robot state before each expert update; the paired
    noise stays in model coordinates).  A slot at flow time t holds
    a = t eps + (1 - t) a_hat, so expressing a_hat relative to the state s
    moves it by -(1 - t) s on the relative dimensions (rel_mask = 1)."""
    shift = (1.0 - per_slot(slot_times)) * (_f64(rel_mask)[None, None, :] * _f64(state)[:, None, :])
    return _f64(buffer) - shift


def to_absolute(buffer_rel, slot_times, state, rel_mask):
    """The inverse of to_relative at the given flow times."""
    shift = (1.0 - per_slot(slot_times)) * (_f64(rel_mask)[None, None, :] * _f64(state)[:, None, :])
    return _f64(buffer_rel) + shift


def roll_step(cfg, W, buffer, slot_times, ctx_k, ctx_v, prefix_len, fop, delta, seeds, counters,
              mask: str = "full", state=None, rel_mask=None):
    """One rolling action-expert step.  Returns (released, new buffer, new
    counters, velocity).

    With ``state`` [B, A] and ``rel_mask`` [A] (1 = a dimension the expert
    predicts relative to the robot state, 0 = absolute, e.g. a gripper), the
    buffer holds absolute coordinates: it is converted to relative ones at the
    slots' times, the expert and the Euler update act there, and every slot is
    converted back at its new time t_{j-1} (the released slot at t = 0 becomes
    its absolute target).  The appended noise slot (t = 1) needs no shift."""
    if state is None:
        v = expert_velocity(cfg, W, buffer, slot_times, ctx_k, ctx_v, prefix_len, fop, delta, mask)
        released, new, counters = euler_roll(buffer, v, slot_times, seeds, counters)
        return released, new, counters, v
    rel = to_relative(buffer, slot_times, state, rel_mask)
    v = expert_velocity(cfg, W, rel, slot_times, ctx_k, ctx_v, prefix_len, fop, delta, mask)
    return (*roll_relative(rel, v, slot_times, seeds, counters, state, rel_mask), v)


def roll_relative(rel, velocity, slot_times, seeds, counters, state, rel_mask):
    """Eq. 3 in relative coordinates, then each slot back to absolute ones at
    its new time (slot j moves from t_j to t_{j-1}, t_{-1} = 0), then the
    release / shift / append.  Returns (released, new buffer, new counters)."""
    t = _f64(slot_times)
    t_new = np.concatenate([np.zeros(t.shape[:-1] + (1,)), t[..., :-1]], axis=-1)
    a_rel = _f64(rel) + per_slot(slot_dt(slot_times)) * _f64(velocity)
    a = to_absolute(a_rel, t_new, state, rel_mask)
    B, H, A = a.shape
    released = a[:, 0].copy()
    counters = np.asarray(counters, dtype=np.uint64)
    fresh = np.stack([action_noise(int(seeds[b]), counters[b], A) for b in range(B)]) \
        if B else np.zeros((0, A), np.float32)
    new = np.concatenate([a[:, 1:], _f64(fresh)[:, None, :]], axis=1)
    return released, new, counters + np.uint64(1)


def denoise_chunk(cfg, W, seeds, counters, n_steps: int, ctx_k, ctx_v, prefix_len, fop, delta,
                  field=None, mask: str = "full"):
    """The full-horizon (synchronous) denoising baseline the paper compares
    rolling inference with (Experiments, synchronous simulation: ten
    full-horizon denoising steps per policy query, Table 1): a fresh chunk of H
    Gaussian actions -- robot b's actions of indices counters_b ..
    counters_b + H - 1 -- starts at flow time t = 1 and all H slots take
    ``n_steps`` Euler steps together, step n at t_n = 1 - n / n_steps (as
    float32, the precision of the flow times the step takes) with
    dt_n = t_n - t_{n+1}, t_{n_steps} = 0 (Eq. 3 with every slot at the same
    time; the step is read off the time grid as in the rolling update), each
    one expert pass at that single flow time.  The chunk ends at t = 0, where
    every action is executable.

    ``field(n, a, times) -> [B, H, A]`` replaces the expert (for closed-form
    checks).  Returns (chunk [B, H, A] float64, counters + H)."""
    H, A = cfg.slots, cfg.action_dim
    counters = np.asarray(counters, dtype=np.uint64)
    B = len(seeds)
    a = np.stack([action_noise(int(seeds[b]), counters[b] + np.arange(H, dtype=np.uint64), A)
                  for b in range(B)]).astype(np.float64) if B else np.zeros((0, H, A))
    grid = np.array([1.0 - n / n_steps for n in range(n_steps)] + [0.0], dtype=np.float32).astype(np.float64)
    for n in range(n_steps):
        times = np.full(H, grid[n], dtype=np.float32)
        if field is not None:
            v = field(n, a, times)
        else:
            v = expert_velocity(cfg, W, a, times, ctx_k, ctx_v, prefix_len, fop, delta, mask)
        a = a + (grid[n] - grid[n + 1]) * _f64(v)
    return a, counters + np.uint64(H)


def reset(cfg, seeds, H: int | None = None):
    """Warm start with no extra initialization (App. A.1): every slot j holds
    the Gaussian action of index j; the next appended action has index H.
    Returns (buffer [B, H, A] float32, counters [B] uint64)."""
    H = cfg.slots if H is None else H
    B = len(seeds)
    buf = np.stack([action_noise(int(s), np.arange(H, dtype=np.uint64), cfg.action_dim) for s in seeds]) \
        if B else np.zeros((0, H, cfg.action_dim), np.float32)
    return buf.astype(np.float32), np.full(B, H, dtype=np.uint64)
