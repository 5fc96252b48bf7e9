"""RollingSession: one handle plus the device tensors of a rollout (buffer,
released action, optional velocity), driven through the C ABI.  Every tensor
argument may be a numpy array (copied to the device in the handle's dtype) or
a CUDA tensor already in the right dtype."""
from __future__ import annotations

import numpy as np

from . import _binding as B


class RollingSession:
    def __init__(self, cfg, weights: dict, device: int = 0, max_batch: int | None = None,
                 max_prefix: int | None = None, mask_mode: int = B.RAVEL_MASK_FULL):
        import torch
        self.torch = torch
        self.cfg = cfg
        self.device = torch.device("cuda", device)
        self.dtype = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
        self.handle = B.ravel_create(cfg, weights, device, max_batch, max_prefix, mask_mode)
        self.batch = 0

    # -- helpers
    def to_dev(self, a, dtype=None):
        t = self.torch
        dtype = dtype or self.dtype
        if isinstance(a, np.ndarray):
            return t.from_numpy(np.ascontiguousarray(a)).to(device=self.device, dtype=dtype)
        return a.to(device=self.device, dtype=dtype).contiguous()

    def reset(self, seeds, stream=None):
        t = self.torch
        seeds = np.ascontiguousarray(seeds, dtype=np.uint64)
        Bn, H, A = len(seeds), self.cfg.slots, self.cfg.action_dim
        self.batch = Bn
        self.buffer = t.empty((Bn, H, A), device=self.device, dtype=t.float32)
        self.chunk = t.empty((Bn, H, A), device=self.device, dtype=t.float32)
        self.released = t.empty((Bn, A), device=self.device, dtype=t.float32)
        self.velocity = t.empty((Bn, H, A), device=self.device, dtype=t.float32)
        # persistent step inputs: the step graph is captured on their addresses
        # one schedule for every robot, or one per robot
        nt = Bn * H if getattr(self.cfg, "per_robot_times", 0) else H
        self.slot_times = t.zeros((nt,), device=self.device, dtype=t.float32)
        self.obs = t.zeros((Bn, self.cfg.fop_tokens, self.cfg.width), device=self.device, dtype=self.dtype)
        self.delta = t.zeros((Bn,), device=self.device, dtype=t.float32)
        B.ravel_reset(self.handle, Bn, seeds, self.buffer, stream)
        return self.buffer

    def set_context(self, k, v, prefix_len: int | None = None, side_stream=None):
        k, v = self.to_dev(k), self.to_dev(v)
        self._ctx = (k, v)   # keep alive until the side-stream copy has run
        B.ravel_set_context(self.handle, k, v, int(prefix_len or k.shape[3]), side_stream)

    def set_context_robots(self, robots, k, v, prefix_len: int | None = None, side_stream=None):
        """New contexts for the listed robots only: k, v [L, len(robots), Hkv, P, hd]."""
        k, v = self.to_dev(k), self.to_dev(v)
        self._ctx_robots = (k, v)   # keep alive until the side-stream copy has run
        B.ravel_set_context_robots(self.handle, robots, k, v, int(prefix_len or k.shape[3]), side_stream)

    def step(self, slot_times, obs, delta, want_velocity: bool = False, stream=None, state=None):
        """One rolling step; with `state` ([B, A]) the buffer holds absolute
        targets and the expert works relative to that state (see
        ravel_roll_step_rel and set_relative_dims)."""
        t = self.torch
        ts = self.to_dev(slot_times, t.float32).reshape(-1)
        self.slot_times[:ts.numel()].copy_(ts)
        if self.cfg.fop_tokens:
            self.obs.copy_(self.to_dev(obs))
        self.delta.copy_(self.to_dev(delta, t.float32))
        obs_arg = self.obs if self.cfg.fop_tokens else None
        vel_arg = self.velocity if want_velocity else None
        if state is None:
            B.ravel_roll_step(self.handle, self.buffer, self.slot_times, obs_arg, self.delta, self.released, vel_arg,
                              stream)
        else:
            if not hasattr(self, "state"):
                self.state = t.zeros((self.batch, self.cfg.action_dim), device=self.device, dtype=t.float32)
            self.state.copy_(self.to_dev(state, t.float32))
            B.ravel_roll_step_rel(self.handle, self.buffer, self.slot_times, obs_arg, self.delta, self.state,
                                  self.released, vel_arg, stream)
        return self.released

    def set_relative_dims(self, mask):
        B.ravel_set_relative_dims(self.handle, mask)

    def denoise_chunk(self, n_steps: int, obs, delta, want_velocity: bool = False, stream=None):
        """Full-horizon denoising of a fresh chunk (the paper's synchronous
        baseline): returns the [B, H, A] chunk tensor (t = 0)."""
        t = self.torch
        if not hasattr(self, "chunk"):
            self.chunk = t.empty_like(self.buffer)
        if self.cfg.fop_tokens:
            self.obs.copy_(self.to_dev(obs))
        self.delta.copy_(self.to_dev(delta, t.float32))
        B.ravel_denoise_chunk(self.handle, self.chunk, n_steps, self.obs if self.cfg.fop_tokens else None, self.delta,
                              self.velocity if want_velocity else None, stream)
        return self.chunk

    def counters(self) -> np.ndarray:
        return B.ravel_get_state(self.handle, self.batch)

    def set_counters(self, c):
        B.ravel_set_state(self.handle, c)

    def kernel_count(self) -> int:
        return B.ravel_step_kernel_count(self.handle)

    def close(self):
        if getattr(self, "handle", None) is not None:
            B.ravel_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
