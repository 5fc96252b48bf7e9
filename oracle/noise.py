"""Oracle: the Gaussian noise appended to the rolling buffer (test infrastructure).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg
may import this module; the CUDA library never does.

Section 3.1 of the paper appends a fresh slot drawn from N(0, I) after every
release.  The paper fixes no generator; this build fixes one so that the GPU
and this oracle must agree bit for bit:

* Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy
  as 1, 2, 3", SC'11): 10 rounds of the Philox S-box on a 4x32-bit counter with
  a 2x32-bit key bumped by the Weyl constants between rounds;
* key = (lo32(seed_b), hi32(seed_b)); counter = (lo32(n), hi32(n), g,
  0x4E4F4953) where n is the robot's absolute action index and g the group of
  four action dimensions 4g..4g+3;
* u_i = (2*(x_i >> 9) + 1) * 2^-24, an exact float32 in (0, 1);
* Box-Muller on (u0, u1) -> (z0, z1) and (u2, u3) -> (z2, z3):
  R = sqrt(-2 ln u_a), z = R cos(2 pi u_b), z' = R sin(2 pi u_b);
* ln and sincos(2 pi .) are this build's own float32 routines (below), written
  as a fixed sequence of individually rounded IEEE float32 operations (no fused
  multiply-add), so any IEEE-conforming machine reproduces them exactly.

numpy float32 ufuncs round every +, -, *, / and sqrt to float32 separately,
which is exactly that sequence.
"""
from __future__ import annotations

import numpy as np

F32 = np.float32
U32 = np.uint32

# Philox4x32 multipliers and Weyl key increments (SC'11, Philox-4x32).
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
NOISE_TAG = 0x4E4F4953  # fourth counter word of every action-noise draw


def philox4x32_10(ctr, key):
    """Philox4x32 with 10 rounds.

    ctr: four uint32 arrays (or scalars) of the same shape; key: two.  Returns
    four uint32 arrays.  Each round: (hi0, lo0) = M0 * c0, (hi1, lo1) = M1 * c2
    (full 64-bit products), new counter = (hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1,
    lo0); the key is bumped by (W0, W1) before every round after the first.
    """
    m = np.uint64(0xFFFFFFFF)
    c0, c1, c2, c3 = (np.asarray(c, dtype=np.uint64) & m for c in ctr)
    k0, k1 = (np.asarray(k, dtype=np.uint64) & m for k in key)
    for r in range(10):
        if r:
            k0 = (k0 + np.uint64(PHILOX_W0)) & m
            k1 = (k1 + np.uint64(PHILOX_W1)) & m
        p0 = np.uint64(PHILOX_M0) * c0
        p1 = np.uint64(PHILOX_M1) * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & m
        hi1, lo1 = p1 >> np.uint64(32), p1 & m
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return tuple(c.astype(U32) for c in (c0, c1, c2, c3))


def bits_to_uniform(x):
    """u = (2*(x >> 9) + 1) * 2^-24: odd multiples of 2^-24, exact in float32."""
    k = (np.asarray(x, dtype=U32) >> U32(9)).astype(np.int64)
    return ((2 * k + 1).astype(F32) * F32(2.0 ** -24)).astype(F32)


def _f(bits: int) -> np.float32:
    return np.array([bits], dtype=U32).view(F32)[0]


# float32 constants of the own ln: ln2 split into a 15-bit head (so e*LN2_HI is
# exact for |e| < 2^9) and the correctly rounded float32 of the remainder, plus
# the correctly rounded float32 of 1/3, 1/5, 1/7, 1/9 (the atanh series).
LN2_HI = _f(0x3F317200)   # 0.693145751953125
LN2_LO = _f(0x35BFBE8E)   # 1.4286068e-06
LN_C3, LN_C5, LN_C7, LN_C9 = _f(0x3EAAAAAB), _f(0x3E4CCCCD), _f(0x3E124925), _f(0x3DE38E39)
SQRT2_BITS = 0x3FB504F3   # float32 just below sqrt(2)

# Taylor coefficients of sin(pi r / 2) and cos(pi r / 2) in r, each the
# correctly rounded float32 of (-1)^k (pi/2)^n / n!.
SIN_C = [_f(0x3FC90FDB), _f(0xBF255DE7), _f(0x3DA335E3), _f(0xBB996966), _f(0x39283C1A)]   # n = 1,3,5,7,9
COS_C = [_f(0x3F800000), _f(0xBF9DE9E6), _f(0x3E81E0F8), _f(0xBCAAE9E4), _f(0x3A70FA83),
         _f(0xB7D368F9)]                                                                   # n = 0,2,..,10


def ln_f32(u):
    """Natural log of positive normal float32 values, as float32.

    u = m * 2^e with m in [sqrt(1/2), sqrt(2)); s = (m-1)/(m+1);
    ln m = 2 s (1 + s^2/3 + s^4/5 + s^6/7 + s^8/9) (the atanh series, |s| < 0.172,
    truncation < 1e-9 relative); ln u = e*LN2_HI + (e*LN2_LO + ln m).
    """
    u = np.asarray(u, dtype=F32)
    bits = u.view(U32)
    e = ((bits >> U32(23)) & U32(0xFF)).astype(np.int32) - 127
    mbits = (bits & U32(0x007FFFFF)) | U32(0x3F800000)
    big = mbits > U32(SQRT2_BITS)
    mbits = np.where(big, mbits - U32(0x00800000), mbits)   # m / 2, exact
    e = np.where(big, e + 1, e)
    m = mbits.view(F32)
    s = (m - F32(1)) / (m + F32(1))
    s2 = s * s
    p = LN_C9
    for c in (LN_C7, LN_C5, LN_C3, F32(1)):
        p = p * s2
        p = p + c
    lnm = (s + s) * p
    ef = e.astype(F32)
    return (ef * LN2_HI + (ef * LN2_LO + lnm)).astype(F32)


def sincos_2pi_f32(u):
    """(sin(2 pi u), cos(2 pi u)) for float32 u in [0, 1], as float32.

    x = 4u (exact), q = rint(x) (ties to even), r = x - q in [-1/2, 1/2] (exact),
    so 2 pi u = (pi/2)(q + r).  sin(pi r/2) and cos(pi r/2) are Horner-evaluated
    Taylor polynomials in r (degree 9 and 10); the quadrant q mod 4 then permutes
    and negates them.
    """
    u = np.asarray(u, dtype=F32)
    x = u * F32(4)
    q = np.rint(x)
    r = x - q
    r2 = r * r
    ps = SIN_C[4]
    for c in (SIN_C[3], SIN_C[2], SIN_C[1], SIN_C[0]):
        ps = ps * r2
        ps = ps + c
    sr = r * ps
    pc = COS_C[5]
    for c in (COS_C[4], COS_C[3], COS_C[2], COS_C[1], COS_C[0]):
        pc = pc * r2
        pc = pc + c
    cr = pc
    quad = q.astype(np.int64) & 3
    sin = np.select([quad == 0, quad == 1, quad == 2], [sr, cr, -sr], -cr).astype(F32)
    cos = np.select([quad == 0, quad == 1, quad == 2], [cr, -sr, -cr], sr).astype(F32)
    return sin, cos


def box_muller(ua, ub):
    """(R cos(2 pi ub), R sin(2 pi ub)) with R = sqrt(-2 ln ua), float32."""
    rad = np.sqrt(ln_f32(ua) * F32(-2)).astype(F32)
    s, c = sincos_2pi_f32(ub)
    return (rad * c).astype(F32), (rad * s).astype(F32)


def action_noise(seed: int, n, dim: int) -> np.ndarray:
    """The Gaussian action of absolute index n (scalar or array) for the robot
    whose noise seed is ``seed``: float32 [..., dim]."""
    n = np.asarray(n, dtype=np.uint64)
    groups = (dim + 3) // 4
    g = np.arange(groups, dtype=np.uint64)
    nn, gg = np.broadcast_arrays(n[..., None], g)
    seed = int(seed)
    x0, x1, x2, x3 = philox4x32_10(
        (nn & np.uint64(0xFFFFFFFF), nn >> np.uint64(32), gg, np.full(gg.shape, NOISE_TAG, np.uint64)),
        (seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF))
    z0, z1 = box_muller(bits_to_uniform(x0), bits_to_uniform(x1))
    z2, z3 = box_muller(bits_to_uniform(x2), bits_to_uniform(x3))
    z = np.stack([z0, z1, z2, z3], axis=-1).reshape(*n.shape, groups * 4)
    return np.ascontiguousarray(z[..., :dim])
