"""Pins for the RRQ oracle: facts fixed by the paper and by mathematics, not by
the oracle itself.

Each ``pin_*`` function takes an ``oracle.Oracle`` (the committed library or a
test's deliberately mutated copy) and returns a list of failure strings (empty
when the pin holds).  ``tests/test_oracle_pins.py`` requires every pin to hold
for the committed oracle; ``tests/test_oracle_mutants.py`` requires every
planted mistake to break at least one pin.

Sources of truth:
  * hand-worked groups (tests/golden/worked_groups.json), derived by hand in
    exact arithmetic from Eq. 1-8 and Algorithm 1;
  * brute force: on dyadic inputs whose arithmetic is exact, each code must be
    the nearest of the stage's four levels (Eq. 2-3 with round-half-to-even),
    checked with exact rationals;
  * invariants of the method: half-step bound per stage, exact reconstruction
    of groups already on a 4-level grid, L-infinity error shrinking by >= 3x
    per stage (Eq. 5-8), prefix reconstruction equal to input minus residual.
"""
from __future__ import annotations

import json
import os
import struct
from fractions import Fraction

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                      "worked_groups.json")


def f32_from_bits(h: str) -> np.float32:
    return np.frombuffer(struct.pack("<I", int(h, 16)), dtype=np.float32)[0]


def bits_of(f) -> int:
    return int(np.asarray(f, dtype=np.float32).view(np.uint32))


def bf16_bits_of_f32(x: np.ndarray) -> np.ndarray:
    """bf16 bit patterns of exactly-bf16-representable float32 values."""
    u = np.asarray(x, np.float32).view(np.uint32)
    assert np.all((u & 0xFFFF) == 0), "value is not bf16-representable"
    return (u >> 16).astype(np.uint16)


def _golden_cases():
    with open(GOLDEN) as f:
        return {c["name"]: c for c in json.load(f)["cases"]}


# ---------------------------------------------------------------------------
# hand-worked groups
# ---------------------------------------------------------------------------
# WE3: eight bf16 weights, four stages; values derived for the design by hand
# from Eq. 1-8 and re-checked in exact rational arithmetic.
WE3_X = [0.0234375, -0.01171875, 0.0517578125, -0.0400390625,
         0.00439453125, -0.0029296875, 0.0146484375, -0.0625]
WE3_Q = [[2, 1, 3, 1, 2, 2, 2, 0], [3, 3, 2, 0, 1, 0, 2, 2],
         [0, 2, 0, 3, 0, 2, 1, 0], [1, 2, 1, 1, 3, 2, 0, 1]]
WE3_SCALE_BITS = [0x3D1C0000, 0x3C200000, 0x3AAAAAAB, 0x398E38E4]
WE3_ZERO = [-0.0625, -0.0166015625, -0.0029296875, -0.0003255208721384406]


def pin_worked_groups(orc) -> list[str]:
    fails = []
    cases = _golden_cases()
    for name in ("WE1", "WE2"):
        c = cases[name]
        x = np.array(c["x"], np.float32)
        Q, s, z, _ = orc.quantize_group(x, 4)
        if Q.tolist() != c["Q"]:
            fails.append(f"{name}: codes {Q.tolist()} != {c['Q']}")
        if [bits_of(v) for v in s] != [int(h, 16) for h in c["scale_bits"]]:
            fails.append(f"{name}: scales {[hex(bits_of(v)) for v in s]}")
        if [bits_of(v) for v in z] != [int(h, 16) for h in c["zero_bits"]]:
            fails.append(f"{name}: zeros {[hex(bits_of(v)) for v in z]}")
        # the packed matrix form and the bf16 prefix reconstructions
        W = bf16_bits_of_f32(x).reshape(1, 4)
        codes, scales, zeros = orc.quantize(W, group=4, n_stages=4)
        packed = [hex(int(cd[0])) for cd in codes]
        if packed != [hex(int(h, 16)) for h in c["packed"]]:
            fails.append(f"{name}: packed {packed} != {c['packed']}")
        for k in range(1, 5):
            rec = orc.reconstruct(codes, scales, zeros, 1, 4, 4, k)[0]
            want = [int(h, 16) for h in c["recon_bf16"][k - 1]]
            if rec.tolist() != want:
                fails.append(f"{name}: recon k={k} {[hex(v) for v in rec]} != {c['recon_bf16'][k-1]}")

    x = np.array(WE3_X, np.float32)
    Q, s, z, _ = orc.quantize_group(x, 4)
    if Q.tolist() != WE3_Q:
        fails.append(f"WE3: codes {Q.tolist()}")
    if [bits_of(v) for v in s] != WE3_SCALE_BITS:
        fails.append(f"WE3: scales {[hex(bits_of(v)) for v in s]}")
    if [float(v) for v in z] != WE3_ZERO:
        fails.append(f"WE3: zeros {[float(v) for v in z]}")

    c = cases["WE4_subnormal_clamp"]
    x = np.array([f32_from_bits(h) for h in c["x_bits"]], np.float32)
    Q, s, z, r = orc.quantize_group(x, 4)
    if Q.tolist() != c["Q"]:
        fails.append(f"WE4: codes {Q.tolist()}")
    if [bits_of(v) for v in s] != [int(h, 16) for h in c["scale_bits"]]:
        fails.append(f"WE4: scales {[hex(bits_of(v)) for v in s]}")
    if [[bits_of(v) for v in row] for row in r] != [[int(h, 16) for h in row] for row in c["resid_bits"]]:
        fails.append("WE4: residuals")

    c = cases["WE5_signed_zero"]
    x = np.array([f32_from_bits(h) for h in c["x_bits"]], np.float32)
    Q, s, z, r = orc.quantize_group(x, 4)
    if Q[0].tolist() != c["Q0"]:
        fails.append(f"WE5: codes {Q[0].tolist()}")
    if bits_of(s[0]) != int(c["scale0_bits"], 16):
        fails.append(f"WE5: scale {hex(bits_of(s[0]))}")
    if bits_of(z[0]) != int(c["zero0_bits"], 16):
        fails.append(f"WE5: zero {hex(bits_of(z[0]))}")
    if [bits_of(v) for v in r[0][:2]] != [int(h, 16) for h in c["resid0_bits_first_two"]]:
        fails.append("WE5: residual signs")

    c = cases["WE6_all_negative_zero"]
    x = np.array([f32_from_bits(h) for h in c["x_bits"]], np.float32)
    Q, s, z, r = orc.quantize_group(x, 4)
    if [bits_of(v) for v in s] != [int(h, 16) for h in c["scale_bits"]] or \
       [bits_of(v) for v in z] != [int(h, 16) for h in c["zero_bits"]] or Q.any():
        fails.append(f"WE6: scales {[hex(bits_of(v)) for v in s]} zeros {[hex(bits_of(v)) for v in z]}")
    return fails


# ---------------------------------------------------------------------------
# brute force: nearest level in exact arithmetic
# ---------------------------------------------------------------------------
def _exact_dyadic_groups(rng, count):
    """Groups where every binary32 step is exact: lo = a/16, s = 2^e, values
    lo + m*2^(e-2) for m in 0..12 with both ends present.  Then d/s = m/4
    exactly and ties (m/4 = 0.5, 1.5, 2.5) are exact."""
    out = []
    for _ in range(count):
        g = int(rng.integers(2, 17))
        e = int(rng.integers(-4, 2))
        lo = Fraction(int(rng.integers(-16, 17)), 16)
        ms = list(rng.integers(0, 13, size=g))
        ms[0], ms[-1] = 0, 12
        rng.shuffle(ms)
        xs = [lo + Fraction(int(m)) * Fraction(2) ** (e - 2) for m in ms]
        out.append((xs, lo, Fraction(2) ** e, [int(m) for m in ms]))
    return out


def pin_brute_force_exact(orc, seed=7, count=300) -> list[str]:
    rng = np.random.default_rng(seed)
    fails = []
    for xs, lo, s, ms in _exact_dyadic_groups(rng, count):
        x = np.array([float(v) for v in xs], np.float32)
        Q, sc, z, r = orc.quantize_group(x, 1)
        if Fraction(float(sc[0])) != s or Fraction(float(z[0])) != lo:
            fails.append(f"exact grid: s={sc[0]} z={z[0]} want {float(s)} {float(lo)}")
            continue
        for j, v in enumerate(xs):
            dist = [abs(v - (lo + q * s)) for q in range(4)]
            best = min(dist)
            cands = [q for q in range(4) if dist[q] == best]
            want = cands[0] if len(cands) == 1 else [q for q in cands if q % 2 == 0][0]
            if int(Q[0, j]) != want:
                fails.append(f"nearest level: x={float(v)} lo={float(lo)} s={float(s)} "
                             f"Q={int(Q[0, j])} want {want}")
                break
            if Fraction(float(r[0, j])) != v - (lo + want * s):
                fails.append(f"exact residual wrong at x={float(v)}")
                break
        if len(fails) > 5:
            break
    return fails


def pin_brute_force_tiny(orc) -> list[str]:
    """All groups of 3 values over a small bf16 alphabet: at every stage each
    code picks a level whose distance to the value is the minimum over the
    four levels, up to a few units in the last place of the arithmetic."""
    alphabet = [-1.0, -0.75, -0.3125, 0.0, 0.125, 0.5, 0.6875, 1.0, 1.375]
    fails = []
    for a in alphabet:
        for b in alphabet:
            for c in alphabet:
                x = np.array([a, b, c], np.float32)
                Q, s, z, r = orc.quantize_group(x, 4)
                v = x.astype(np.float64)
                for k in range(4):
                    lv = [float(np.float32(z[k]) + np.float32(np.float32(q) * s[k])) for q in range(4)]
                    tol = 4 * float(np.spacing(np.float32(max(abs(z[k]), s[k] * 4, 1e-30))))
                    for j in range(3):
                        d = [abs(v[j] - lv[q]) for q in range(4)]
                        if d[int(Q[k, j])] > min(d) + tol:
                            fails.append(f"tiny x={x.tolist()} stage {k} elem {j}: Q={Q[k, j]} d={d}")
                    v = r[k].astype(np.float64)
                if len(fails) > 5:
                    return fails
    return fails


# ---------------------------------------------------------------------------
# invariants
# ---------------------------------------------------------------------------
def _random_groups(rng, count, g):
    """Gaussian, heavy-tailed (Student-t, 3 dof) and outlier-injected groups,
    rounded to bf16 like real weights."""
    out = []
    for i in range(count):
        kind = i % 3
        if kind == 0:
            x = rng.normal(0, 0.02, g)
        elif kind == 1:
            x = rng.standard_t(3, g) * 0.02 / np.sqrt(3)
        else:
            x = rng.normal(0, 0.02, g)
            x[rng.integers(0, g)] = 0.4 * (1 if rng.random() < 0.5 else -1)
        x = x.astype(np.float32)
        u = x.view(np.uint32)
        u = ((u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000).astype(np.uint32)
        out.append(u.view(np.float32))
    return out


def pin_invariants(orc, seed=11, count=120, g=128) -> list[str]:
    rng = np.random.default_rng(seed)
    fails = []
    for x in _random_groups(rng, count, g):
        Q, s, z, r = orc.quantize_group(x, 4)
        prev = x.astype(np.float64)
        prev_max = float(np.max(np.abs(x)))
        for k in range(4):
            sk, lo = float(s[k]), float(z[k])
            if lo != float(np.min(prev)):
                fails.append(f"stage {k}: zero {lo} is not the group minimum {np.min(prev)}")
            hi = float(np.max(prev))
            if abs(sk - (hi - lo) / 3) > 2 ** -22 * (hi - lo) + 1e-45:
                fails.append(f"stage {k}: scale {sk} is not (max-min)/3")
            # half-step bound (Eq. 3 with nearest rounding)
            bound = 0.5 * sk + 2 ** -21 * (abs(lo) + 4 * sk) + 1e-45
            rk = r[k].astype(np.float64)
            if np.max(np.abs(rk)) > bound:
                fails.append(f"stage {k}: |residual| {np.max(np.abs(rk))} > half step {0.5*sk}")
            # residual = previous value - dequantized level (Eq. 5/7)
            lev = lo + Q[k].astype(np.float64) * sk
            if np.max(np.abs(prev - lev - rk)) > 2 ** -20 * (abs(lo) + 4 * sk) + 1e-45:
                fails.append(f"stage {k}: residual is not value minus level")
            # L-infinity error shrinks at least 3x per stage (up to rounding)
            cur_max = float(np.max(np.abs(rk)))
            if cur_max > prev_max / 3 * (1 + 2 ** -18) + 2 ** -20 * (abs(lo) + 4 * sk):
                fails.append(f"stage {k}: max|r| {cur_max} > max|r_prev|/3 {prev_max/3}")
            prev, prev_max = rk, cur_max
        if len(fails) > 5:
            break
    return fails


def pin_exact_grid(orc, seed=5, count=60, g=128) -> list[str]:
    """A group whose values lie on {a, a+d, a+2d, a+3d} and include both ends
    reconstructs exactly from the base stage alone (k = 1)."""
    rng = np.random.default_rng(seed)
    fails = []
    for _ in range(count):
        a = int(rng.integers(-60, 61)) / 1024.0
        d = int(rng.integers(1, 64)) / 1024.0
        q = rng.integers(0, 4, g)
        q[0], q[-1] = 0, 3
        x = (a + q * d).astype(np.float32)
        W = bf16_bits_of_f32(x).reshape(1, g)
        codes, scales, zeros = orc.quantize(W, group=g, n_stages=4)
        rec = orc.reconstruct(codes, scales, zeros, 1, g, g, 1)[0]
        if not np.array_equal(rec, W[0]):
            fails.append(f"exact grid a={a} d={d} not reconstructed at k=1")
        Qg, _, _, r = orc.quantize_group(x, 1)
        if not np.array_equal(Qg[0], q.astype(np.uint8)):
            fails.append(f"exact grid a={a} d={d}: codes differ from grid indices")
        if len(fails) > 5:
            break
    return fails


def pin_prefix_reconstruction(orc, seed=3, rows=6, g=64) -> list[str]:
    """Eq. 8: the prefix-k reconstruction equals x minus the residual after
    stage k-1, up to fp32 summation rounding and the final bf16 rounding;
    packed codes agree with the per-group codes (byte c/4, bits 2*(c%4))."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 3 * g
    xs = np.concatenate(_random_groups(rng, rows * 3, g)).reshape(rows, cols)
    W = bf16_bits_of_f32(xs)
    codes, scales, zeros = orc.quantize(W, group=g, n_stages=4)
    n = rows * cols
    for gi in range(n // g):
        x = xs.reshape(-1)[gi * g:(gi + 1) * g]
        Q, s, z, r = orc.quantize_group(x, 4)
        for k in range(4):
            c = np.arange(gi * g, (gi + 1) * g)
            unpacked = (codes[k][c // 4] >> (2 * (c % 4))) & 3
            if not np.array_equal(unpacked, Q[k]):
                fails.append(f"group {gi} stage {k}: packed codes disagree")
            if bits_of(scales[k][gi]) != bits_of(s[k]) or bits_of(zeros[k][gi]) != bits_of(z[k]):
                fails.append(f"group {gi} stage {k}: metadata disagrees")
    for k in range(1, 5):
        rec = orc.reconstruct(codes, scales, zeros, rows, cols, g, k).reshape(-1)
        recf = (rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        for gi in range(n // g):
            x = xs.reshape(-1)[gi * g:(gi + 1) * g].astype(np.float64)
            _, s, z, r = orc.quantize_group(x.astype(np.float32), 4)
            want = x - r[k - 1]
            err = np.abs(recf[gi * g:(gi + 1) * g] - want)
            tol = np.abs(want) * 2 ** -8 + 8 * 2 ** -24 * (np.abs(x).max() + 1e-30)
            if np.any(err > tol):
                fails.append(f"group {gi}: prefix k={k} is not x - r_(k-1)")
                break
    return fails


def pin_bf16_rounding(orc, seed=13, count=4000) -> list[str]:
    """The oracle's float -> bf16 conversion is round-to-nearest-even, the
    same as torch's CPU conversion (a library routine), on random values,
    exact ties and the overflow edge."""
    import torch
    rng = np.random.default_rng(seed)
    u = rng.integers(0, 2 ** 32, count, dtype=np.uint64).astype(np.uint32)
    u = u[(u & 0x7F800000) != 0x7F800000]  # finite only
    ties = (rng.integers(0, 2 ** 15, 200).astype(np.uint32) << 16) | 0x8000
    ties = ties[(ties & 0x7F800000) != 0x7F800000]
    u = np.concatenate([u, ties, np.array([0x7F7FFFFF, 0x7F7F8000, 0x00008000, 0x80018000], np.uint32)])
    f = u.view(np.float32)
    want = torch.from_numpy(f.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([orc.f32_to_bf16(float(v)) for v in f], np.uint16)
    bad = np.nonzero(got != want)[0]
    return [f"bf16({hex(int(u[i]))}) = {hex(int(got[i]))}, want {hex(int(want[i]))}" for i in bad[:5]]


ALL_PINS = [pin_worked_groups, pin_bf16_rounding, pin_brute_force_exact, pin_brute_force_tiny,
            pin_invariants, pin_exact_grid, pin_prefix_reconstruction]


def all_failures(orc) -> list[str]:
    out = []
    for p in ALL_PINS:
        try:
            out += [f"{p.__name__}: {m}" for m in p(orc)]
        except Exception as e:  # a crash of a mutated oracle counts as caught
            out.append(f"{p.__name__}: raised {type(e).__name__}: {e}")
    return out
