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
    per stage (Eq. 5-8), prefix reconstruction equal to input minus residual;
  * library conversions: bf16 rounding against torch, binary16 rounding
    against numpy's float16.
The symmetric grid (levels (Q-2)s, s = 2 max|x| / 3, binary32 or binary16
scales) has its own worked groups, brute force and invariants below.
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


def bf16_round_bits(x) -> np.ndarray:
    """bf16 bit patterns of float32 values rounded to nearest-even."""
    u = np.asarray(x, np.float32).view(np.uint32)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


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


def pin_f16_rounding(orc, seed=17, count=6000) -> list[str]:
    """The oracle's binary32 -> binary16 conversion is IEEE round-to-nearest-
    even with subnormals and overflow to infinity, the same as numpy's
    float16 cast (a library routine): random values across the whole binary16
    range, exact ties (normal and subnormal), and the edges 65504 / 65520 /
    2^-24 / 2^-25.  binary16 -> binary32 is checked for every finite pattern."""
    rng = np.random.default_rng(seed)
    fails = []
    # random binary32 values whose exponent lands around the binary16 range
    e = rng.integers(127 - 30, 127 + 17, count).astype(np.uint32)
    u = (rng.integers(0, 2, count).astype(np.uint32) << 31) | (e << 23) | \
        rng.integers(0, 2 ** 23, count).astype(np.uint32)
    # exact ties: a binary16 value plus half its spacing
    h = rng.integers(0, 0x7BFF, 400).astype(np.uint16)
    lo = h.view(np.float16).astype(np.float64)
    hi = (h + 1).astype(np.uint16).view(np.float16).astype(np.float64)
    ties = ((lo + hi) / 2).astype(np.float32)  # exact: at most 12 significant bits
    edges = np.array([65504.0, 65519.99, 65520.0, 65536.0, 2.0 ** -24, 2.0 ** -25,
                      2.0 ** -25 * 1.0000001, 3 * 2.0 ** -26, 2.0 ** -14, 0.0, -0.0, 1e-30],
                     np.float32)
    f = np.concatenate([u.view(np.float32), ties, -ties, edges])
    with np.errstate(over="ignore"):
        want = f.astype(np.float16).view(np.uint16)
    got = np.array([orc.f32_to_f16(float(v)) for v in f], np.uint16)
    for i in np.nonzero(got != want)[0][:5]:
        fails.append(f"f16({f[i]!r}) = {hex(int(got[i]))}, want {hex(int(want[i]))}")
    allh = np.arange(0, 0x10000, dtype=np.uint32).astype(np.uint16)
    allh = allh[(allh & 0x7C00) != 0x7C00]
    wantf = allh.view(np.float16).astype(np.float32)
    gotf = np.array([orc.f16_to_f32(int(x)) for x in allh], np.float32)
    bad = np.nonzero(gotf.view(np.uint32) != wantf.view(np.uint32))[0]
    for i in bad[:5]:
        fails.append(f"f16 decode {hex(int(allh[i]))} = {gotf[i]!r}, want {wantf[i]!r}")
    return fails


# ---------------------------------------------------------------------------
# symmetric grid: hand-worked groups
# ---------------------------------------------------------------------------
# WS1 (binary32 scales), x = [-1.5, -1, 0.5, 1.5]:
#   stage 0: amax = 1.5, s = fl(3/3) = 1; x/s = -1.5 -> rhe -2 -> Q 0;
#            -1 -> Q 1; 0.5 -> rhe 0 (tie to even) -> Q 2; 1.5 -> rhe 2 ->
#            Q 4, clamped to 3 (level s = 1).  r = [0.5, 0, 0.5, 0.5].
#   stage 1: amax = 0.5, s = fl(1/3) = 0x3EAAAAAB; fl(0.5/s) = 1.5 exactly
#            (0.49999998 / 0.33333334 = 1.49999996, within half an ulp of
#            1.5), so rhe gives 2 and the clamp 3; 0 -> Q 2.
#            r = 0.5 - s = 0x3E2AAAAA (exact), and 0.
#   prefix k=1: (Q-2)s = [-2, -1, 0, 1]; k=2 adds [s, 0, s, s]:
#            fl(-2 + s) = 0xBFD55555 -> bf16 0xBFD5; s -> 0x3EAB;
#            fl(1 + s) = 0x3FAAAAAB -> 0x3FAB.
WS1 = dict(x=[-1.5, -1.0, 0.5, 1.5], Q=[[0, 1, 2, 3], [3, 2, 3, 3]],
           scale_bits=[0x3F800000, 0x3EAAAAAB],
           resid_bits=[[0x3F000000, 0x00000000, 0x3F000000, 0x3F000000],
                       [0x3E2AAAAA, 0x00000000, 0x3E2AAAAA, 0x3E2AAAAA]],
           recon=[[0xC000, 0xBF80, 0x0000, 0x3F80], [0xBFD5, 0xBF80, 0x3EAB, 0x3FAB]])
# WS2 (binary16 scales), a = 0.10009765625 = 1640 * 2^-14 (bf16 0x3DCD),
# x = [a, 0, -a, a/2]:
#   stage 0: fl(2a/3) = 0.066731770..., as binary16 (spacing 2^-14 in
#            [2^-4, 2^-3)) 1093.33 * 2^-14 -> 1093 * 2^-14 = 0x2C45.
#            In units of 2^-14: 1640/1093 = 1.5005 -> rhe 2 -> Q 3, r = 547;
#            0 -> Q 2, r = 0; -1.5005 -> rhe -2 -> Q 0, r = -1640 + 2186 = 546;
#            820/1093 = 0.750 -> rhe 1 -> Q 3, r = 820 - 1093 = -273.
#            (547 > 1093/2: rounding the scale down to binary16 lets the top
#            element exceed the half step.)
#   stage 1: amax = 547 * 2^-14; fl(2*547/3 * 2^-14) in binary16 (spacing
#            2^-16 in [2^-6, 2^-5)): 1458.67 * 2^-16 -> 1459 * 2^-16 = 0x25B3.
#            In units of 2^-16, r = [2188, 0, 2184, -1092]:
#            2188/1459 = 1.4997 -> rhe 1 -> Q 3, r = 729; 0 -> Q 2;
#            2184/1459 = 1.4969 -> Q 3, r = 725; -1092/1459 = -0.748 -> rhe -1
#            -> Q 1, r = -1092 + 1459 = 367.
WS2 = dict(x=[0.10009765625, 0.0, -0.10009765625, 0.050048828125],
           Q=[[3, 2, 0, 3], [3, 2, 3, 1]], scale_f16=[0x2C45, 0x25B3],
           resid=[[547 * 2.0 ** -14, 0.0, 546 * 2.0 ** -14, -273 * 2.0 ** -14],
                  [729 * 2.0 ** -16, 0.0, 725 * 2.0 ** -16, 367 * 2.0 ** -16]])
# WS3: x = [-3, -1, 0.75, 1.5]: amax 3, s = 2; x/s = [-1.5, -0.5, 0.375, 0.75]
#   -> rhe [-2, -0 (tie to even), 0, 1] -> Q [0, 2, 2, 3];
#   levels [-4, 0, 0, 2], r = [1, -1, 0.75, -0.5] (|r| = s/2 at the ties).
WS3 = dict(x=[-3.0, -1.0, 0.75, 1.5], Q0=[0, 2, 2, 3], scale0=2.0, resid0=[1.0, -1.0, 0.75, -0.5])


def pin_sym_worked_groups(orc) -> list[str]:
    fails = []
    Q, s, r = orc.quantize_group_sym(np.array(WS1["x"], np.float32), 2, False)
    if Q.tolist() != WS1["Q"]:
        fails.append(f"WS1: codes {Q.tolist()}")
    if [bits_of(v) for v in s] != WS1["scale_bits"]:
        fails.append(f"WS1: scales {[hex(bits_of(v)) for v in s]}")
    if [[bits_of(v) for v in row] for row in r] != WS1["resid_bits"]:
        fails.append(f"WS1: residuals {[[hex(bits_of(v)) for v in row] for row in r]}")
    W = bf16_bits_of_f32(np.array(WS1["x"], np.float32)).reshape(1, 4)
    codes, scales = orc.quantize_sym(W, group=4, n_stages=2, scale_f16=False)
    for k in (1, 2):
        rec = orc.reconstruct_sym(codes, scales, 1, 4, 4, k, scale_f16=False)[0]
        if rec.tolist() != WS1["recon"][k - 1]:
            fails.append(f"WS1: recon k={k} {[hex(v) for v in rec]}")

    Q, s, r = orc.quantize_group_sym(np.array(WS2["x"], np.float32), 2, True)
    if Q.tolist() != WS2["Q"]:
        fails.append(f"WS2: codes {Q.tolist()}")
    if [orc.f32_to_f16(float(v)) for v in s] != WS2["scale_f16"]:
        fails.append(f"WS2: scales {[float(v) for v in s]}")
    if r.astype(np.float64).tolist() != WS2["resid"]:
        fails.append(f"WS2: residuals {r.tolist()}")
    W = bf16_bits_of_f32(np.array(WS2["x"], np.float32)).reshape(1, 4)
    codes, scales = orc.quantize_sym(W, group=4, n_stages=2, scale_f16=True)
    if [int(a[0]) for a in scales] != WS2["scale_f16"]:
        fails.append(f"WS2: stored binary16 scales {[hex(int(a[0])) for a in scales]}")
    packed = [int(c[0]) for c in codes]
    want = [sum(q << (2 * j) for j, q in enumerate(row)) for row in WS2["Q"]]
    if packed != want:
        fails.append(f"WS2: packed {packed} != {want}")

    Q, s, r = orc.quantize_group_sym(np.array(WS3["x"], np.float32), 1, False)
    if Q[0].tolist() != WS3["Q0"] or float(s[0]) != WS3["scale0"] or r[0].tolist() != WS3["resid0"]:
        fails.append(f"WS3: {Q[0].tolist()} {s[0]} {r[0].tolist()}")

    # signed zeros only: s = 0, every code 2, residual keeps each sign,
    # reconstruction +0
    x = np.array([-0.0, 0.0, -0.0, 0.0], np.float32)
    for f16 in (False, True):
        Q, s, r = orc.quantize_group_sym(x, 4, f16)
        if (Q != 2).any() or (s != 0).any() or [bits_of(v) for v in r[3]] != [0x80000000, 0, 0x80000000, 0]:
            fails.append(f"zero group f16={f16}: {Q.tolist()} {s.tolist()} {[hex(bits_of(v)) for v in r[3]]}")
    return fails


# ---------------------------------------------------------------------------
# symmetric grid: brute force and invariants
# ---------------------------------------------------------------------------
def pin_sym_brute_force_exact(orc, seed=19, count=300) -> list[str]:
    """Dyadic groups with amax = 1.5 * 2^e, so s = 2^e exactly (also as
    binary16), and values m * 2^(e-2), |m| <= 6: every step is exact.  Each
    code must select the level of {-2s, -s, 0, s} nearest the value, an exact
    tie going to the even code, and the residual must be exact."""
    rng = np.random.default_rng(seed)
    fails = []
    for _ in range(count):
        g = int(rng.integers(2, 17))
        e = int(rng.integers(-6, 4))
        ms = list(rng.integers(-6, 7, size=g))
        ms[0] = 6 if rng.random() < 0.5 else -6
        rng.shuffle(ms)
        s = Fraction(2) ** e
        xs = [Fraction(int(m)) * Fraction(2) ** (e - 2) for m in ms]
        x = np.array([float(v) for v in xs], np.float32)
        for f16 in (False, True):
            Q, sc, r = orc.quantize_group_sym(x, 1, f16)
            if Fraction(float(sc[0])) != s:
                fails.append(f"sym exact: s={sc[0]} want {float(s)}")
                break
            for j, v in enumerate(xs):
                dist = [abs(v - (q - 2) * s) for q in range(4)]
                best = min(dist)
                cands = [q for q in range(4) if dist[q] == best]
                want = cands[0] if len(cands) == 1 else [q for q in cands if q % 2 == 0][0]
                if int(Q[0, j]) != want:
                    fails.append(f"sym nearest level: x={float(v)} s={float(s)} Q={int(Q[0, j])} want {want}")
                    break
                if Fraction(float(r[0, j])) != v - (want - 2) * s:
                    fails.append(f"sym exact residual wrong at x={float(v)}")
                    break
        if len(fails) > 5:
            break
    return fails


def _is_f16(v) -> bool:
    return float(np.float32(v).astype(np.float16)) == float(v)


def pin_sym_invariants(orc, seed=23, count=120, g=128) -> list[str]:
    """Random bf16 groups (Gaussian, Student-t, outliers), 4 stages:
    s_k = 2 max|r_{k-1}| / 3 to binary32 rounding (binary16: to half a
    binary16 spacing, and representable); |r_k| <= s_k / 2 up to rounding
    (binary16: up to the scale's relative rounding, 2^-11, times 1.5);
    max |r_k| <= max |r_{k-1}| / 3 up to the same; codes in 0..3."""
    rng = np.random.default_rng(seed)
    fails = []
    for x in _random_groups(rng, count, g):
        for f16 in (False, True):
            Q, s, r = orc.quantize_group_sym(x, 4, f16)
            prev = x.astype(np.float64)
            for k in range(4):
                amax = float(np.max(np.abs(prev)))
                sk = float(s[k])
                ideal = 2 * amax / 3
                rel = 2.0 ** -11 if f16 else 2.0 ** -23
                if abs(sk - ideal) > rel * ideal * 1.01 + (2.0 ** -25 if f16 else 1e-45):
                    fails.append(f"sym stage {k} f16={f16}: scale {sk} vs 2*amax/3 {ideal}")
                if f16 and not _is_f16(sk):
                    fails.append(f"sym stage {k}: scale {sk} not a binary16 value")
                rk = r[k].astype(np.float64)
                slack = 3 * rel + 2.0 ** -22
                if np.max(np.abs(rk)) > 0.5 * sk * (1 + slack) + 1e-45:
                    fails.append(f"sym stage {k} f16={f16}: |r| {np.max(np.abs(rk))} > s/2 {0.5 * sk}")
                if np.max(np.abs(rk)) > amax / 3 * (1 + 2 * slack) + 1e-45:
                    fails.append(f"sym stage {k} f16={f16}: max|r| not reduced 3x")
                lev = (Q[k].astype(np.float64) - 2) * sk
                if np.max(np.abs(prev - lev - rk)) > 2.0 ** -23 * amax + 1e-45:
                    fails.append(f"sym stage {k}: residual is not value minus level")
                prev = rk
            if len(fails) > 5:
                return fails
    return fails


def pin_sym_prefix_reconstruction(orc, seed=29, rows=5, g=64) -> list[str]:
    """Eq. 8 for the symmetric package: packed codes and stored scales equal
    the per-group results (binary16 scales stored as their bit patterns), and
    the prefix-k reconstruction is x minus the residual after stage k-1 up to
    summation and bf16 rounding."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 3 * g
    xs = np.concatenate(_random_groups(rng, rows * 3, g)).reshape(rows, cols)
    W = bf16_bits_of_f32(xs)
    n = rows * cols
    for f16 in (False, True):
        codes, scales = orc.quantize_sym(W, group=g, n_stages=4, scale_f16=f16)
        resid = []
        for gi in range(n // g):
            x = xs.reshape(-1)[gi * g:(gi + 1) * g]
            Q, s, r = orc.quantize_group_sym(x, 4, f16)
            resid.append(r)
            c = np.arange(gi * g, (gi + 1) * g)
            for k in range(4):
                if not np.array_equal((codes[k][c // 4] >> (2 * (c % 4))) & 3, Q[k]):
                    fails.append(f"sym group {gi} stage {k}: packed codes disagree")
                stored = orc.f16_to_f32(int(scales[k][gi])) if f16 else float(scales[k][gi])
                if bits_of(stored) != bits_of(s[k]):
                    fails.append(f"sym group {gi} stage {k}: stored scale disagrees")
        for k in range(1, 5):
            rec = orc.reconstruct_sym(codes, scales, rows, cols, g, k, scale_f16=f16).reshape(-1)
            recf = (rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
            for gi in range(n // g):
                x = xs.reshape(-1)[gi * g:(gi + 1) * g].astype(np.float64)
                want = x - resid[gi][k - 1]
                err = np.abs(recf[gi * g:(gi + 1) * g] - want)
                tol = np.abs(want) * 2 ** -8 + 8 * 2 ** -24 * (np.abs(x).max() + 1e-30)
                if np.any(err > tol):
                    fails.append(f"sym group {gi} f16={f16}: prefix k={k} is not x - r_(k-1)")
                    break
    return fails


# ---------------------------------------------------------------------------
# Algorithm 1 with a base checkpoint
# ---------------------------------------------------------------------------
# WB1 (asymmetric), x = [-1, 0, 0.5, 2], given base: every code 0, scale 1,
# zero -1 (not the RTN base): L0 = -1 for all, R0 = [0, 1, 1.5, 3].
#   stage 1: lo 0, hi 3, s 1, codes rhe([0, 1, 1.5, 3]) = [0, 1, 2, 3] (1.5 ties
#            to 2), r = [0, 0, -0.5, 0];
#   stage 2: lo -0.5, hi 0, s = fl(0.5/3) = 0x3E2AAAAB; fl(0.5/s) = 3 exactly
#            (2.99999991 rounds up), so Q = [3, 3, 0, 3]; fl(3s) = 0.5, level
#            -0.5 + 0.5 = 0, r = +0 everywhere;
#   stage 3: constant +0 group, s = 0, zero +0, codes 0.
#   prefixes: k=1 [-1]*4; k=2 [-1, 0, 1, 2]; k=3 = x.
WB1 = dict(x=[-1.0, 0.0, 0.5, 2.0], base=([0x00], [1.0], [-1.0]),
           Q=[[0, 1, 2, 3], [3, 3, 0, 3], [0, 0, 0, 0]],
           scale_bits=[0x3F800000, 0x3E2AAAAB, 0x00000000], zero_bits=[0x00000000, 0xBF000000, 0x00000000],
           recon=[[0xBF80] * 4, [0xBF80, 0x0000, 0x3F80, 0x4000], [0xBF80, 0x0000, 0x3F00, 0x4000]])
# WB2 (symmetric, binary16), x = [0.75, -0.25, 0.5, -1], given base codes
# [3, 2, 3, 0] with scale 0.5 (0x3800): L0 = (Q-2) 0.5 = [0.5, 0, 0.5, -1],
# R0 = [0.25, -0.25, +0, +0].
#   stage 1: amax 0.25, fl(0.5/3) as binary16 (spacing 2^-13 in [1/8, 1/4)):
#            1365.33 -> 1365 * 2^-13 = 0x3155.  In units of 2^-13: 2048/1365 =
#            1.5004 -> rhe 2 -> clamped Q 3, r = 2048 - 1365 = 683;
#            -1.5004 -> rhe -2 -> Q 0, r = -2048 + 2730 = 682; zeros -> Q 2.
WB2 = dict(x=[0.75, -0.25, 0.5, -1.0], base=([3 | (2 << 2) | (3 << 4) | (0 << 6)], [0x3800]),
           Q1=[3, 0, 2, 2], scale1=0x3155)


def _as_base(codes_byte, scales, zeros=None, f16=False):
    return (np.array(codes_byte, np.uint8), np.array(scales, np.uint16 if f16 else np.float32),
            None if zeros is None else np.array(zeros, np.float32))


def pin_base_worked_groups(orc) -> list[str]:
    fails = []
    W = bf16_bits_of_f32(np.array(WB1["x"], np.float32)).reshape(1, 4)
    codes, scales, zeros = orc.quantize_from_base(W, _as_base(*WB1["base"]), group=4, n_stages=4)
    got_q = [[int((codes[k][0] >> (2 * j)) & 3) for j in range(4)] for k in (1, 2, 3)]
    if got_q != WB1["Q"]:
        fails.append(f"WB1: codes {got_q}")
    if [bits_of(scales[k][0]) for k in (1, 2, 3)] != WB1["scale_bits"]:
        fails.append(f"WB1: scales {[hex(bits_of(scales[k][0])) for k in (1, 2, 3)]}")
    if [bits_of(zeros[k][0]) for k in (1, 2, 3)] != WB1["zero_bits"]:
        fails.append(f"WB1: zeros {[hex(bits_of(zeros[k][0])) for k in (1, 2, 3)]}")
    for k in (1, 2, 3):
        rec = orc.reconstruct(codes, scales, zeros, 1, 4, 4, k)[0]
        if rec.tolist() != WB1["recon"][k - 1]:
            fails.append(f"WB1: recon k={k} {[hex(v) for v in rec]}")

    W = bf16_bits_of_f32(np.array(WB2["x"], np.float32)).reshape(1, 4)
    codes, scales, _ = orc.quantize_from_base(W, _as_base(*WB2["base"], f16=True), group=4,
                                              n_stages=2, sym=True, scale_f16=True)
    got = [int((codes[1][0] >> (2 * j)) & 3) for j in range(4)]
    if got != WB2["Q1"] or int(scales[1][0]) != WB2["scale1"]:
        fails.append(f"WB2: codes {got} scale {hex(int(scales[1][0]))}")
    if int(codes[0][0]) != WB2["base"][0][0] or int(scales[0][0]) != WB2["base"][1][0]:
        fails.append("WB2: the given base was not kept as stage 0")
    return fails


def pin_base_branch_equivalence(orc, seed=31, rows=4, g=64) -> list[str]:
    """Algorithm 1's two branches are one recursion once the base is fixed:
    given the base stage the build itself computes (RTN), the checkpoint
    branch yields the same residual stages, for every format."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 4 * g
    xs = np.concatenate(_random_groups(rng, rows * 4, g)).reshape(rows, cols)
    W = bf16_bits_of_f32(xs)
    c, s, z = orc.quantize(W, group=g, n_stages=4)
    c2, s2, z2 = orc.quantize_from_base(W, (c[0], s[0], z[0]), group=g, n_stages=4)
    for k in range(4):
        if not (np.array_equal(c[k], c2[k]) and np.array_equal(s[k].view(np.uint32), s2[k].view(np.uint32))
                and np.array_equal(z[k].view(np.uint32), z2[k].view(np.uint32))):
            fails.append(f"asym: stage {k} differs between the two branches")
    for f16 in (False, True):
        c, s = orc.quantize_sym(W, group=g, n_stages=4, scale_f16=f16)
        c2, s2, _ = orc.quantize_from_base(W, (c[0], s[0], None), group=g, n_stages=4, sym=True, scale_f16=f16)
        for k in range(4):
            if not (np.array_equal(c[k], c2[k]) and np.array_equal(s[k].view(np.uint8), s2[k].view(np.uint8))):
                fails.append(f"sym f16={f16}: stage {k} differs between the two branches")
    return fails


def pin_base_residual_invariants(orc, seed=37, rows=3, g=128) -> list[str]:
    """With an arbitrary given base (random codes, scales and zeros), the
    prefix-1 reconstruction is the base's own dequantization, and every
    residual stage obeys the half-step bound relative to the range of what it
    quantizes, so the reconstruction error of the last prefix is at most half
    of the last stage's step (asymmetric grid)."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 2 * g
    xs = np.concatenate(_random_groups(rng, rows * 2, g)).reshape(rows, cols)
    W = bf16_bits_of_f32(xs)
    n = rows * cols
    base = (rng.integers(0, 256, n // 4).astype(np.uint8),
            rng.uniform(0.001, 0.05, n // g).astype(np.float32),
            rng.uniform(-0.1, 0.0, n // g).astype(np.float32))
    codes, scales, zeros = orc.quantize_from_base(W, base, group=g, n_stages=4)
    rec1 = orc.reconstruct(codes, scales, zeros, rows, cols, g, 1).reshape(-1)
    c = np.arange(n)
    q0 = (base[0][c // 4] >> (2 * (c % 4))) & 3
    lev = (base[2][c // g] + (q0.astype(np.float32) * base[1][c // g]).astype(np.float32)).astype(np.float32)
    want1 = ((lev.view(np.uint32) + 0x7FFF + ((lev.view(np.uint32) >> 16) & 1)) >> 16).astype(np.uint16)
    if not np.array_equal(rec1, want1):
        fails.append("prefix 1 is not the given base's dequantization")
    rec4 = orc.reconstruct(codes, scales, zeros, rows, cols, g, 4).reshape(-1)
    recf = (rec4.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    err = np.abs(recf - xs.reshape(-1).astype(np.float64))
    bound = 0.5 * scales[3][c // g].astype(np.float64) * (1 + 2 ** -20) + \
        np.abs(xs.reshape(-1)) * 2 ** -8 + 2 ** -30
    if np.any(err > bound):
        fails.append(f"last-prefix error {err.max()} exceeds half the last step")
    return fails


# ---------------------------------------------------------------------------
# stage-wise product with the prefix weights (Appendix C)
# ---------------------------------------------------------------------------
# GV1: the WE1 package (x = [-1, 0, 0.5, 2]; prefix 1 = [-1, 0, 1, 2], prefix 2
# = x exactly) times A = [[2, -1, 4, 0.25], [1, 1, 1, 1]]:
#   k=1: [-2 + 0 + 4 + 0.5, -1 + 0 + 1 + 2] = [2.5, 2];  k=2: [-2 + 0 + 2 + 0.5, 1.5].
# GV2: the WS1 symmetric package (x = [-1.5, -1, 0.5, 1.5], binary32 scales),
#   k=1 levels [-2, -1, 0, 1] -> A[0] . = -4 + 1 + 0 + 0.25 = -2.75.
GV_A = [[2.0, -1.0, 4.0, 0.25], [1.0, 1.0, 1.0, 1.0]]


def pin_gemv_worked(orc) -> list[str]:
    fails = []
    A = bf16_bits_of_f32(np.array(GV_A, np.float32))
    W = bf16_bits_of_f32(np.array([-1.0, 0.0, 0.5, 2.0], np.float32)).reshape(1, 4)
    codes, scales, zeros = orc.quantize(W, group=4, n_stages=2)
    for k, want in ((1, [2.5, 2.0]), (2, [0.5, 1.5])):
        Y = orc.gemv(codes, scales, zeros, 1, 4, 4, k, A)
        if Y[:, 0].tolist() != want:
            fails.append(f"GV1 k={k}: {Y[:, 0].tolist()} != {want}")
    W = bf16_bits_of_f32(np.array(WS1["x"], np.float32)).reshape(1, 4)
    codes, scales = orc.quantize_sym(W, group=4, n_stages=2, scale_f16=False)
    Y = orc.gemv(codes, scales, None, 1, 4, 4, 1, A[:1], sym=True)
    if Y[0, 0] != -2.75:
        fails.append(f"GV2: {Y[0, 0]} != -2.75")
    return fails


def pin_gemv_is_input_minus_residual(orc, seed=41, rows=6, g=64) -> list[str]:
    """Eq. 8 with Eq. 5-7 in product form: A W~_(k) = A X - A R_(k-1) (the
    prefix-k weight is the input minus the residual after stage k-1, taken
    from the stage-by-stage quantizer), up to the binary32 rounding of the
    stage sums; for every format."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 3 * g
    xs = np.concatenate(_random_groups(rng, rows * 3, g)).reshape(rows, cols)
    W = bf16_bits_of_f32(xs)
    A = bf16_round_bits(rng.normal(0, 1, (3, cols)).astype(np.float32))
    Af = (A.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    for sym, f16 in ((False, False), (True, False), (True, True)):
        if sym:
            codes, scales = orc.quantize_sym(W, group=g, n_stages=4, scale_f16=f16)
            zeros = None
        else:
            codes, scales, zeros = orc.quantize(W, group=g, n_stages=4)
        resid = []
        for gi in range(rows * cols // g):
            x = xs.reshape(-1)[gi * g:(gi + 1) * g]
            r = orc.quantize_group_sym(x, 4, f16)[2] if sym else orc.quantize_group(x, 4)[3]
            resid.append(r)
        resid = np.concatenate(resid, axis=1).astype(np.float64)  # [4, n]
        for k in range(1, 5):
            Y = orc.gemv(codes, scales, zeros, rows, cols, g, k, A, sym, f16)
            wk = (xs.reshape(-1).astype(np.float64) - resid[k - 1]).reshape(rows, cols)
            want = Af @ wk.T
            tol = np.abs(Af) @ (np.abs(xs).astype(np.float64) + np.abs(wk)).T * (k + 1) * 2.0 ** -23
            if np.any(np.abs(Y - want) > tol + 1e-300):
                fails.append(f"sym={sym} f16={f16} k={k}: A W~ != A X - A R")
    return fails


def pin_gemv_vs_bf16_reconstruction(orc, seed=43, rows=5, g=128) -> list[str]:
    """The product equals A times the bf16 reconstruction (a separately
    pinned routine) up to the bf16 rounding of each weight (2^-9 relative)."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 2 * g
    xs = np.concatenate(_random_groups(rng, rows * 2, g)).reshape(rows, cols)
    W = bf16_bits_of_f32(xs)
    codes, scales, zeros = orc.quantize(W, group=g, n_stages=4)
    A = bf16_round_bits(rng.normal(0, 1, (2, cols)).astype(np.float32))
    Af = (A.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    for k in range(1, 5):
        rec = orc.reconstruct(codes, scales, zeros, rows, cols, g, k)
        recf = (rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        Y = orc.gemv(codes, scales, zeros, rows, cols, g, k, A)
        tol = np.abs(Af) @ np.abs(recf).T * 2.0 ** -8 + 1e-300
        if np.any(np.abs(Y - Af @ recf.T) > tol):
            fails.append(f"k={k}: product differs from A x bf16 reconstruction beyond bf16 rounding")
    return fails


# ---------------------------------------------------------------------------
# heterogeneous stage widths (asymmetric grid) and the group peak-to-mean ratio
# ---------------------------------------------------------------------------
# WH1: x = [-1, 0, 0.5, 2], widths [1, 3] (a 1-bit base, a 3-bit residual):
#   stage 0: lo -1, hi 2, one step s = 3; d/s = [0, 1/3, 1/2, 1] -> rhe
#            [0, 0, 0 (tie to even), 1]; levels [-1, -1, -1, 2], r = [0, 1, 1.5, 0];
#   stage 1: lo 0, hi 1.5, seven steps s = fl(1.5/7); 1/s = 4.67 -> 5,
#            1.5/s = 6.99999986 rounds to 7.0 -> 7, zeros -> 0.
WH1 = dict(x=[-1.0, 0.0, 0.5, 2.0], bits=[1, 3], Q=[[0, 0, 0, 1], [0, 5, 7, 0]], s0=3.0, z=[-1.0, 0.0],
           r0=[0.0, 1.0, 1.5, 0.0])


def pin_bits_worked_and_two_bit_case(orc) -> list[str]:
    fails = []
    Q, s, z, r = orc.quantize_group_bits(np.array(WH1["x"], np.float32), WH1["bits"])
    if Q.tolist() != WH1["Q"] or float(s[0]) != WH1["s0"] or z.tolist() != WH1["z"] or r[0].tolist() != WH1["r0"]:
        fails.append(f"WH1: {Q.tolist()} {s.tolist()} {z.tolist()} {r[0].tolist()}")
    if bits_of(s[1]) != bits_of(np.float32(1.5) / np.float32(7.0)):
        fails.append(f"WH1: stage-1 scale {s[1]!r}")
    # every width 2: the 2-bit quantizer (separately pinned) bit for bit
    rng = np.random.default_rng(47)
    for x in _random_groups(rng, 30, 128):
        a = orc.quantize_group(x, 4)
        b = orc.quantize_group_bits(x, [2, 2, 2, 2])
        for u, v in zip(a, b):
            if not np.array_equal(np.asarray(u).view(np.uint8), np.asarray(v).view(np.uint8)):
                fails.append("widths [2, 2, 2, 2] differ from the 2-bit quantizer")
                return fails
    W = bf16_bits_of_f32(np.concatenate(_random_groups(rng, 6, 64)).reshape(3, 128))
    a = orc.quantize(W, 64, 4)
    b = orc.quantize_bits(W, 64, [2, 2, 2, 2])
    for u, v in zip(a, b):
        for uu, vv in zip(u, v):
            if not np.array_equal(uu.view(np.uint8), vv.view(np.uint8)):
                fails.append("packed widths [2, 2, 2, 2] differ from the 2-bit package")
                return fails
    return fails


def pin_bits_brute_force_exact(orc, seed=53, count=200) -> list[str]:
    """Dyadic groups for widths 1, 3, 4: lo = a/16, s = 2^e, values
    lo + m 2^(e-2) with both ends present (range = (2^b - 1) 2^e): every step
    exact; each code is the nearest of the 2^b levels, ties to the even code."""
    rng = np.random.default_rng(seed)
    fails = []
    for i in range(count):
        b = (1, 3, 4)[i % 3]
        steps = (1 << b) - 1
        g = int(rng.integers(2, 17))
        e = int(rng.integers(-4, 2))
        lo = Fraction(int(rng.integers(-16, 17)), 16)
        ms = list(rng.integers(0, 4 * steps + 1, size=g))
        ms[0], ms[-1] = 0, 4 * steps
        rng.shuffle(ms)
        s = Fraction(2) ** e
        xs = [lo + Fraction(int(m)) * Fraction(2) ** (e - 2) for m in ms]
        Q, sc, z, r = orc.quantize_group_bits(np.array([float(v) for v in xs], np.float32), [b])
        if Fraction(float(sc[0])) != s or Fraction(float(z[0])) != lo:
            fails.append(f"b={b}: s={sc[0]} z={z[0]}")
            continue
        for j, v in enumerate(xs):
            dist = [abs(v - (lo + q * s)) for q in range(steps + 1)]
            best = min(dist)
            cands = [q for q in range(steps + 1) if dist[q] == best]
            want = cands[0] if len(cands) == 1 else [q for q in cands if q % 2 == 0][0]
            if int(Q[0, j]) != want or Fraction(float(r[0, j])) != v - (lo + want * s):
                fails.append(f"b={b}: x={float(v)} Q={int(Q[0, j])} want {want}")
                break
        if len(fails) > 5:
            break
    return fails


def pin_bits_invariants_and_packing(orc, seed=59, g=64) -> list[str]:
    """Random groups, widths [1, 3], [3, 1], [4, 2, 1], [2, 4]: zero = group
    minimum, s = range / (2^b - 1) to rounding, half-step bound, the L-inf
    error shrinks by 2^b - 1 per stage (to rounding); the packed codes equal
    the per-group codes read back with numpy's little-endian bit unpacking;
    prefix k reconstructs x - r_(k-1) to summation and bf16 rounding."""
    rng = np.random.default_rng(seed)
    fails = []
    rows, cols = 4, 2 * g
    xs = np.concatenate(_random_groups(rng, rows * 2, g)).reshape(rows, cols)
    W = bf16_bits_of_f32(xs)
    for bits in ([1, 3], [3, 1], [4, 2, 1], [2, 4]):
        codes, scales, zeros = orc.quantize_bits(W, g, bits)
        for gi in range(rows * cols // g):
            x = xs.reshape(-1)[gi * g:(gi + 1) * g]
            Q, s, z, r = orc.quantize_group_bits(x, bits)
            prev = x.astype(np.float64)
            for k, b in enumerate(bits):
                steps = (1 << b) - 1
                lo, hi = float(np.min(prev)), float(np.max(prev))
                if float(z[k]) != lo or abs(float(s[k]) - (hi - lo) / steps) > 2 ** -22 * (hi - lo) + 1e-45:
                    fails.append(f"{bits} stage {k}: zero/scale")
                rk = r[k].astype(np.float64)
                bound = 0.5 * float(s[k]) + 2 ** -21 * (abs(lo) + (steps + 1) * float(s[k])) + 1e-45
                if np.max(np.abs(rk)) > bound:
                    fails.append(f"{bits} stage {k}: half step")
                if np.max(np.abs(rk)) > np.max(np.abs(prev)) / steps * (1 + 2 ** -18) + 2 ** -20 * (abs(lo) + (steps + 1) * float(s[k])):
                    fails.append(f"{bits} stage {k}: max|r| not reduced by 2^b - 1")
                bitsarr = np.unpackbits(codes[k], bitorder="little")
                c0 = gi * g
                got = [int(sum(int(bitsarr[(c0 + j) * b + t]) << t for t in range(b))) for j in range(g)]
                if got != Q[k].tolist():
                    fails.append(f"{bits} stage {k}: packed codes")
                prev = rk
            if len(fails) > 5:
                return fails
        for k in range(1, len(bits) + 1):
            rec = orc.reconstruct_bits(codes, scales, zeros, rows, cols, g, k, bits).reshape(-1)
            recf = (rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
            for gi in range(rows * cols // g):
                x = xs.reshape(-1)[gi * g:(gi + 1) * g].astype(np.float64)
                r = orc.quantize_group_bits(x.astype(np.float32), bits)[3]
                want = x - r[k - 1]
                tol = np.abs(want) * 2 ** -8 + 8 * 2 ** -24 * (np.abs(x).max() + 1e-30)
                if np.any(np.abs(recf[gi * g:(gi + 1) * g] - want) > tol):
                    fails.append(f"{bits}: prefix {k} is not x - r")
                    break
    return fails


def pin_group_pmr(orc, seed=61) -> list[str]:
    """Closed forms of max|x| / mean|x|: a constant nonzero group gives 1, a
    group with one nonzero gives g, j equal magnitudes (any signs) and zeros
    give g / j, an all-zero group 0; random groups match the definition to
    binary64 rounding."""
    rng = np.random.default_rng(seed)
    fails = []
    g = 128
    rows = []
    rows.append(np.full(g, 0.5, np.float32))
    one = np.zeros(g, np.float32); one[17] = -3.0; rows.append(one)
    j = 5
    some = np.zeros(g, np.float32); some[:j] = [0.25, -0.25, 0.25, -0.25, 0.25]; rows.append(some)
    rows.append(np.zeros(g, np.float32))
    W = bf16_bits_of_f32(np.stack(rows)).reshape(1, 4 * g)
    p = orc.group_pmr(W, g)
    want = [1.0, float(g), g / j, 0.0]
    if p.tolist() != want:
        fails.append(f"closed forms {p.tolist()} != {want}")
    xs = np.concatenate(_random_groups(rng, 8, g)).reshape(2, 4 * g)
    p = orc.group_pmr(bf16_bits_of_f32(xs), g)
    a = np.abs(xs.astype(np.float64)).reshape(-1, g)
    ref = a.max(1) / a.mean(1)
    if np.max(np.abs(p - ref) / ref) > 1e-12:
        fails.append("random groups: pmr differs from max/mean")
    return fails


# ---------------------------------------------------------------------------
# prefill product (bf16 operands: the prefix reconstruction is the weight)
# ---------------------------------------------------------------------------
# PF1: a hand-built one-stage package, codes [0, 1, 2, 3] (byte 0xE4, LSB
#   first), scale s = 1 + 3*2^-9, zero 0.  Levels fl(Q s) = [0, 1.005859375,
#   2.01171875, 3.017578125] (exact); their bf16 nearest-even values are
#   [0, 1.0078125, 2.015625, 3.015625] (truncation would give [0, 1, 2,
#   3.015625]).  A = [[1, 1, 1, 1], [0, 0, 0, 1], [1, -1, 0.5, 2]]:
#   Y = [6.0390625, 3.015625, -1.0078125 + 1.0078125 + 6.03125 = 6.03125].
# PF2: the same codes, symmetric grid, binary16 scale 1.0 (0x3C00): levels
#   (Q - 2) = [-2, -1, 0, 1]; Y = [-2, 1, -2 + 1 + 0 + 2 = 1].
PF1 = dict(byte=0xE4, scale=1.0 + 3 * 2.0 ** -9, Y=[6.0390625, 3.015625, 6.03125])
PF_A = [[1.0, 1.0, 1.0, 1.0], [0.0, 0.0, 0.0, 1.0], [1.0, -1.0, 0.5, 2.0]]
PF2_Y = [-2.0, 1.0, 1.0]


def pin_prefill_worked(orc) -> list[str]:
    fails = []
    A = bf16_bits_of_f32(np.array(PF_A, np.float32))
    codes = [np.array([PF1["byte"]], np.uint8)]
    Y = orc.prefill(codes, [np.array([PF1["scale"]], np.float32)], [np.zeros(1, np.float32)], 1, 4, 4, 1, A)
    if Y[:, 0].tolist() != PF1["Y"]:
        fails.append(f"PF1: {Y[:, 0].tolist()} != {PF1['Y']}")
    Y = orc.prefill(codes, [np.array([0x3C00], np.uint16)], None, 1, 4, 4, 1, A, sym=True, scale_f16=True)
    if Y[:, 0].tolist() != PF2_Y:
        fails.append(f"PF2: {Y[:, 0].tolist()} != {PF2_Y}")
    return fails


def pin_prefill_one_hot(orc, seed=67, rows=5, g=64) -> list[str]:
    """One-hot activation rows pick single weights: with A[t] = e_(p(t)) for a
    permutation p of the columns, Y[t][r] is the bf16 reconstruction (a
    separately pinned routine) at [r][p(t)], exactly; every format, k = 1..4."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 2 * g
    xs = np.concatenate(_random_groups(rng, rows * 2, g)).reshape(rows, cols)
    W = bf16_bits_of_f32(xs)
    perm = rng.permutation(cols)
    A = np.zeros((cols, cols), np.float32)
    A[np.arange(cols), perm] = 1.0
    A = bf16_bits_of_f32(A)
    for sym, f16 in ((False, False), (True, False), (True, True)):
        if sym:
            codes, scales = orc.quantize_sym(W, group=g, n_stages=4, scale_f16=f16)
            zeros = None
        else:
            codes, scales, zeros = orc.quantize(W, group=g, n_stages=4)
        for k in range(1, 5):
            rec = (orc.reconstruct_sym(codes, scales, rows, cols, g, k, f16) if sym
                   else orc.reconstruct(codes, scales, zeros, rows, cols, g, k))
            recf = (rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
            Y = orc.prefill(codes, scales, zeros, rows, cols, g, k, A, sym, f16)
            if not np.array_equal(Y, recf[:, perm].T):
                fails.append(f"sym={sym} f16={f16} k={k}: one-hot rows do not select the reconstruction")
    return fails


def pin_prefill_integer_exact(orc, seed=71, rows=6, g=32) -> list[str]:
    """Packages with scale 1 and integer zeros have integer levels z + Q, so
    every prefix weight is a small integer (exact in bf16) and, with integer
    activations, the product is an integer matrix: numpy's int64 matmul of the
    weights unpacked here (LSB-first 2-bit codes, group-wise zeros) must equal
    the oracle exactly."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 4 * g
    n = rows * cols
    q = rng.integers(0, 4, (4, n))
    z = rng.integers(-3, 4, (4, n // g))
    codes = [np.zeros(n // 4, np.uint8) for _ in range(4)]
    for i in range(4):
        for s in range(4):
            codes[i] |= (q[i, s::4] << (2 * s)).astype(np.uint8)
    scales = [np.ones(n // g, np.float32) for _ in range(4)]
    zeros = [z[i].astype(np.float32) for i in range(4)]
    A_int = rng.integers(-4, 5, (7, cols))
    A = bf16_bits_of_f32(A_int.astype(np.float32))
    for k in range(1, 5):
        w = sum(q[i] + np.repeat(z[i], g) for i in range(k)).reshape(rows, cols)
        Y = orc.prefill(codes, scales, zeros, rows, cols, g, k, A)
        if not np.array_equal(Y, (A_int @ w.T).astype(np.float64)):
            fails.append(f"k={k}: integer package product differs from the int64 matmul")
    return fails


def pin_prefill_vs_binary32_product(orc, seed=73, rows=4, g=128) -> list[str]:
    """The bf16-weight product differs from the binary32-weight product (the
    decode form, pinned above) by at most the bf16 rounding of each weight:
    |Y_bf16 - Y_f32| <= 2^-9 sum |a| |w~| (plus the binary64 sums)."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 2 * g
    xs = np.concatenate(_random_groups(rng, rows * 2, g)).reshape(rows, cols)
    codes, scales, zeros = orc.quantize(bf16_bits_of_f32(xs), group=g, n_stages=4)
    A = bf16_round_bits(rng.normal(0, 1, (9, cols)).astype(np.float32))
    Af = (A.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    for k in range(1, 5):
        Yb = orc.prefill(codes, scales, zeros, rows, cols, g, k, A)
        Yf = orc.gemv(codes, scales, zeros, rows, cols, g, k, A)
        rec = orc.reconstruct(codes, scales, zeros, rows, cols, g, k)
        recf = (rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        tol = np.abs(Af) @ np.abs(recf).T * 2.0 ** -8 + 1e-300
        if np.any(np.abs(Yb - Yf) > tol) or np.array_equal(Yb, Yf):
            fails.append(f"k={k}: bf16-weight product not within bf16 rounding of the binary32 one")
    return fails


# ---------------------------------------------------------------------------
# products with per-stage widths (decode form: binary32 weights; prefill form:
# bf16 weights)
# ---------------------------------------------------------------------------
BITS_SPLITS = ([1, 3], [3, 1], [4, 2, 1], [2, 4], [1, 1, 1, 1])


def _bits_package(orc, rng, rows, cols, g, bits):
    xs = np.concatenate(_random_groups(rng, rows * cols // g, g)).reshape(rows, cols)
    return orc.quantize_bits(bf16_bits_of_f32(xs), g, bits)


def pin_product_bits_two_bit_case(orc, seed=79, rows=5, g=64) -> list[str]:
    """With every width 2 the product equals the 2-bit products pinned above:
    the decode form rrq_oracle_gemv and the prefill form rrq_oracle_prefill,
    exactly."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 3 * g
    xs = np.concatenate(_random_groups(rng, rows * 3, g)).reshape(rows, cols)
    codes, scales, zeros = orc.quantize(bf16_bits_of_f32(xs), group=g, n_stages=4)
    A = bf16_round_bits(rng.normal(0, 1, (3, cols)).astype(np.float32))
    for k in range(1, 5):
        yd = orc.product_bits(codes, scales, zeros, rows, cols, g, k, [2] * 4, A, False)
        yp = orc.product_bits(codes, scales, zeros, rows, cols, g, k, [2] * 4, A, True)
        if not np.array_equal(yd, orc.gemv(codes, scales, zeros, rows, cols, g, k, A)):
            fails.append(f"k={k}: decode form with widths 2 differs from the 2-bit product")
        if not np.array_equal(yp, orc.prefill(codes, scales, zeros, rows, cols, g, k, A)):
            fails.append(f"k={k}: prefill form with widths 2 differs from the 2-bit prefill product")
    return fails


def pin_product_bits_one_hot(orc, seed=83, rows=4, g=32) -> list[str]:
    """One-hot activation rows pick single weights: the prefill form returns the
    width reconstruction (pinned above) exactly, and the decode form rounds to
    it, for several splits and every prefix."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 4 * g
    perm = rng.permutation(cols)
    E = np.zeros((cols, cols), np.float32)
    E[np.arange(cols), perm] = 1.0
    E = bf16_bits_of_f32(E)
    for bits in BITS_SPLITS:
        codes, scales, zeros = _bits_package(orc, rng, rows, cols, g, bits)
        for k in range(1, len(bits) + 1):
            rec = orc.reconstruct_bits(codes, scales, zeros, rows, cols, g, k, bits)
            recf = (rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
            yp = orc.product_bits(codes, scales, zeros, rows, cols, g, k, bits, E, True)
            yd = orc.product_bits(codes, scales, zeros, rows, cols, g, k, bits, E, False)
            if not np.array_equal(yp, recf[:, perm].T):
                fails.append(f"{bits} k={k}: one-hot prefill form is not the width reconstruction")
            if not np.array_equal(bf16_round_bits(yd.astype(np.float32)), rec[:, perm].T):
                fails.append(f"{bits} k={k}: one-hot decode form does not round to the reconstruction")
    return fails


def pin_product_bits_integer_exact(orc, seed=89, rows=5, g=32) -> list[str]:
    """Scale 1 and integer zeros make every level an integer: the products
    (both forms) equal numpy's int64 matmul of weights whose codes are
    unpacked here with numpy's little-endian bit order."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 4 * g
    n = rows * cols
    A_int = rng.integers(-4, 5, (6, cols))
    A = bf16_bits_of_f32(A_int.astype(np.float32))
    for bits in BITS_SPLITS:
        q = [rng.integers(0, 1 << b, n) for b in bits]
        z = [rng.integers(-3, 4, n // g) for _ in bits]
        codes = []
        for qi, b in zip(q, bits):
            bitsarr = ((qi[:, None] >> np.arange(b)) & 1).astype(np.uint8).reshape(-1)
            codes.append(np.packbits(bitsarr, bitorder="little"))
        scales = [np.ones(n // g, np.float32) for _ in bits]
        zeros = [zi.astype(np.float32) for zi in z]
        for k in range(1, len(bits) + 1):
            w = sum(q[i] + np.repeat(z[i], g) for i in range(k)).reshape(rows, cols)
            want = (A_int @ w.T).astype(np.float64)
            for bf in (False, True):
                Y = orc.product_bits(codes, scales, zeros, rows, cols, g, k, bits, A, bf)
                if not np.array_equal(Y, want):
                    fails.append(f"{bits} k={k} bf16={bf}: integer product differs from the int64 matmul")
    return fails


def pin_product_bits_forms(orc, seed=97, rows=4, g=64) -> list[str]:
    """The prefill form differs from the decode form by at most the bf16
    rounding of each weight (2^-9 relative), and does differ."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 2 * g
    A = bf16_round_bits(rng.normal(0, 1, (5, cols)).astype(np.float32))
    Af = (A.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    for bits in BITS_SPLITS[:3]:
        codes, scales, zeros = _bits_package(orc, rng, rows, cols, g, bits)
        k = len(bits)
        rec = orc.reconstruct_bits(codes, scales, zeros, rows, cols, g, k, bits)
        recf = (rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        yd = orc.product_bits(codes, scales, zeros, rows, cols, g, k, bits, A, False)
        yp = orc.product_bits(codes, scales, zeros, rows, cols, g, k, bits, A, True)
        tol = np.abs(Af) @ np.abs(recf).T * 2.0 ** -8 + 1e-300
        if np.any(np.abs(yp - yd) > tol) or np.array_equal(yp, yd):
            fails.append(f"{bits}: the two forms are not within bf16 rounding of each other")
    return fails


# ---------------------------------------------------------------------------
# Algorithm 1 with a base checkpoint and per-stage widths
# ---------------------------------------------------------------------------
FB_SPLITS = ([1, 3], [3, 1], [4, 2, 1], [2, 4, 2, 1])


def pin_base_bits_branch_equivalence(orc, seed=101, rows=4, g=64) -> list[str]:
    """Given the RTN base of the width quantizer (pinned above), the base
    branch rebuilds exactly the same package: Algorithm 1's two branches agree."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 3 * g
    for bits in FB_SPLITS:
        xs = np.concatenate(_random_groups(rng, rows * 3, g)).reshape(rows, cols)
        W = bf16_bits_of_f32(xs)
        codes, scales, zeros = orc.quantize_bits(W, g, bits)
        fc, fs, fz = orc.quantize_from_base_bits(W, (codes[0], scales[0], zeros[0]), g, bits)
        for k in range(len(bits)):
            if not (np.array_equal(fc[k], codes[k]) and np.array_equal(fs[k].view(np.uint32), scales[k].view(np.uint32))
                    and np.array_equal(fz[k].view(np.uint32), zeros[k].view(np.uint32))):
                fails.append(f"{bits} stage {k}: base branch differs from the full build")
    return fails


def pin_base_bits_zero_base(orc, seed=103, rows=3, g=32) -> list[str]:
    """A base whose every level is +0 (codes 0, zero +0, any scale) leaves
    R_0 = x, so stages 1.. are the width quantizer of x with widths bits[1:]."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 4 * g
    n = rows * cols
    for bits in FB_SPLITS:
        xs = np.concatenate(_random_groups(rng, rows * 4, g)).reshape(rows, cols)
        W = bf16_bits_of_f32(xs)
        base = (np.zeros((n * bits[0] + 7) // 8, np.uint8), rng.uniform(0.1, 2.0, n // g).astype(np.float32),
                np.zeros(n // g, np.float32))
        fc, fs, fz = orc.quantize_from_base_bits(W, base, g, bits)
        rc, rs, rz = orc.quantize_bits(W, g, bits[1:])
        for k in range(1, len(bits)):
            if not (np.array_equal(fc[k], rc[k - 1]) and np.array_equal(fs[k].view(np.uint32), rs[k - 1].view(np.uint32))
                    and np.array_equal(fz[k].view(np.uint32), rz[k - 1].view(np.uint32))):
                fails.append(f"{bits} stage {k}: zero base does not reduce to the width quantizer of x")
    return fails


def pin_base_bits_random_base(orc, seed=107, rows=3, g=64) -> list[str]:
    """With an arbitrary base (random codes, scales, zeros), the last prefix of
    the base branch is within half a last step (plus the binary32 roundings
    of the stage sums) of the input in every group."""
    rng = np.random.default_rng(seed)
    fails = []
    cols = 2 * g
    n = rows * cols
    for bits in FB_SPLITS:
        xs = np.concatenate(_random_groups(rng, rows * 2, g)).reshape(rows, cols)
        W = bf16_bits_of_f32(xs)
        b0 = bits[0]
        q0 = rng.integers(0, 1 << b0, n)
        c0 = np.packbits(((q0[:, None] >> np.arange(b0)) & 1).astype(np.uint8).reshape(-1), bitorder="little")
        base = (c0, rng.uniform(0.0, 0.05, n // g).astype(np.float32), rng.normal(0, 0.05, n // g).astype(np.float32))
        fc, fs, fz = orc.quantize_from_base_bits(W, base, g, bits)
        k = len(bits)
        rec = orc.reconstruct_bits(fc, fs, fz, rows, cols, g, k, bits)
        recf = (rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64).reshape(-1)
        x = (W.astype(np.uint32) << 16).view(np.float32).astype(np.float64).reshape(-1)
        half = np.repeat(fs[k - 1].astype(np.float64), g) / 2
        bound = half + np.abs(x) * 2.0 ** -8 + 1e-30
        if np.any(np.abs(recf - x) > bound):
            fails.append(f"{bits}: last prefix beyond half a last step")
    return fails


ALL_PINS = [pin_worked_groups, pin_bf16_rounding, pin_brute_force_exact, pin_brute_force_tiny,
            pin_invariants, pin_exact_grid, pin_prefix_reconstruction, pin_f16_rounding,
            pin_sym_worked_groups, pin_sym_brute_force_exact, pin_sym_invariants,
            pin_sym_prefix_reconstruction, pin_base_worked_groups, pin_base_branch_equivalence,
            pin_base_residual_invariants, pin_gemv_worked, pin_gemv_is_input_minus_residual,
            pin_gemv_vs_bf16_reconstruction, pin_bits_worked_and_two_bit_case, pin_bits_brute_force_exact,
            pin_bits_invariants_and_packing, pin_group_pmr, pin_prefill_worked, pin_prefill_one_hot,
            pin_prefill_integer_exact, pin_prefill_vs_binary32_product, pin_product_bits_two_bit_case,
            pin_product_bits_one_hot, pin_product_bits_integer_exact, pin_product_bits_forms,
            pin_base_bits_branch_equivalence, pin_base_bits_zero_base, pin_base_bits_random_base]


def all_failures(orc) -> list[str]:
    out = []
    for p in ALL_PINS:
        try:
            out += [f"{p.__name__}: {m}" for m in p(orc)]
        except Exception as e:  # a crash of a mutated oracle counts as caught
            out.append(f"{p.__name__}: raised {type(e).__name__}: {e}")
    return out
