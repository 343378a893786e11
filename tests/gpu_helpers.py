"""Helpers for the GPU parity tests: run the CUDA path through the C ABI, run
the CPU oracle on the same bf16 input, and compare bit for bit."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2608_04048_gb300 import binding


def bf16_bits(W: torch.Tensor) -> np.ndarray:
    """uint16 bit patterns of a bf16 tensor, on the host."""
    return W.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def gpu_package_host(pkg: binding.Package):
    torch.cuda.synchronize()
    return ([c.cpu().numpy() for c in pkg.codes], [s.cpu().numpy() for s in pkg.scales],
            [z.cpu().numpy() for z in pkg.zeros])


def assert_package_equal(gpu, ref, n_stages, where=""):
    gc, gs, gz = gpu
    rc, rs, rz = ref
    for k in range(n_stages):
        for name, a, b in (("codes", gc[k], rc[k]), ("scales", gs[k], rs[k]), ("zeros", gz[k], rz[k])):
            a8 = np.ascontiguousarray(a).view(np.uint8)
            b8 = np.ascontiguousarray(b).view(np.uint8)
            if a8.shape != b8.shape or not np.array_equal(a8, b8):
                if name == "codes":
                    bad = np.nonzero(a8 != b8)[0]
                else:
                    bad = np.nonzero(np.ascontiguousarray(a).view(np.uint32) != np.ascontiguousarray(b).view(np.uint32))[0]
                i = int(bad[0]) if bad.size else -1
                raise AssertionError(f"{where} stage {k} {name}: {bad.size} mismatches, first at {i}: "
                                     f"gpu={a.reshape(-1)[i] if i >= 0 else None!r} "
                                     f"oracle={b.reshape(-1)[i] if i >= 0 else None!r}")


def check_full(W: torch.Tensor, group: int, n_stages: int, ks=None, where=""):
    """Quantize W on the GPU and in the oracle; compare the whole package and
    the reconstructions at every prefix k."""
    rows, cols = W.shape
    pkg = binding.rrq_quantize(W, group, n_stages)
    gpu = gpu_package_host(pkg)
    ref = oracle.quantize(bf16_bits(W), group, n_stages)
    assert_package_equal(gpu, ref, n_stages, where)
    for k in (ks or range(1, n_stages + 1)):
        out = binding.rrq_reconstruct(pkg, k)
        torch.cuda.synchronize()
        want = oracle.reconstruct(*ref, rows, cols, group, k)
        got = bf16_bits(out)
        if not np.array_equal(got, want):
            bad = np.nonzero(got.reshape(-1) != want.reshape(-1))[0]
            raise AssertionError(f"{where} reconstruct k={k}: {bad.size} mismatches, first at {bad[0]}")
    return pkg


def sample_groups(n_groups: int, count: int, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    head = np.arange(min(64, n_groups))
    tail = np.arange(max(0, n_groups - 64), n_groups)
    mid = rng.integers(0, n_groups, size=count)
    return np.unique(np.concatenate([head, tail, mid]))


def check_sampled(W: torch.Tensor, pkg: binding.Package, idx: np.ndarray, ks=(1, 2, 3, 4), where=""):
    """Compare the GPU package of W at the sampled group indices with the
    oracle run on exactly those groups (groups are independent)."""
    g, S = pkg.group, pkg.n_stages
    it = torch.from_numpy(idx).to(W.device)
    Wg = W.reshape(-1, g).index_select(0, it)
    ref = oracle.quantize(bf16_bits(Wg), g, S)
    gc = [c.view(-1, g // 4).index_select(0, it).cpu().numpy().reshape(-1) for c in pkg.codes]
    gs = [s.index_select(0, it).cpu().numpy() for s in pkg.scales]
    gz = [z.index_select(0, it).cpu().numpy() for z in pkg.zeros]
    assert_package_equal((gc, gs, gz), ref, S, where)
    for k in ks:
        if k > S:
            continue
        out = binding.rrq_reconstruct(pkg, k)
        got = bf16_bits(out.reshape(-1, g).index_select(0, it))
        want = oracle.reconstruct(*ref, idx.size, g, g, k)
        if not np.array_equal(got, want):
            bad = np.nonzero(got.reshape(-1) != want.reshape(-1))[0]
            raise AssertionError(f"{where} sampled reconstruct k={k}: {bad.size} mismatches")
        del out


# ---------------------------------------------------------------------------
# symmetric grid (binary32 or binary16 scales)
# ---------------------------------------------------------------------------
def _cmp_bytes(a, b, what):
    a8 = np.ascontiguousarray(a).view(np.uint8)
    b8 = np.ascontiguousarray(b).view(np.uint8)
    if a8.shape != b8.shape or not np.array_equal(a8, b8):
        bad = np.nonzero(a8 != b8)[0] if a8.shape == b8.shape else []
        raise AssertionError(f"{what}: {len(bad)} byte mismatches, first at {bad[0] if len(bad) else None}")


def scales_host(pkg):
    """Stored scales as numpy: float32, or uint16 binary16 bit patterns."""
    torch.cuda.synchronize()
    if pkg.scale_type == binding.SCALE_F16:
        return [s.view(torch.int16).cpu().numpy().view(np.uint16) for s in pkg.scales]
    return [s.cpu().numpy() for s in pkg.scales]


def check_full_sym(W: torch.Tensor, group: int, n_stages: int, f16: bool, where=""):
    """Symmetric package of W through rrq_quantize_ex against the oracle (codes
    and scales bit for bit), then every prefix through rrq_reconstruct_ex, one
    at a time and all at once."""
    rows, cols = W.shape
    st = binding.SCALE_F16 if f16 else binding.SCALE_F32
    (pkg,) = binding.rrq_quantize_ex([W], group, n_stages, binding.GRID_SYM, st)
    rc, rs = oracle.quantize_sym(bf16_bits(W), group, n_stages, f16)
    gs = scales_host(pkg)
    for k in range(n_stages):
        _cmp_bytes(pkg.codes[k].cpu().numpy(), rc[k], f"{where} stage {k} codes")
        _cmp_bytes(gs[k], rs[k], f"{where} stage {k} scales")
    allp = binding.rrq_reconstruct_ex([pkg], n_stages, all_prefixes=True)[0]
    for k in range(1, n_stages + 1):
        one = binding.rrq_reconstruct_ex([pkg], k)[0][0]
        torch.cuda.synchronize()
        want = oracle.reconstruct_sym(rc, rs, rows, cols, group, k, f16)
        _cmp_bytes(bf16_bits(one), want, f"{where} reconstruct k={k}")
        _cmp_bytes(bf16_bits(allp[k - 1]), want, f"{where} all-prefix reconstruct k={k}")
    return pkg


def check_sampled_sym(W: torch.Tensor, pkg, idx: np.ndarray, outs=None, where=""):
    """Sampled groups of a symmetric package (and optionally of its prefix
    reconstructions outs[j] = prefix j+1) against the oracle run on exactly
    those groups."""
    g, S = pkg.group, pkg.n_stages
    f16 = pkg.scale_type == binding.SCALE_F16
    it = torch.from_numpy(idx).to(W.device)
    Wg = W.reshape(-1, g).index_select(0, it)
    rc, rs = oracle.quantize_sym(bf16_bits(Wg), g, S, f16)
    for k in range(S):
        gc = pkg.codes[k].view(-1, g // 4).index_select(0, it).cpu().numpy().reshape(-1)
        _cmp_bytes(gc, rc[k], f"{where} stage {k} codes")
        s = pkg.scales[k].index_select(0, it)
        gs = s.view(torch.int16).cpu().numpy().view(np.uint16) if f16 else s.cpu().numpy()
        _cmp_bytes(gs, rs[k], f"{where} stage {k} scales")
    for j, o in enumerate(outs or []):
        got = bf16_bits(o.reshape(-1, g).index_select(0, it))
        want = oracle.reconstruct_sym(rc, rs, idx.size, g, g, j + 1, f16)
        _cmp_bytes(got, want, f"{where} sampled prefix {j + 1}")


SENTINEL = 0x7FA5A5A5  # a NaN pattern no kernel writes


def guarded_outputs(shapes, batch, guard=1024):
    """float32 [batch, rows] outputs, each inside a buffer with `guard`
    sentinel floats (4 KiB) on both sides; 16-byte aligned."""
    bufs, ys = [], []
    for rows, _cols in shapes:
        buf = torch.empty((batch * rows + 2 * guard,), dtype=torch.float32, device="cuda")
        buf.view(torch.int32).fill_(SENTINEL)
        bufs.append(buf)
        ys.append(buf[guard:guard + batch * rows].view(batch, rows))
    return bufs, ys, guard


def bands_intact(bufs, guard) -> bool:
    torch.cuda.synchronize()
    return all(bool((b.view(torch.int32)[:guard] == SENTINEL).all()) and
               bool((b.view(torch.int32)[-guard:] == SENTINEL).all()) for b in bufs)
