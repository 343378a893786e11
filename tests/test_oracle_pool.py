"""The oracle over many processes (oracle/pool.py), on the CPU: row-range
tasks on a shared region reproduce the single-process oracle's package and
prefixes exactly, and a planted difference in any compared array is
reported at its element."""
import numpy as np
import pytest

import oracle
from oracle.pool import Layout, OraclePool, SharedRegion, Task, host_description

pytestmark = pytest.mark.filterwarnings("ignore::UserWarning")


@pytest.fixture(scope="module")
def pool():
    with OraclePool(3) as p:
        yield p


def _bf16_bits(x: np.ndarray) -> np.ndarray:
    u = x.astype(np.float32).view(np.uint32)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


@pytest.mark.parametrize("fmt", ["asym", "sym32", "sym16"])
def test_row_tasks_equal_whole_matrix_and_find_planted_differences(pool, fmt):
    rows, cols, g, S = 37, 384, 128, 4
    rng = np.random.default_rng(5)
    Wb = _bf16_bits(rng.standard_t(3, (rows, cols)) * 0.02)
    n = rows * cols
    if fmt == "asym":
        codes, scales, zeros = oracle.quantize(Wb, g, S)
        pre = [oracle.reconstruct(codes, scales, zeros, rows, cols, g, k) for k in range(1, S + 1)]
    else:
        f16 = fmt == "sym16"
        codes, scales = oracle.quantize_sym(Wb, g, S, f16)
        zeros = []
        pre = [oracle.reconstruct_sym(codes, scales, rows, cols, g, k, f16) for k in range(1, S + 1)]
    lay = Layout()
    off = {"w": lay.take(2 * n), "c": [lay.take(n // 4) for _ in range(S)],
           "s": [lay.take(scales[0].nbytes) for _ in range(S)], "z": [lay.take(4 * n // g) for _ in zeros],
           "p": [lay.take(2 * n) for _ in range(S)], "r": lay.take(2 * n)}
    with SharedRegion(lay.size) as reg:
        reg.array(off["w"], np.uint16, n)[:] = Wb.reshape(-1)
        for k in range(S):
            reg.array(off["c"][k], np.uint8, n // 4)[:] = codes[k]
            reg.array(off["s"][k], np.uint8, scales[k].nbytes)[:] = scales[k].view(np.uint8)
            reg.array(off["p"][k], np.uint16, n)[:] = pre[k].reshape(-1)
        for k, z in enumerate(zeros):
            reg.array(off["z"][k], np.float32, n // g)[:] = z
        reg.array(off["r"], np.uint16, n)[:] = pre[2].reshape(-1)
        t = Task(reg.name, "m", fmt, g, S, rows, cols, off["w"], codes=tuple(off["c"]), scales=tuple(off["s"]),
                 zeros=tuple(off["z"]), prefixes=tuple(off["p"]), recon=((3, off["r"]),))
        parts = t.split(1000)
        assert len(parts) == 19 and sum(p.nrows for p in parts) == rows
        res = pool.run(parts)
        assert sum(r["weights"] for r in res) == n
        assert not [m for r in res for m in r["mismatches"]]
        # one planted difference per array kind
        reg.array(off["c"][3], np.uint8, n // 4)[1000] ^= 4
        reg.array(off["p"][0], np.uint16, n)[n - 1] ^= 1
        reg.array(off["r"], np.uint16, n)[5] ^= 0x8000
        reg.array(off["s"][2], np.uint8, scales[0].nbytes)[0] ^= 1
        if zeros:
            reg.array(off["z"][1], np.uint32, n // g)[7] ^= 1
        lines = [m for r in pool.run(parts) for m in r["mismatches"]]
        assert any("stage 3 codes" in m and "element 1000:" in m for m in lines), lines
        assert any("prefix 1:" in m and f"element {n - 1}:" in m for m in lines), lines
        assert any("prefix 3:" in m and "element 5:" in m for m in lines), lines
        assert any("stage 2 scales" in m and "element 0:" in m for m in lines), lines
        assert any("stage 1 zeros" in m and "element 7:" in m for m in lines) == bool(zeros), lines
        assert len(lines) == (5 if zeros else 4)


def test_host_description():
    d = host_description()
    assert d["cores"] >= 1 and isinstance(d["cpu_model"], str) and d["cpu_model"]
