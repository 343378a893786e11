"""The committed CPU oracle against facts fixed by the paper and by
mathematics (see tests/_pins.py for each pin and its source)."""
import numpy as np
import pytest

import oracle
import _pins


@pytest.fixture(scope="module")
def orc():
    return oracle.load()


@pytest.mark.parametrize("pin", _pins.ALL_PINS, ids=lambda p: p.__name__)
def test_pin_holds(orc, pin):
    fails = pin(orc)
    assert not fails, "\n".join(fails[:10])


def test_oracle_is_deterministic(orc):
    rng = np.random.default_rng(1)
    W = (rng.normal(0, 0.02, (8, 256)).astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    a = orc.quantize(W, 128, 4)
    b = orc.quantize(W, 128, 4)
    for x, y in zip(a, b):
        for u, v in zip(x, y):
            assert np.array_equal(u.view(np.uint8), v.view(np.uint8))


def test_oracle_rejects_bad_arguments(orc):
    W = np.zeros((2, 100), np.uint16)
    with pytest.raises(ValueError):
        orc.quantize(W, group=128, n_stages=4)  # cols % group != 0
    with pytest.raises(ValueError):
        orc.quantize_group(np.zeros(0, np.float32), 4)


def test_package_size_closed_form(orc):
    """Bytes of the package in this layout: per stage n/4 code bytes plus
    n/group fp32 scales and fp32 zeros, i.e. 3 + 32/group bytes per weight
    for 4 stages together with the 2-byte bf16 input read once."""
    rows, cols, g = 4, 512, 128
    W = np.zeros((rows, cols), np.uint16)
    codes, scales, zeros = orc.quantize(W, g, 4)
    n = rows * cols
    total = sum(c.nbytes for c in codes) + sum(s.nbytes for s in scales) + sum(z.nbytes for z in zeros)
    assert total == 4 * (n // 4 + 8 * n // g)
    assert (2 * n + total) / n == 3 + 32 / g


def test_paper_size_estimate_formula():
    """Appendix G: Size_b = Size_16 * (b + 16/128) / 16 reproduces the
    paper's Table 11 estimates for Qwen3-8B from its Table 10 16-bit size."""
    size16 = 13_581_708
    est = {b: size16 * (b + 16 / 128) / 16 for b in (8, 6, 4, 3, 2)}
    printed = {8: 6_896_961, 6: 5_199_248, 4: 3_501_534, 3: 2_652_677, 2: 1_803_821}
    for b, v in printed.items():
        assert abs(est[b] - v) <= 1, (b, est[b], v)
    # Table 12: the separate (2,4,6,8) estimate is the sum of the four rows
    assert abs(sum(est[b] for b in (2, 4, 6, 8)) - 17_401_564) <= 2
