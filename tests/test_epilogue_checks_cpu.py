"""The bounded-parity checks used for the fused SwiGLU epilogues accept what
the quantizer's recipe produces within the stated approximation error and
reject a misplaced scale or code.  Runs on the CPU (no kernel involved)."""
import numpy as np
import pytest

from _util import assert_mxfp4_within, assert_nvfp4_within, rotated_tolerance, swiglu_tolerance
from oracle import mxfp4_oracle as X
from oracle import nvfp4_oracle as O


def _h():
    rng = np.random.default_rng(0)
    G = rng.standard_normal((64, 256)) * 2
    U = rng.standard_normal((64, 256))
    h = O.silu(G) * U
    return h, swiglu_tolerance(G, U, h)


def test_nvfp4_check_accepts_the_recipe_and_rejects_planted_mistakes():
    h, tol = _h()
    g = O.tensor_scale(h.astype(np.float32))
    c, s = O.quantize(h.astype(np.float32), g)
    assert_nvfp4_within(c, s, h, tol, g)
    # h moved inside the bound by half of it: still the recipe's output for some h'
    c2, s2 = O.quantize((h + 0.5 * tol).astype(np.float32), g)
    assert_nvfp4_within(c2, s2, h, tol, g)
    s_bad = s.copy()
    s_bad[3, 5] += 1
    with pytest.raises(AssertionError, match="block scales"):
        assert_nvfp4_within(c, s_bad, h, tol, g)
    c_bad = c.copy()
    c_bad[7, 9] ^= 0x11
    with pytest.raises(AssertionError, match="codes"):
        assert_nvfp4_within(c_bad, s, h, tol, g)


@pytest.mark.parametrize("rotate", [False, True])
def test_mxfp4_check_accepts_the_recipe_and_rejects_planted_mistakes(rotate):
    h, tol = _h()
    c, s = X.quantize_mx(h.astype(np.float32), rotate=rotate)
    t = X.rotate_blocks(h) if rotate else h
    tt = rotated_tolerance(h, tol) if rotate else tol
    assert_mxfp4_within(c, s, t, tt)
    s_bad = s.copy()
    s_bad[1, 2] += 1
    with pytest.raises(AssertionError, match="block scales"):
        assert_mxfp4_within(c, s_bad, t, tt)
    c_bad = c.copy()
    c_bad[2, 3] ^= 0x22
    with pytest.raises(AssertionError, match="codes"):
        assert_mxfp4_within(c_bad, s, t, tt)
