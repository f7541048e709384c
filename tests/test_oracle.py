"""The fp64 oracle against closed forms, invariants, a library and brute force (CPU only)."""
import pytest

import oracle_pins


@pytest.mark.parametrize("pin", oracle_pins.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(orc, pin):
    pin(orc)


def test_rejects_bad_rows(orc):
    import numpy as np
    q = np.zeros((1, 1, 4, 8), np.uint16)
    with pytest.raises(RuntimeError):
        orc.attn_fwd(q, q, q, 1.0, rows=np.array([[4]], np.int32))


def test_threads(orc):
    assert orc.set_threads(0) >= 1
