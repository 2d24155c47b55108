"""The CPU oracle against its pins (values and invariants fixed by the paper and
by mathematics, not by the oracle); no GPU needed."""
import pytest

import oracle
import oracle_pins


@pytest.mark.parametrize("pin", oracle_pins.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    pin(oracle.load())


def test_degenerate_inputs_rejected():
    import numpy as np
    q = np.zeros((0, 2, 4), np.float32)
    k = np.zeros((3, 2, 4), np.float32)
    with pytest.raises(oracle.OracleError):  # visual tokens without any text query
        oracle.score(q, k, [0, 3], [0, 0], 2, 2, 4, "f32")
    with pytest.raises(oracle.OracleError):  # k larger than the request
        oracle.topk([0, 3], np.zeros(3, np.float32), keep_k=[4])
    with pytest.raises(oracle.OracleError):  # Hq not a multiple of Hkv
        oracle.score(np.zeros((1, 3, 4), np.float32), k, [0, 3], [0, 1], 3, 2, 4, "f32")
    kept, off = oracle.topk([0, 0, 3], np.ones(3, np.float32), keep_k=[0, 0])
    assert kept.size == 0 and off.tolist() == [0, 0, 0]
