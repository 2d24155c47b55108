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


@pytest.mark.parametrize("name,threads", [("tiny", 3), ("single", 4), ("fp8_ragged", 7), ("gqa", 16), ("ragged", 5)])
def test_threaded_scores_equal_the_serial_oracle_bit_for_bit(name, threads):
    # the all-cores score of the CPU baseline keeps the serial summation order,
    # so its scores are the serial oracle's, bit for bit
    import math
    import numpy as np
    from paper_2506_07416_gb300 import inputs
    if name == "gqa":
        w = inputs.Workload("gqa", 2, [300, 129], [40, 7], 28, 4, 128, 256, "bf16", keep_ratio=0.3,
                            sigma=1.0 / math.sqrt(128), seed=5)
    elif name == "ragged":
        w = inputs.Workload("ragged", 5, [1, 0, 257, 64, 3], [9, 4, 16, 1, 2], 4, 2, 64, 256, "bf16",
                            keep_ratio=0.3, sigma=1.0, seed=6)
    elif name == "fp8_ragged":
        w = inputs.sub_batch(inputs.workload("fp8_ragged"), [0, 1])
    else:
        w = inputs.workload(name)
    x = inputs.make_numpy(w)
    args = (x["q"], x["k"], x["seq_offsets"], x["text_offsets"], w.hq, w.hkv, w.head_dim, w.dtype,
            x.get("q_scale", 1.0), x.get("k_scale", 1.0))
    serial = oracle.score(*args)
    par = oracle.score_threads(*args, threads=threads)
    assert np.array_equal(serial.view(np.uint32), par.view(np.uint32))
