"""Pins of the attention oracle (CPU only): see ``oracle_pins`` for what each
check compares against."""

import numpy as np
import pytest

import oracle_pins
from oracle import attention as att


@pytest.mark.parametrize("pin", oracle_pins.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    pin(att)


def test_streaming_cache_image_layout():
    """Sinks land in slots 0..S-1 and position p >= S in slot S + (p - S) mod W."""
    S, W, T, d = 3, 4, 13, 2
    k = np.arange(T * d, dtype=np.float64).reshape(T, d)
    img, written = att.streaming_cache_image(k, S, W)
    assert written.all()
    # positions held: sinks 0,1,2 and the last four 9..12
    want_pos = {0: 0, 1: 1, 2: 2}
    for p in range(9, 13):
        want_pos[S + (p - S) % W] = p
    for slot, p in want_pos.items():
        np.testing.assert_array_equal(img[slot], k[p])


def test_short_sequence_leaves_slots_unwritten():
    S, W = 4, 8
    k = np.ones((6, 2))
    _, written = att.streaming_cache_image(k, S, W)
    assert written.tolist() == [True] * 6 + [False] * 6


def test_rejects_bad_group_split():
    q = np.zeros((2, 3, 4))
    k = np.zeros((2, 2, 4))
    with pytest.raises(ValueError):
        att.prefill(q, k, k, [0, 0], 1, 1)
