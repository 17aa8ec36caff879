"""Pins the oracle's Philox4x64-10 against numpy's independent implementation of the
same published generator (numpy.random.Philox)."""
import numpy as np
import pytest

from oracle.philox import CUTOFF_KEY_TAG, MASK64, cutoff_uniform62, philox4x64_10


def _numpy_block(counter, key):
    # numpy increments its 256-bit counter before producing a block, so start one below.
    c = (counter[0] | (counter[1] << 64) | (counter[2] << 128) | (counter[3] << 192)) - 1
    c %= 1 << 256
    words = np.array([(c >> (64 * i)) & MASK64 for i in range(4)], dtype=np.uint64)
    bg = np.random.Philox(key=np.array(key, dtype=np.uint64), counter=words)
    return tuple(int(x) for x in bg.random_raw(4))


@pytest.mark.parametrize("counter,key", [
    ((1, 0, 0, 0), (0, 0)),
    ((0, 0, 0, 0), (0, 0)),
    ((7, 3, 0, 0), (123456789, CUTOFF_KEY_TAG)),
    ((MASK64, MASK64, MASK64, MASK64), (MASK64, MASK64)),
    ((0x243F6A8885A308D3, 0x13198A2E03707344, 0xA4093822299F31D0, 0x082EFA98EC4E6C89),
     (0x452821E638D01377, 0xBE5466CF34E90C6C)),
])
def test_block_matches_numpy(counter, key):
    assert philox4x64_10(counter, key) == _numpy_block(counter, key)


def test_cutoff_stream_matches_numpy():
    for seed in (0, 1, 2**63 + 5):
        for step in (0, 1, 17):
            for k in range(1, 40):
                ref = _numpy_block((k, step, 0, 0), (seed, CUTOFF_KEY_TAG))[0] >> 2
                assert cutoff_uniform62(seed, step, k) == ref
                assert 0 <= ref < (1 << 62)


def test_reward_stream_matches_numpy():
    from oracle.philox import REWARD_KEY_TAG, reward_uniform53
    assert REWARD_KEY_TAG != CUTOFF_KEY_TAG
    for seed in (0, 3, 2**64 - 1):
        for step in (0, 9):
            for k in range(1, 30):
                ref = _numpy_block((k, step, 0, 0), (seed, REWARD_KEY_TAG))[0] >> 11
                assert reward_uniform53(seed, step, k) == ref
                assert 0 <= ref < (1 << 53)
