"""Philox4x64-10, from its published definition.

J. K. Salmon, M. A. Moraes, R. O. Dror, D. E. Shaw, "Parallel Random Numbers: As
Easy as 1, 2, 3", SC'11. One block maps a 4-word counter and a 2-word key to 4
64-bit words through 10 rounds. Each round multiplies counter words 0 and 2 by
fixed constants, takes the high and low halves of the 128-bit products, mixes
the high halves with the other two counter words and the key, and permutes; the
key is bumped by the Weyl increments between rounds.

Written with Python integers (exact 128-bit products); test infrastructure only.
"""
MASK64 = (1 << 64) - 1
PHILOX_M4x64_0 = 0xD2E7470EE14C6C93
PHILOX_M4x64_1 = 0xCA5A826395121157
PHILOX_W64_0 = 0x9E3779B97F4A7C15   # golden ratio
PHILOX_W64_1 = 0xBB67AE8584CAA73B   # sqrt(3) - 1

# Key word 1 of the cutoff sampler's stream: the ASCII bytes "PSPP0001".
CUTOFF_KEY_TAG = 0x5053505030303031


def _mulhilo(a: int, b: int):
    p = a * b
    return (p >> 64) & MASK64, p & MASK64


def philox4x64_10(counter, key):
    """One Philox4x64 block with 10 rounds. counter: 4 ints, key: 2 ints -> 4 ints."""
    c0, c1, c2, c3 = (int(x) & MASK64 for x in counter)
    k0, k1 = (int(x) & MASK64 for x in key)
    for r in range(10):
        if r > 0:
            k0 = (k0 + PHILOX_W64_0) & MASK64
            k1 = (k1 + PHILOX_W64_1) & MASK64
        hi0, lo0 = _mulhilo(PHILOX_M4x64_0, c0)
        hi1, lo1 = _mulhilo(PHILOX_M4x64_1, c2)
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return c0, c1, c2, c3


def cutoff_uniform62(seed: int, step: int, traj: int) -> int:
    """The 62-bit uniform integer that decides trajectory `traj`'s cutoff.

    key = (seed, tag), counter = (global trajectory index, step, 0, 0); the first
    output word shifted right by 2 is uniform on [0, 2^62).
    """
    out = philox4x64_10((traj, step, 0, 0), (seed, CUTOFF_KEY_TAG))
    return out[0] >> 2


# Key word 1 of the reward-binarisation stream: the ASCII bytes "PSPPRWD1".
REWARD_KEY_TAG = 0x5053505052574431


def reward_uniform53(seed: int, step: int, traj: int) -> int:
    """The 53-bit uniform integer that binarises trajectory `traj`'s reward for u_t.

    key = (seed, "PSPPRWD1"), counter = (global trajectory index, step, 0, 0); the first output
    word shifted right by 11 is uniform on [0, 2^53), i.e. u = k 2^-53 on [0, 1).
    """
    out = philox4x64_10((traj, step, 0, 0), (seed, REWARD_KEY_TAG))
    return out[0] >> 11
