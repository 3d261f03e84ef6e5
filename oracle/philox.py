"""Philox4x32-10 counter-based generator (oracle side).

Written from the published definition in Salmon, Moraes, Dror and Shaw,
"Parallel random numbers: as easy as 1, 2, 3" (SC'11): a 4x32-bit counter and
a 2x32-bit key; each of the 10 rounds multiplies counter words 0 and 2 by two
fixed odd constants, swaps and XORs the high halves with the other counter
words and the key, and the key is bumped by two Weyl constants between rounds.

The paper being implemented (1-Bit FQT, Sec. 3.2) only requires stochastic
rounding to be unbiased; it does not name a generator.  Every random draw of
the method is a pure function of (seed, stream, index) through `uniform_u32`
so that any implementation can reproduce it.

Test infrastructure: this package is imported only by tests, the smoke check
and the CPU-baseline leg of the benchmark.
"""
import numpy as np

_M0 = np.uint64(0xD2511F53)   # round multiplier applied to counter word 0
_M1 = np.uint64(0xCD9E8D57)   # round multiplier applied to counter word 2
_W0 = 0x9E3779B9              # key bump (golden ratio)
_W1 = 0xBB67AE85              # key bump (sqrt(3) - 1)
_MASK32 = np.uint64(0xFFFFFFFF)
_SH32 = np.uint64(32)


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Apply Philox4x32 with 10 rounds element-wise.

    c0..c3 are arrays (or scalars) of 32-bit counter words, k0/k1 the two key
    words (python ints).  Returns four uint32 arrays.
    """
    x0 = np.asarray(c0, dtype=np.uint64) & _MASK32
    x1 = np.asarray(c1, dtype=np.uint64) & _MASK32
    x2 = np.asarray(c2, dtype=np.uint64) & _MASK32
    x3 = np.asarray(c3, dtype=np.uint64) & _MASK32
    x0, x1, x2, x3 = np.broadcast_arrays(x0, x1, x2, x3)
    key0, key1 = int(k0) & 0xFFFFFFFF, int(k1) & 0xFFFFFFFF
    for _ in range(10):
        p0 = x0 * _M0            # full 64-bit products of 32-bit words
        p1 = x2 * _M1
        hi0, lo0 = p0 >> _SH32, p0 & _MASK32
        hi1, lo1 = p1 >> _SH32, p1 & _MASK32
        x0, x1, x2, x3 = (hi1 ^ x1 ^ np.uint64(key0), lo1,
                          hi0 ^ x3 ^ np.uint64(key1), lo0)
        key0 = (key0 + _W0) & 0xFFFFFFFF
        key1 = (key1 + _W1) & 0xFFFFFFFF
    return (x0.astype(np.uint32), x1.astype(np.uint32),
            x2.astype(np.uint32), x3.astype(np.uint32))


def uniform_u32(seed, stream, index):
    """32-bit random word number `index` of stream `stream` under `seed`.

    Word i is word (i mod 4) of Philox4x32-10 with key (seed low 32 bits,
    seed high 32 bits) and counter (i div 4 low 32 bits, i div 4 high 32 bits,
    stream, 0).
    """
    idx = np.asarray(index, dtype=np.uint64)
    blk = idx >> np.uint64(2)
    seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    r = philox4x32_10(blk & _MASK32, blk >> _SH32, np.uint64(stream), np.uint64(0),
                      seed & 0xFFFFFFFF, seed >> 32)
    words = np.stack(r, axis=-1)
    lane = (idx & np.uint64(3)).astype(np.int64)
    return np.take_along_axis(words, lane[..., None], axis=-1)[..., 0]
