"""The bucket test of the replayed hash partition (Eq. 7, Supp. A.8 partition replay).

Element membership in subspace k of the hash partition (K, seed) is
floor(x K / 2^32) == k for its Philox word x.  The replay kernels evaluate the same
predicate as one unsigned range test, (x - lo) mod 2^32 <= span, with
lo = ceil(k 2^32 / K) and span = ceil((k + 1) 2^32 / K) - lo - 1 computed on the host.
This checks that the two agree for every k < K <= 64 at the range edges and on random
words; the GPU tests then check the kernels against the index lists."""
import numpy as np

TWO32 = 1 << 32


def bounds(K, k):
    lo = (k * TWO32 + K - 1) // K
    hi = ((k + 1) * TWO32 + K - 1) // K
    return lo, hi - lo - 1


def in_range(x, lo, span):
    return ((x - lo) % TWO32) <= span


def test_range_test_equals_bucket_at_edges():
    for K in range(1, 65):
        for k in range(K):
            lo, span = bounds(K, k)
            assert 0 <= span < TWO32
            hi = lo + span + 1
            for x in {0, 1, TWO32 - 1, lo - 1, lo, lo + 1, hi - 2, hi - 1, hi, hi + 1}:
                if 0 <= x < TWO32:
                    assert in_range(x, lo, span) == ((x * K) >> 32 == k), (K, k, x)


def test_range_test_equals_bucket_on_random_words():
    rng = np.random.default_rng(7)
    x = rng.integers(0, TWO32, size=1 << 16, dtype=np.uint64)
    for K in (1, 2, 3, 7, 16, 33, 64):
        bucket = (x * np.uint64(K)) >> np.uint64(32)
        hits = np.zeros(x.size, np.int64)
        for k in range(K):
            lo, span = bounds(K, k)
            m = ((x - np.uint64(lo)) & np.uint64(TWO32 - 1)) <= np.uint64(span)
            assert np.array_equal(m, bucket == k)
            hits += m
        assert np.all(hits == 1)  # the K ranges tile the words


def test_single_bucket_takes_every_word():
    lo, span = bounds(1, 0)
    assert lo == 0 and span == TWO32 - 1
