"""GPU generator parity: Philox words bit-exact with the oracle, the word -> normal
transform against the oracle's exact quantile on all 2^23 inputs it can see, and the
normals of global indices (including beyond 2^32 and across tags)."""
import numpy as np
import pytest
import torch

import oracle
from tolerances import assert_normals_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def copes():
    from paper_2608_02391_gb300 import copes as c
    c.load()
    return c


@pytest.mark.parametrize("seed,q0,aux,tag", [
    (0, 0, 0, 0), (33, 1 << 32, 0, 0), (0xFFFFFFFFFFFFFFFF, (1 << 40) - 7, 5, 2),
    (1234567, 99, 0, 1), (2**63 + 1, 0, 0xFFFFFFFF, 4)])
def test_philox_words_bit_exact(copes, seed, q0, aux, tag):
    n = 4099
    got = copes.debug_philox(seed, q0, n, aux, tag).cpu().numpy().view(np.uint32).reshape(n, 4)
    ref = oracle.philox_stream(seed, q0, n, aux, tag)
    assert np.array_equal(got, ref)


def test_philox_known_answer_vectors(copes):
    # KAT 0: counter 0, key 0 (SC'11 / Random123): seed 0, q 0, aux 0, tag 0
    got = copes.debug_philox(0, 0, 1, 0, 0).cpu().numpy().view(np.uint32)
    assert list(got) == [0x6627e8d5, 0xe169c58d, 0xbc57ac4c, 0x9b00dbd8]
    # KAT 1: all-ones counter and key
    got = copes.debug_philox(0xFFFFFFFFFFFFFFFF, 0xFFFFFFFFFFFFFFFF, 1, 0xFFFFFFFF, 0xFFFFFFFF)
    assert list(got.cpu().numpy().view(np.uint32)) == [0x408f276d, 0x41c83b0e, 0xa20bc7c6, 0x6d5451fd]


def test_transform_exhaustive(copes):
    """Every distinct uniform the transform can see: words 2m, m < 2^22 (bits 1..22),
    plus the same words with the ignored bits set."""
    m = torch.arange(1 << 22, dtype=torch.int64, device="cuda")
    words = (2 * m).to(torch.int32)
    got = copes.debug_transform(words).cpu().numpy().astype(np.float64)
    noisy = (2 * m + 1 + (0x1FF << 23)).to(torch.int32)  # bit 0 and bits 23..31 set
    assert np.array_equal(copes.debug_transform(noisy).cpu().numpy().astype(np.float64), got)
    u = (2.0 * np.arange(1 << 22, dtype=np.float64) + 1.0) * 2.0**-23
    ref = oracle.normal_quantile_array(u)
    assert_normals_close(got, ref)
    rel = np.abs(got - ref) / np.abs(ref)
    # relative accuracy everywhere, including near the centre and the tails
    assert rel.max() < 6e-7, rel.max()
    # the odd symmetry of the transform survives in fp32 (x and -x are both exact)
    assert np.array_equal(got, -got[::-1])


@pytest.mark.parametrize("seed,g0,tag", [(33, 0, 0), (7, (1 << 34) + 3, 0), (0, 12345, 1)])
def test_normals_of_global_indices(copes, seed, g0, tag):
    n = 100_003
    got = copes.debug_normals(seed, g0, n, tag).cpu().numpy()
    ref = oracle.noise_range(seed, g0, n, tag)
    assert_normals_close(got, ref)


def test_normal_statistics_on_device(copes):
    n = 1 << 24
    x = copes.debug_normals(2026, 0, n).double()
    se = 1.0 / np.sqrt(n)
    assert abs(x.mean().item()) < 5 * se
    assert abs(x.var(unbiased=False).item() - 1.0) < 5 * np.sqrt(2.0 / n)
    z = x.cpu().numpy()
    from scipy import stats
    assert abs(stats.skew(z)) < 5 * np.sqrt(6.0 / n)
    assert abs(stats.kurtosis(z)) < 5 * np.sqrt(24.0 / n)
