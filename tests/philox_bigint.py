"""A second Philox4x32-10, written independently of the oracle from the SC'11 description
(Salmon, Moraes, Dror, Shaw, "Parallel Random Numbers: As Easy as 1, 2, 3"), in Python
integers.  It pins the oracle's generator; it is not used by either implementation."""

MULT = (0xD2511F53, 0xCD9E8D57)
WEYL = (0x9E3779B9, 0xBB67AE85)
M32 = (1 << 32) - 1


def philox(counter, key, rounds=10):
    x = list(counter)
    k = list(key)
    for _ in range(rounds):
        a = MULT[0] * x[0]
        b = MULT[1] * x[2]
        x = [(b >> 32) ^ x[1] ^ k[0], b & M32, (a >> 32) ^ x[3] ^ k[1], a & M32]
        k = [(k[0] + WEYL[0]) & M32, (k[1] + WEYL[1]) & M32]
    return tuple(v & M32 for v in x)


def words(seed, q, aux=0, tag=0):
    """This project's counter layout: (q low, q high, aux, tag), key (seed low, seed high)."""
    return philox((q & M32, q >> 32, aux, tag), (seed & M32, seed >> 32))
