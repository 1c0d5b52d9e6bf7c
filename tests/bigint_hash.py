"""Independent evaluation of the PSS location hash with Python integers.

Used only to pin the oracle: arbitrary-precision arithmetic, no 128-bit
folding, no shared code with either implementation under test.
"""
P61 = (1 << 61) - 1


def bucket(A: int, B0: int, R: int, key: int) -> int:
    return ((A * key + B0) % P61) % R


def location(A, B0, R, G, T, J, i, t, j) -> int:
    key = (i * T + t) * J + j
    return G * bucket(A, B0, R, key)


def params(seed: int):
    """(A, B0) from the splitmix64 stream seeded with ``seed``."""
    mask = (1 << 64) - 1
    state = seed
    outs = []
    for _ in range(2):
        state = (state + 0x9E3779B97F4A7C15) & mask
        z = state
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & mask
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & mask
        outs.append(z ^ (z >> 31))
    return 1 + outs[0] % (P61 - 1), outs[1] % P61


def sign_params(seed: int):
    """(A2, B2) of the sign hash: the third and fourth splitmix64 outputs."""
    mask = (1 << 64) - 1
    state = seed
    outs = []
    for _ in range(4):
        state = (state + 0x9E3779B97F4A7C15) & mask
        z = state
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & mask
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & mask
        outs.append(z ^ (z >> 31))
    return 1 + outs[2] % (P61 - 1), outs[3] % P61


def sign(A2, B2, T, J, i, t, j) -> int:
    """-1 when the sign hash of key (i, t, j) is odd, else +1."""
    key = (i * T + t) * J + j
    return -1 if ((A2 * key + B2) % P61) & 1 else 1
