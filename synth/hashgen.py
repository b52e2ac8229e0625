"""Counter-based generator for the initial parameter store.

The store of the large workloads (11M x 200, 5M x 512, 100M x 64 floats) is
generated on the GPU, while a CPU checker needs the same rows for a sample of
keys.  Both sides therefore derive every initial value from an integer hash of
(seed, key, column) with integer arithmetic only, and convert the integer to a
float by one IEEE double multiply and one round-to-nearest cast, which numpy
and torch (CPU or CUDA) perform identically.  The result is bit-identical on
every backend.

Hash: the 32-bit "lowbias32" mixer (xor-shift 16, multiply 0x7feb352d,
xor-shift 15, multiply 0x846ca68b, xor-shift 16) published with Chris
Wellons' hash-prospector.  Multiplications are done modulo 2^32 on 16-bit
halves so that no intermediate exceeds 2^49 (safe in signed int64 torch
tensors as well as in numpy).

Value families
  normal_ih4  Irwin-Hall sum of four 16-bit uniforms, centred and scaled to a
              requested standard deviation: a bounded, near-normal value
              (kurtosis 2.7) used for "init N(0, sigma)".
  dyadic      integers in [-1024, 1024] times 2^-10: every sum of a few
              thousand of them is exact in fp32, which makes results of any
              summation order bit-identical.
"""
import math

import numpy as np

_M32 = 0xFFFFFFFF


def _mul32(x, c):
    """(x * c) mod 2^32 for 0 <= x < 2^32 without intermediates above 2^49."""
    lo = x & 0xFFFF
    hi = x >> 16
    return (lo * c + (((hi * c) & 0xFFFF) << 16)) & _M32


def lowbias32(x):
    """lowbias32 mixer on an int64 array/tensor holding values in [0, 2^32)."""
    x = x ^ (x >> 16)
    x = _mul32(x, 0x7FEB352D)
    x = x ^ (x >> 15)
    x = _mul32(x, 0x846CA68B)
    x = x ^ (x >> 16)
    return x


def _seed_word(seed, salt):
    # plain Python ints: the same on every backend
    v = (int(seed) * 0x9E3779B9 + int(salt) * 0x632BE5AB + 0x165667B1) & _M32
    v ^= v >> 16
    v = (v * 0x7FEB352D) & _M32
    v ^= v >> 15
    v = (v * 0x846CA68B) & _M32
    v ^= v >> 16
    return v


def hash2(keys, cols, seed, salt=0):
    """Two independent 32-bit hash words of (seed, salt, key, col).

    keys, cols: broadcastable int64 arrays/tensors with 0 <= key, col < 2^32.
    """
    s0 = _seed_word(seed, 2 * salt)
    s1 = _seed_word(seed, 2 * salt + 1)
    hk = lowbias32(keys ^ s0)
    h0 = lowbias32(hk ^ lowbias32((cols ^ s1) & _M32))
    h1 = lowbias32(h0 ^ 0x5BD1E995)
    return h0, h1


_IH4_MEAN = 2 * 65535          # mean of the sum of four 16-bit uniforms
_IH4_STD = math.sqrt(4 * (65536.0 ** 2 - 1) / 12.0)


def _ih4_int(h0, h1):
    return ((h0 & 0xFFFF) + (h0 >> 16) + (h1 & 0xFFFF) + (h1 >> 16)) - _IH4_MEAN


def normal_ih4_np(keys, cols, seed, std, salt=0):
    """float32 values ~ near-normal(0, std) for int64 numpy keys x cols."""
    keys = np.asarray(keys, dtype=np.int64)
    cols = np.asarray(cols, dtype=np.int64)
    h0, h1 = hash2(keys, cols, seed, salt)
    return (_ih4_int(h0, h1).astype(np.float64) * (std / _IH4_STD)).astype(np.float32)


def normal_ih4_torch(keys, cols, seed, std, salt=0):
    """The same values as normal_ih4_np, for int64 torch tensors (any device)."""
    import torch
    h0, h1 = hash2(keys, cols, seed, salt)
    return (_ih4_int(h0, h1).to(torch.float64) * (std / _IH4_STD)).to(torch.float32)


def dyadic_np(keys, cols, seed, half_range=1024, salt=0):
    """float32 multiples of 2^-10 in [-half_range, half_range] * 2^-10."""
    keys = np.asarray(keys, dtype=np.int64)
    cols = np.asarray(cols, dtype=np.int64)
    h0, _ = hash2(keys, cols, seed, salt)
    ints = (h0 % (2 * half_range + 1)) - half_range
    return (ints.astype(np.float64) * 2.0 ** -10).astype(np.float32)


def dyadic_torch(keys, cols, seed, half_range=1024, salt=0):
    import torch
    h0, _ = hash2(keys, cols, seed, salt)
    ints = (h0 % (2 * half_range + 1)) - half_range
    return (ints.to(torch.float64) * 2.0 ** -10).to(torch.float32)


# --------------------------------------------------------------------------
# whole-row initialisers: value row = [theta (theta_dim) | zeros (rest)]
# --------------------------------------------------------------------------

def init_rows_np(keys, value_len, theta_dim, seed, std, kind="normal"):
    """Initial rows for the given keys, shape (len(keys), value_len) float32.

    Columns [0, theta_dim) carry the parameter; columns [theta_dim, value_len)
    (an AdaGrad accumulator, when present) start at zero.
    """
    keys = np.asarray(keys, dtype=np.int64).reshape(-1, 1)
    cols = np.arange(theta_dim, dtype=np.int64).reshape(1, -1)
    out = np.zeros((keys.shape[0], value_len), dtype=np.float32)
    if kind == "normal":
        out[:, :theta_dim] = normal_ih4_np(keys, cols, seed, std)
    elif kind == "dyadic":
        out[:, :theta_dim] = dyadic_np(keys, cols, seed)
    else:
        raise ValueError(kind)
    return out


def init_store_torch(num_keys, value_len, theta_dim, seed, std, device, kind="normal",
                     chunk_rows=1 << 20, out=None):
    """The whole initial store on `device`, generated in chunks of rows.

    Bit-identical to init_rows_np(arange(num_keys), ...).
    """
    import torch
    if out is None:
        out = torch.zeros((num_keys, value_len), dtype=torch.float32, device=device)
    else:
        out.zero_()
    cols = torch.arange(theta_dim, dtype=torch.int64, device=device).view(1, -1)
    for r0 in range(0, num_keys, chunk_rows):
        r1 = min(num_keys, r0 + chunk_rows)
        keys = torch.arange(r0, r1, dtype=torch.int64, device=device).view(-1, 1)
        if kind == "normal":
            out[r0:r1, :theta_dim] = normal_ih4_torch(keys, cols, seed, std)
        elif kind == "dyadic":
            out[r0:r1, :theta_dim] = dyadic_torch(keys, cols, seed)
        else:
            raise ValueError(kind)
    return out
