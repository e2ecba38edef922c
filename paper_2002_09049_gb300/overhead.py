"""Deployment overhead of multipoint quantization (Sec. 3.4, Table 1), as closed forms.

A channel of d weights quantized with N-bit codes and dotted with an N-bit input costs, in the
paper's bit-operation count: memory d*N bits, d*N^2 binary MULs and (d-1)*N ADDs.  With n points,
each point adds its own code vector and a 32-bit integer coefficient A_i (Eq. 13): memory
n*d*N + 32n, MULs n*(d*N^2 + 32^2), ADDs n*(d-1)*N + 32*(n-1).  Used for reporting the model-size
and OPs overhead of an allocation.
"""
from __future__ import annotations


def naive_cost(d: int, nbits: int) -> dict:
    return dict(memory_bits=d * nbits, muls=d * nbits * nbits, adds=(d - 1) * nbits)


def multipoint_cost(d: int, nbits: int, n: int) -> dict:
    return dict(memory_bits=n * d * nbits + 32 * n,
                muls=n * (d * nbits * nbits + 32 * 32),
                adds=n * (d - 1) * nbits + 32 * (n - 1))


def layer_overhead(npoints, d: int, nbits: int) -> dict:
    """Ratios (multipoint / naive) of memory, MULs and ADDs for one layer given its per-channel
    point counts."""
    tot = dict(memory_bits=0, muls=0, adds=0)
    base = dict(memory_bits=0, muls=0, adds=0)
    nv = naive_cost(d, nbits)
    for n in npoints:
        c = multipoint_cost(d, nbits, int(n))
        for key in tot:
            tot[key] += c[key]
            base[key] += nv[key]
    return {key: tot[key] / base[key] for key in tot}
