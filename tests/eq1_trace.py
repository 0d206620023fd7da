"""Shared check of Eq. 1's reuse semantics on a device trace (the residual
added at every lattice cell, [T][U][N][H][E] float32): a cell the lattice
skips adds exactly the cached value stored at the unit's last refresh -- in
bf16 mode the refresh's output rounded to bfloat16 (round to nearest even),
bit for bit -- and a cell whose unit has not been refreshed yet in the query
adds zero (the reset cache)."""
import numpy as np


def round_bf16_f32(x):
    """float32 -> nearest bfloat16 value (ties to even), as float32."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return u.astype(np.uint32).view(np.float32)


def check_reuse(trace, S, bf16: bool, force: bool = False):
    """trace [T][U][...], S [U][T] unit lattice.  Returns the number of skipped
    cells checked against a stored value."""
    T, U = trace.shape[:2]
    last = {}
    n = 0
    for t in range(T):
        for b in range(U):
            refreshed = bool(S[b, t]) or (force and t == 0)
            if refreshed:
                last[b] = round_bf16_f32(trace[t, b]) if bf16 else trace[t, b].copy()
                if bf16:
                    assert not np.array_equal(last[b], trace[t, b]), "refresh traced after rounding"
            elif b in last:
                assert np.array_equal(trace[t, b].view(np.uint32), last[b].view(np.uint32)), (t, b)
                n += 1
            else:
                assert not trace[t, b].any(), (t, b)
    return n
