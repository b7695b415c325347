"""The decode-attention kernel's work split, restated on the host (CPU): the n_heads * ceil(L / 16)
units of 16 positions, head-major, go to warp z as [z U / Z, (z + 1) U / Z).  The kernel keeps at
most two partial results per warp and its merge finds each head's covering warps by search; both
rest on facts checked here for the 7B-class head count and contexts from 1 to 32K positions, and
for head counts up to the warp count (the host rejects more)."""
import pytest

Z = 152 * 8


def seg(z, U):
    return z * U // Z


def covering(h, nch, U):
    """The merge kernel's search: the warps holding the head's first and last unit."""
    ua, ub = h * nch, h * nch + nch - 1
    zlo = ua * Z // U
    while zlo > 0 and seg(zlo, U) > ua:
        zlo -= 1
    while seg(zlo + 1, U) <= ua:
        zlo += 1
    zhi = ub * Z // U
    while zhi > 0 and seg(zhi, U) > ub:
        zhi -= 1
    while seg(zhi + 1, U) <= ub:
        zhi += 1
    return zlo, zhi


@pytest.mark.parametrize("n_heads,L", [(32, 1), (32, 15), (32, 16), (32, 17), (32, 2048), (32, 2047), (32, 32768),
                                       (1, 5), (7, 1000), (1216, 16), (1216, 33), (600, 100)])
def test_partition_facts(n_heads, L):
    nch = -(-L // 16)
    U = n_heads * nch
    heads_of = {}
    for z in range(Z):
        u0, u1 = seg(z, U), seg(z + 1, U)
        heads = {u // nch for u in range(u0, u1)}
        assert len(heads) <= 2                      # at most two partial records per warp
        for h in heads:
            heads_of.setdefault(h, []).append(z)
    for h in range(n_heads):
        zlo, zhi = covering(h, nch, U)
        # the search finds exactly the warps whose units include the head's (empty warps between
        # them are skipped by the merge)
        nonempty = [z for z in range(zlo, zhi + 1) if seg(z + 1, U) > seg(z, U)]
        assert nonempty == heads_of[h]
        for z in nonempty:                          # the record the merge reads is the one the warp wrote
            first = seg(z, U) // nch
            rec = 0 if first == h else 1
            assert rec == sorted({u // nch for u in range(seg(z, U), seg(z + 1, U))}).index(h)
