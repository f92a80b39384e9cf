"""The tensor-core backward's item order (one launch, Algorithm 1's reverse
sweep), read from the library through slim_bwd_schedule: pure host code, no GPU.

The launch hands out items by ticket.  Its progress argument needs every wait
of an item to be on a lower ticket; the tests check that for the order the
library uses, then run the order under random progress with the kernel's own
flag and counter conditions and check that no item ever waits forever and no
condition is met before the work it stands for is done.
"""
import random

import pytest
import torch

from paper_2012_11346_gb300 import slim

TILE, R1, R2 = 0, 2, 3
T = 128

# (B, H, L, C): full slices, a ragged last slice with fewer tiles, one-tile
# slices, many chains, a single slice (C > L)
SHAPES = [(8, 8, 4096, 1024), (2, 2, 1000, 320), (2, 3, 700, 64), (1, 1, 8192, 1024),
          (16, 16, 256, 128), (1, 2, 130, 4096), (3, 1, 5000, 640)]


def schedule(B, H, L, C, M=256):
    return slim.bwd_schedule(B, H, L, 64, M, C, torch.bfloat16, "exp")[0]


def ring(B, H, L, C, M=256):
    return slim.bwd_schedule(B, H, L, 64, M, C, torch.bfloat16, "exp")[1]


def geometry(B, H, L, C):
    cs = min(C, L)
    N = (L + cs - 1) // cs
    ntn = [(min(cs, L - n * cs) + T - 1) // T for n in range(N)]
    return B * H, N, ntn


def tile_item(ntn, ch, n, t, c):
    # last tile first, chains inside a tile position
    return (ntn[n] - 1 - t) * ch + c


def dependencies(B, H, L, C, items):
    """For every ticket, the tickets of the items its waits stand for.  A tile
    item runs the tile's dq part and then its dk/dv part."""
    ch, N, ntn = geometry(B, H, L, C)
    R = ring(B, H, L, C)
    ticket = {it: x for x, it in enumerate(items)}
    r1n = sum(1 for it in items if it[0] == R1)
    deps = []
    for kind, n, idx in items:
        d = []
        if kind == TILE:
            c, t = idx % ch, ntn[n] - 1 - idx // ch
            if t + 1 < ntn[n]:  # rollback and state-gradient chains
                d.append(ticket[(TILE, n, tile_item(ntn, ch, n, t + 1, c))])
            elif n + 1 < N:
                d.append(ticket[(TILE, n + 1, tile_item(ntn, ch, n + 1, 0, c))])
            if n + R < N and t < ntn[n + R]:  # hand-off ring slot n % R
                d.append(ticket[(TILE, n + R, tile_item(ntn, ch, n + R, t, c))])
            if n + 1 < N and t < ntn[n + 1]:  # the dOmega sum at this position
                d.append(ticket[(TILE, n + 1, tile_item(ntn, ch, n + 1, t, c))])
        elif kind == R1:
            d += [ticket[(TILE, 0, i)] for i in range(ch * ntn[0])]
        else:
            d += [ticket[(R1, 0, r)] for r in range(r1n)]
        deps.append(d)
    return deps


@pytest.mark.parametrize("shape", SHAPES)
def test_every_item_once(shape):
    B, H, L, C = shape
    ch, N, ntn = geometry(B, H, L, C)
    items = schedule(B, H, L, C)
    assert len(set(items)) == len(items)
    for n in range(N):
        got = sorted(i for k, s, i in items if k == TILE and s == n)
        assert got == list(range(ch * ntn[n])), n
    r1 = sorted(i for k, s, i in items if k == R1)
    r2 = sorted(i for k, s, i in items if k == R2)
    assert r1 == list(range(len(r1))) and r2 == list(range(len(r2)))
    assert 4 <= len(r1) <= 128 and len(r1) % 4 == 0 and 4 <= len(r2) <= 32
    assert {s for k, s, _ in items if k in (R1, R2)} == {0}
    assert items[-len(r1) - len(r2):] == [(R1, 0, i) for i in range(len(r1))] + \
        [(R2, 0, i) for i in range(len(r2))]


@pytest.mark.parametrize("shape", SHAPES)
def test_waits_are_on_lower_tickets(shape):
    items = schedule(*shape)
    for x, d in enumerate(dependencies(*shape, items)):
        assert all(y < x for y in d), (x, items[x])


@pytest.mark.parametrize("shape", SHAPES)
def test_ring_keeps_the_reuse_wait_far_back(shape):
    # slice n-R's tile waits on slice n's tile at its position to have read the
    # hand-off: at least 320 tickets apart (about two waves of tile CTAs), R in
    # [2, 16]
    B, H, L, C = shape
    ch, N, ntn = geometry(B, H, L, C)
    R = ring(B, H, L, C)
    assert 2 <= R <= 16
    stage = ch * ntn[0]
    assert (R - 1) * stage >= 320 or R == 16
    assert R == 2 or (R - 2) * stage < 320


def test_stage_order():
    # stage j: the tiles of slice N-1-j, last tile first, chains inside a tile
    # position
    B, H, L, C = 8, 8, 4096, 1024
    ch, N, ntn = geometry(B, H, L, C)
    items = schedule(B, H, L, C)
    off = 0
    for j in range(N):
        n = N - 1 - j
        assert items[off:off + ch * ntn[n]] == [(TILE, n, i) for i in range(ch * ntn[n])]
        off += ch * ntn[n]


def progress(shape, resident, seed):
    """Runs the order with `resident` CTAs: a CTA takes the next ticket when it
    starts and can run its item only once the kernel's conditions hold."""
    B, H, L, C = shape
    ch, N, ntn = geometry(B, H, L, C)
    nt = ntn[0]
    items = schedule(B, H, L, C)
    deps = dependencies(B, H, L, C, items)
    R = ring(B, H, L, C)
    r1n = sum(1 for it in items if it[0] == R1)
    flag1, flag2, accflag = {}, {}, {}
    kvread = [{} for _ in range(R)]
    sums_done = r1done = 0
    done = [False] * len(items)

    def ready(x):
        kind, n, idx = items[x]
        if kind == TILE:
            c, t = idx % ch, ntn[n] - 1 - idx // ch
            ok = True
            inner = t + 1 < ntn[n]
            if inner or n + 1 < N:
                snext, want = (t + 1, n + 1) if inner else (0, n + 2)
                ok &= flag1.get((c, snext), 0) == want and flag2.get((c, snext), 0) == want
            if n + R < N and t < ntn[n + R]:
                ok &= kvread[n % R].get((c, t), 0) == n + R + 1
            if n + 1 < N and t < ntn[n + 1]:
                ok &= accflag.get((c, t), 0) == n + 2
            return ok
        if kind == R1:
            return sums_done >= ch * nt
        return r1done >= r1n

    rng = random.Random(seed)
    nxt, running = 0, []
    while not all(done):
        while len(running) < resident and nxt < len(items):
            running.append(nxt)
            nxt += 1
        can = [x for x in running if ready(x)]
        assert can, f"no resident item can run (next ticket {nxt})"
        x = rng.choice(can)
        assert all(done[y] for y in deps[x]), f"ticket {x} {items[x]} ran early"
        kind, n, idx = items[x]
        if kind == TILE:
            c, t = idx % ch, ntn[n] - 1 - idx // ch
            flag1[(c, t)] = flag2[(c, t)] = n + 1
            kvread[n % R][(c, t)] = n + 1
            accflag[(c, t)] = n + 1
            sums_done += n == 0
        elif kind == R1:
            r1done += 1
        done[x] = True
        running.remove(x)


@pytest.mark.parametrize("shape", SHAPES[1:5])
@pytest.mark.parametrize("resident", [1, 7, 152])
def test_random_progress(shape, resident):
    progress(shape, resident, seed=resident)
