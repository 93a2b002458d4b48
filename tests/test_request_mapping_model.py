"""CPU model of the chunk-digest warps' chunk-to-request mapping
(csrc/pk_device.cuh: lane_request_guess, lane_request_window).

A warp's 32 consecutive chunks g0 .. g0+31 need each lane's request r with
key_off[r] <= g < key_off[r+1].  The device guesses r from the mean request
size, loads 32 offsets from 8 requests before the guess and resolves every lane
with a 6-step search by shuffles; when that window does not bracket every lane
it falls back to a search for the first chunk's request, a 32-wide window from
there (the same 6-step search) and a per-lane search past it.  The model follows
those steps (float guess included) and must give, for every lane, exactly the
request np.searchsorted gives, on layouts that reach all three paths."""
import numpy as np
import pytest


def ref(ko, g):
    return int(np.searchsorted(ko, g, side="right") - 1)


def search32(vals, lo, hi, gg):
    """The device's 6 halvings over [lo, hi] with the shuffle source clamped to lane 31."""
    for _ in range(6):
        mid = (lo + hi) >> 1
        vm = vals[min(mid, 31)]
        if lo < hi:
            if vm <= gg:
                lo = mid + 1
            else:
                hi = mid
    return lo


def window_path(ko, R, g0, total, lane):
    r0 = ref(ko, g0)  # warp_find_request: exact
    big = np.iinfo(np.int64).max
    v = [int(ko[r0 + 1 + j]) if r0 + 1 + j <= R else big for j in range(32)]
    gg = min(g0 + lane, total - 1)
    lo = search32(v, 0, 32, gg)
    return (r0 + lo, "window") if lo < 32 else (ref(ko, gg), "past window")


def guess_path(ko, R, g0, total):
    """Per-lane (request, path) for the warp of chunks g0 .. g0+31."""
    rg = int(np.float32(g0) / np.float32(total) * np.float32(R))
    rg = R - 1 if rg >= R else rg
    w0 = rg - 8 if rg > 8 else 0
    big = np.iinfo(np.int64).max
    u = [int(ko[w0 + j]) if w0 + j <= R else big for j in range(32)]
    res, ok = [], []
    for lane in range(32):
        gg = min(g0 + lane, total - 1)
        lo = search32(u, 1, 32, gg)
        ok.append(u[0] <= g0 and lo < 32)
        res.append(w0 + lo - 1)
    if all(ok):
        return [(r, "guess") for r in res]
    return [window_path(ko, R, g0, total, lane) for lane in range(32)]


def layouts():
    rng = np.random.default_rng(7)
    yield "equal", np.full(3000, 128)
    yield "equal, few", np.full(5, 40)
    yield "one request", np.array([1000])
    n = rng.integers(0, 9, 4000)
    n[rng.integers(0, 4000, 1500)] = 0
    yield "ragged with empties", n
    n = rng.integers(0, 3, 3000)
    n[rng.integers(0, 3000, 12)] = rng.integers(200, 400, 12)
    yield "skewed", n
    n = np.zeros(6000, np.int64)
    i = 0
    while i < n.size:
        n[i] = rng.integers(1, 6)
        i += 1 + (int(rng.integers(40, 200)) if rng.random() < 0.3 else 0)
    yield "runs of empty requests", n
    n = np.zeros(300, np.int64)
    n[-1] = 50
    yield "empties then one", n


@pytest.mark.parametrize("name,n", list(layouts()), ids=[name for name, _ in layouts()])
def test_every_lane_maps_to_its_request(name, n):
    n = np.asarray(n, np.int64)
    R = n.size
    ko = np.zeros(R + 1, np.int64)
    np.cumsum(n, out=ko[1:])
    total = int(ko[-1])
    paths = set()
    for g0 in range(0, total, 32):
        for lane, (r, path) in enumerate(guess_path(ko, R, g0, total)):
            paths.add(path)
            g = g0 + lane
            if g < total:
                assert r == ref(ko, g), (name, g0, lane, path)
                assert ko[r] <= g < ko[r + 1]
    assert paths, name


def test_all_three_paths_are_reached():
    reached = set()
    for name, n in layouts():
        n = np.asarray(n, np.int64)
        ko = np.zeros(n.size + 1, np.int64)
        np.cumsum(n, out=ko[1:])
        for g0 in range(0, int(ko[-1]), 32):
            reached |= {p for _, p in guess_path(ko, n.size, g0, int(ko[-1]))}
    assert reached == {"guess", "window", "past window"}
