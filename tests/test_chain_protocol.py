"""CPU model of the chain kernel's two-warp protocol (csrc/pk_derive.cu, k_chain).

Each layout's rounds warp (R) and schedule warp (S) are written out as their
sequences of named-barrier operations and shared-memory accesses, step by step
as the kernel issues them; every interleaving of the two warps is explored and
must end with both warps done (no deadlock), no warp arriving twice in one
phase of a barrier (count 64: one arrival per warp completes a phase), no
pending arrival left at the end, and no read of a buffer overlapping the other
warp's write of it.  A mutated protocol must fail the same checks, so that the
model is shown to catch what it is meant to catch."""
import pytest

# ops: ("arrive", id) | ("sync", id) | ("w+", buf) | ("w-", buf) | ("r+", buf) | ("r-", buf)


def one_pair(n):
    """One pair per CTA: barriers 1-3 block-1 slices, 4 block 2 ready, 5 k published."""
    S = [("w+", "kw2_0"), ("w-", "kw2_0"), ("arrive", 4)]
    for i in range(n):
        if i > 0:
            S += [("sync", 5), ("r+", "kpub"), ("r-", "kpub"), ("arrive", 4)]
        slices = 6 if i + 1 < n else 3
        for sl in range(1, slices + 1):
            buf = f"kw1_{sl}" if sl <= 3 else f"kw2_{(i + 1) & 1}"
            S += [("w+", buf), ("w-", buf)]
            if sl <= 3:
                S += [("arrive", sl)]
    R = []
    for i in range(n):
        for sl in (1, 2, 3):
            R += [("sync", sl), ("r+", f"kw1_{sl}"), ("r-", f"kw1_{sl}")]
        R += [("sync", 4), ("r+", f"kw2_{i & 1}"), ("r-", f"kw2_{i & 1}")]
        if i + 1 < n:
            R += [("w+", "kpub"), ("w-", "kpub"), ("arrive", 5)]
    return R, S


def four_pairs(n):
    """Four pairs per CTA, one pair's barriers: s1 (block-1 slice 1, and block 2 of the step ready), s1b
    (block-1 slices 2-3), k (k published)."""
    S = [("w+", "kw2_0"), ("w-", "kw2_0")]
    for i in range(n):
        if i > 0:
            S += [("sync", "k"), ("r+", "kpub"), ("r-", "kpub")]
        S += [("w+", "kw1_1"), ("w-", "kw1_1"), ("arrive", "s1")]
        S += [("w+", "kw1_2"), ("w-", "kw1_2"), ("w+", "kw1_3"), ("w-", "kw1_3"), ("arrive", "s1b")]
        if i + 1 < n:
            b = f"kw2_{(i + 1) & 1}"
            S += [("w+", b), ("w-", b)]
    R = []
    for i in range(n):
        R += [("sync", "s1"), ("r+", "kw1_1"), ("r-", "kw1_1"), ("sync", "s1b"), ("r+", "kw1_2"), ("r-", "kw1_2"),
              ("r+", "kw1_3"), ("r-", "kw1_3"), ("r+", f"kw2_{i & 1}"), ("r-", f"kw2_{i & 1}")]
        if i + 1 < n:
            R += [("w+", "kpub"), ("w-", "kpub"), ("arrive", "k")]
    return R, S


class ProtocolError(Exception):
    pass


def explore(R, S):
    """Every interleaving of the two programs; raises ProtocolError on a violation.
    State: (pc of each warp, per barrier the set of warps arrived in its current phase and its phase
    number, the phase each warp waits for, the buffers each warp is accessing)."""
    progs = (R, S)
    seen = set()

    def key(st):
        pcs, bars, waits, acc = st
        return (pcs, tuple(sorted((b, tuple(sorted(a)), p) for b, (a, p) in bars.items())), waits,
                tuple(tuple(sorted(x)) for x in acc))

    def step(st, w):
        pcs, bars, waits, acc = st
        if waits[w] is not None:
            bid, phase = waits[w]
            if bars.get(bid, (frozenset(), 0))[1] <= phase:
                return None  # still blocked
            waits = tuple(None if j == w else waits[j] for j in range(2))
            return (pcs, bars, waits, acc)
        if pcs[w] == len(progs[w]):
            return None
        op, arg = progs[w][pcs[w]]
        bars = dict(bars)
        acc = [set(acc[0]), set(acc[1])]
        new_wait = waits[w]
        if op in ("arrive", "sync"):
            arrived, phase = bars.get(arg, (frozenset(), 0))
            if w in arrived:
                raise ProtocolError(f"warp {'RS'[w]} arrives twice in phase {phase} of barrier {arg}")
            arrived = arrived | {w}
            if len(arrived) == 2:
                bars[arg] = (frozenset(), phase + 1)
            else:
                bars[arg] = (arrived, phase)
                if op == "sync":
                    new_wait = (arg, phase)
        elif op == "w+":
            if arg in acc[1 - w]:
                raise ProtocolError(f"warp {'RS'[w]} writes {arg} while the other warp accesses it")
            acc[w].add(arg)
        elif op == "r+":
            if arg in acc[1 - w]:
                raise ProtocolError(f"warp {'RS'[w]} reads {arg} while the other warp writes it")
            acc[w].add(arg)
        else:  # w- / r-
            acc[w].discard(arg)
        pcs = tuple(pcs[j] + (1 if j == w else 0) for j in range(2))
        waits = tuple(new_wait if j == w else waits[j] for j in range(2))
        return (pcs, bars, waits, (frozenset(acc[0]), frozenset(acc[1])))

    start = ((0, 0), {}, (None, None), (frozenset(), frozenset()))
    stack = [start]
    finals = 0
    while stack:
        st = stack.pop()
        k = key(st)
        if k in seen:
            continue
        seen.add(k)
        nxt = [s for s in (step(st, 0), step(st, 1)) if s is not None]
        if not nxt:
            pcs, bars, waits, _ = st
            if pcs != (len(R), len(S)) or waits != (None, None):
                raise ProtocolError(f"deadlock at R pc {pcs[0]}/{len(R)}, S pc {pcs[1]}/{len(S)}, waits {waits}")
            pending = {b: a for b, (a, _) in bars.items() if a}
            if pending:
                raise ProtocolError(f"arrivals left pending at the end: {pending}")
            finals += 1
            continue
        stack.extend(nxt)
    return len(seen), finals


@pytest.mark.parametrize("layout", [one_pair, four_pairs])
@pytest.mark.parametrize("n", [1, 2, 3, 5])
def test_protocol_has_no_deadlock_double_arrival_or_race(layout, n):
    states, finals = explore(*layout(n))
    assert finals == 1 and states > len(layout(n)[0])


def _mutate(prog, i, new=None):
    p = list(prog)
    if new is None:
        del p[i]
    else:
        p[i] = new
    return p


def test_model_catches_a_missing_sync():
    """Without the rounds warp's wait for block-1 slice 2, its read can overlap the schedule warp's write."""
    R, S = four_pairs(3)
    i = R.index(("sync", "s1b"))
    with pytest.raises(ProtocolError):
        explore(_mutate(R, i), S)


def test_model_catches_a_double_arrival():
    """The schedule warp marking block 2 ready on its own barrier again before the rounds warp has synced
    the previous phase: a second arrival in one phase."""
    R, S = one_pair(3)
    j = S.index(("sync", 5))
    with pytest.raises(ProtocolError):
        explore(R, _mutate(S, j))


def test_model_catches_a_buffer_reused_too_early():
    """Block 2 single-buffered (always kw2_0): the schedule warp would overwrite the buffer the rounds warp
    is still reading."""
    R, S = four_pairs(3)
    S = [(op, "kw2_0" if isinstance(a, str) and a.startswith("kw2_") else a) for op, a in S]
    R = [(op, "kw2_0" if isinstance(a, str) and a.startswith("kw2_") else a) for op, a in R]
    with pytest.raises(ProtocolError):
        explore(R, S)


def test_model_catches_a_deadlock():
    """The schedule warp waiting for k before it has marked the step's first slice (i = 0 included)."""
    R, S = four_pairs(2)
    S = [("sync", "k")] + S
    with pytest.raises(ProtocolError):
        explore(R, S)
