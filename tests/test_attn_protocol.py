"""A model of the barrier protocol of attn_pv_tac_kernel (csrc/attn.cu),
run under random interleavings of its three roles, for many key-chunk
counts and items per CTA.

The kernel's TMA warp, MMA warp and softmax warps communicate only through
mbarriers whose waits name a phase parity. This model replays each role's
sequence of waits and arrivals in the kernel's order, with the kernel's
entry numbering (ring entries of an item: Q, nk pass-1 K chunks, nk pass-2
K / V pairs, M's two halves, the output slot; six ring slots; two S
buffers), and checks under random schedules that

- no schedule deadlocks;
- every wait sees exactly the completed-phase count it means (a parity
  wait that could be satisfied by a phase two ahead would be a bug);
- a ring slot is refilled only after its consumer released it, and an S
  buffer takes new scores only after the softmax warps have finished with
  its previous use (read it in pass 1, written P over it in pass 2).

The softmax warps are one role here: all sixteen run the same program and
a barrier completes when the last of them arrives. MMAs complete in issue
order, so a commit is modelled at the issuing point."""

import random

import pytest

SLOTS = 6


class Bar:
    def __init__(self):
        self.phases = 0          # completed phases

    def arrive(self):
        self.phases += 1


def run(nk, items_per_cta, seed, prefer=None, drop_p_wait=False, drop_s_wait=False):
    """One schedule: each step runs the first role of `prefer` (a priority
    order) whose next step can proceed, else a random one among those that
    can. A priority order starves the roles at its end, where a missing
    wait shows at once."""
    my = items_per_cta
    E = 3 * nk + 4                                   # ring entries per item
    u0, u1 = (nk + 1) // 2, nk // 2                  # uses of S buffer 0 / 1 per pass

    def sbuf(i, it):                                 # S buffer and its use number
        j = it if it < nk else it - nk
        b = j & 1
        per = u0 if b == 0 else u1
        return b, (j >> 1) + (0 if it < nk else per) + i * 2 * per

    bars = {}

    def bar(name):
        return bars.setdefault(name, Bar())

    full = lambda g: ("full", g % SLOTS)
    empty = lambda g: ("empty", g % SLOTS)
    # a wait for phase number `want - 1` to have completed
    W = lambda name, want: ("wait", name, want)
    A = lambda name: ("arrive", name)
    filled, consumed = {}, {}                       # ring: per-slot use counts
    s_written, s_done = [0, 0], [0, 0]               # S buffers: uses written / finished

    def tma():
        for i in range(my):
            for u in range(E):
                g = i * E + u
                yield W(empty(g), g // SLOTS)        # the slot's previous use released
                assert consumed.get(g % SLOTS, 0) == g // SLOTS, "ring slot refilled before release"
                filled[g % SLOTS] = g // SLOTS + 1
                yield A(full(g))
        G = my * E
        for g in range(max(G - SLOTS, 0), G):        # every slot given back before exit
            yield W(empty(g), g // SLOTS + 1)

    def release(g):
        consumed[g % SLOTS] = consumed.get(g % SLOTS, 0) + 1
        return A(empty(g))

    def mma():
        for i in range(my):
            gq, g0 = i * E, i * E + 1
            yield W("q_full", i + 1)                 # Q in TMEM: its ring slot is free again
            yield release(gq)

            def qk(it):
                g = g0 + (it if it < nk else nk + 2 * (it - nk))
                b, n = sbuf(i, it)
                yield W(full(g), g // SLOTS + 1)
                if not drop_s_wait:
                    yield W(("s_empty", b), n)       # previous use of the buffer consumed
                assert s_done[b] == n, "S buffer overwritten before its previous use was consumed"
                s_written[b] += 1
                yield release(g)
                yield A(("s_full", b))
            for it in range(min(nk + 2, 2 * nk)):    # pass 1, then two chunks ahead
                yield from qk(it)
            for j in range(nk):                      # one wait per pass-2 chunk
                gv, gk = g0 + nk + 2 * j + 1, g0 + nk + 2 * j + 4
                more = j + 2 < nk
                b, n = sbuf(i, nk + j)
                if not drop_p_wait:
                    yield W(("s_empty", b), n + 1)   # P(j) written over S(j)
                yield W(full(gv), gv // SLOTS + 1)
                if more:
                    yield W(full(gk), gk // SLOTS + 1)
                yield release(gv)                    # P V^T(j)
                if more:                             # Q K^T(j + 2) into the same buffer
                    b2, n2 = sbuf(i, nk + j + 2)
                    assert (b2, n2) == (b, n + 1)
                    assert s_done[b] == n + 1, "S buffer overwritten before P(j) was written over it"
                    s_written[b] += 1
                    yield release(gk)
                    yield A(("s_full", b))
            yield A("pv_done")
            gm = g0 + 3 * nk
            yield W("z_full", i + 1)
            yield W(full(gm), gm // SLOTS + 1)
            yield W(full(gm + 1), (gm + 1) // SLOTS + 1)
            yield release(gm)
            yield release(gm + 1)
            yield A("tac_done")
        if my:
            yield W("tac_done", my)                  # every MMA done before TMEM is freed

    def softmax():
        def put_q(i):
            gq = i * E
            yield W(full(gq), gq // SLOTS + 1)
            yield A("q_full")
        if my:
            yield from put_q(0)
        for i in range(my):
            g0 = i * E + 1
            for it in range(nk):                     # pass 1: read S, arrive
                b, n = sbuf(i, it)
                yield W(("s_full", b), n + 1)
                assert s_written[b] == n + 1
                s_done[b] += 1
                yield A(("s_empty", b))
            for j in range(nk):                      # pass 2: read S, write P over it, arrive
                b, n = sbuf(i, nk + j)
                yield W(("s_full", b), n + 1)
                s_done[b] += 1
                yield A(("s_empty", b))
            yield W("pv_done", i + 1)
            if i + 1 < my:
                yield from put_q(i + 1)
            yield A("z_full")
            go = g0 + 3 * nk + 2                     # the output boxes' slot
            yield W("tac_done", i + 1)
            yield W(full(go), go // SLOTS + 1)
            yield release(go)

    rng = random.Random(seed)
    roles = {"tma": tma(), "mma": mma(), "softmax": softmax()}
    cur = {k: next(v, None) for k, v in roles.items()}

    def ready(step):
        return step[0] == "arrive" or bar(step[1]).phases >= step[2]

    while any(c is not None for c in cur.values()):
        live = [k for k, c in cur.items() if c is not None and ready(c)]
        assert live, f"deadlock at {cur}"
        k = next((r for r in prefer or () if r in live), None) or rng.choice(live)
        step = cur[k]
        if step[0] == "arrive":
            bar(step[1]).arrive()
        else:
            # a parity wait is sound only if the barrier is not two phases on
            assert bar(step[1]).phases in (step[2], step[2] + 1) or step[2] == 0, \
                f"{k} waits for phase {step[2] - 1} of {step[1]}, which has completed {bar(step[1]).phases}"
        cur[k] = next(roles[k], None)


@pytest.mark.parametrize("nk", [1, 2, 3, 4, 5, 7, 8, 16, 64])
@pytest.mark.parametrize("items", [1, 2, 3])
def test_attention_barrier_protocol(nk, items):
    orders = (None, ("tma", "mma"), ("mma", "tma"), ("softmax",), ("softmax", "mma"), ("mma", "softmax"))
    for prefer in orders:
        for seed in range(6 if nk < 64 else 2):
            run(nk, items, seed, prefer)


def test_model_catches_a_missing_wait():
    """The model is not vacuous: without the MMA warp's wait for P(j)
    (P V^T(j) and Q K^T(j + 2) issued before the softmax warps have written
    P over S(j)), a schedule that runs the MMA warp ahead trips the
    S-buffer check, for every chunk count that has a pass-2 Q K^T."""
    for nk in (3, 4, 8):
        with pytest.raises(AssertionError, match="S buffer"):
            run(nk, 1, 0, prefer=("mma", "tma"), drop_p_wait=True)
        run(nk, 1, 0, prefer=("mma", "tma"))


def test_model_catches_a_missing_s_wait():
    """Without Q K^T's wait for its S buffer (scores written into a buffer
    whose previous scores the softmax warps have not read yet), the same
    schedule trips the check, from two key chunks on."""
    for nk in (2, 3, 8):
        with pytest.raises(AssertionError, match="previous use was consumed"):
            run(nk, 2, 0, prefer=("mma", "tma"), drop_s_wait=True)
