"""A model of the barrier protocol of the TMA pair GEMM
(w4a4_gemm_tma_pair_kernel, csrc/w4a4_gemm.cu) under random and starving
interleavings of its three roles.

The TMA warp fills a ring of STAGES operand stages (`full` / `empty`
barriers); the MMA warp consumes them into two TMEM accumulators, one
accumulator per run of K blocks (a whole tile for the 4-bit kind, KRUN K
blocks for the 8-bit kind), committing `tmem_full` at the end of each run;
the epilogue warps drain each run and hand the accumulator back through
`tmem_empty`. Every wait names a phase parity, and the model replays the
kernel's parities: the MMA waits for parity ((use & 1) ^ 1) on
`tmem_empty` and the epilogue for parity (use & 1) on `tmem_full`, where
use = run counter >> 1. The checks, for many shapes:

- no schedule deadlocks;
- every wait sees the completed-phase count it means (a parity wait that a
  phase two ahead would also satisfy is a bug);
- a stage is refilled only after the MMAs that read it completed, an
  accumulator is written only after its previous run was drained, and the
  epilogue drains exactly the run the MMA warp wrote, in order.
"""

import random

import pytest


class Bar:
    def __init__(self):
        self.phases = 0


def run(num_k, krun, tiles, stages, seed, prefer=None, drop=None):
    """One schedule. krun = 0: one run per tile. `drop` removes one wait
    ("tmem_empty" or "stage_empty") to show that the checks catch it."""
    runs_per_tile = 1 if krun == 0 else (num_k + krun - 1) // krun
    bars = {}

    def bar(name):
        return bars.setdefault(name, Bar())

    W = lambda name, want: ("wait", name, want)     # completed phases >= want
    A = lambda name: ("arrive", name)
    filled, consumed = {}, {}                       # per stage: uses filled / consumed
    written, drained = [[], []], [0, 0]             # per accumulator: runs written, runs drained

    def tma():
        g = 0
        for _ in range(tiles):
            for _ in range(num_k):
                s, u = g % stages, g // stages
                if drop != "stage_empty":
                    yield W(("empty", s), u)        # parity (u & 1) ^ 1
                assert consumed.get(s, 0) == u, "stage refilled before its MMAs completed"
                filled[s] = u + 1
                yield A(("full", s))
                g += 1

    def mma():
        g, it = 0, 0
        for _ in range(tiles):
            for kc in range(num_k):
                kk = kc % krun if krun else kc
                acc = it & 1
                if kk == 0:
                    if drop != "tmem_empty":
                        yield W(("tmem_empty", acc), it >> 1)     # parity ((it >> 1) & 1) ^ 1
                    assert drained[acc] == len(written[acc]), "accumulator overwritten before it was drained"
                    written[acc].append(it)
                s, u = g % stages, g // stages
                yield W(("full", s), u + 1)         # parity u & 1
                assert filled.get(s, 0) == u + 1
                consumed[s] = consumed.get(s, 0) + 1
                yield A(("empty", s))               # the MMAs' commit (they complete in order)
                g += 1
                if kc + 1 == num_k or (krun and kk + 1 == krun):
                    yield A(("tmem_full", acc))
                    it += 1

    def epilogue():
        it = 0
        for _ in range(tiles):
            for _ in range(runs_per_tile):
                acc = it & 1
                yield W(("tmem_full", acc), (it >> 1) + 1)       # parity (it >> 1) & 1
                assert written[acc][drained[acc]] == it, "drained a run other than the one written"
                drained[acc] += 1
                yield A(("tmem_empty", acc))
                it += 1

    rng = random.Random(seed)
    roles = {"tma": tma(), "mma": mma(), "epi": epilogue()}
    cur = {k: next(v, None) for k, v in roles.items()}

    def ready(step):
        return step[0] == "arrive" or bar(step[1]).phases >= step[2]

    while any(c is not None for c in cur.values()):
        live = [k for k, c in cur.items() if c is not None and ready(c)]
        assert live, f"deadlock at {cur}"
        k = next((r for r in prefer or () if r in live), None) or rng.choice(live)
        step = cur[k]
        if step[0] == "arrive":
            bar(step[1]).phases += 1
        else:
            assert bar(step[1]).phases in (step[2], step[2] + 1), \
                f"{k} waits for {step[2]} phases of {step[1]}, which has {bar(step[1]).phases}"
        cur[k] = next(roles[k], None)
    assert drained == [len(written[0]), len(written[1])]
    assert sum(drained) == tiles * runs_per_tile


ORDERS = (None, ("mma", "tma"), ("tma", "mma"), ("epi",), ("mma", "epi"), ("epi", "tma"))


@pytest.mark.parametrize("num_k,krun", [(1, 0), (2, 0), (32, 0), (2, 8), (8, 8), (9, 8), (64, 8), (18, 8),
                                        (5, 1), (7, 2)])
@pytest.mark.parametrize("tiles", [1, 2, 3, 5])
def test_gemm_barrier_protocol(num_k, krun, tiles):
    for stages in (4, 6):
        for prefer in ORDERS:
            for seed in range(3):
                run(num_k, krun, tiles, stages, seed, prefer)


@pytest.mark.parametrize("wait", ["tmem_empty", "stage_empty"])
def test_model_catches_a_missing_wait(wait):
    """Without the MMA warp's wait for a drained accumulator, or the TMA
    warp's wait for a consumed stage, a schedule that runs the producer
    ahead trips the matching hazard check."""
    prefer = ("mma", "tma") if wait == "tmem_empty" else ("tma", "mma")
    what = "accumulator overwritten" if wait == "tmem_empty" else "stage refilled"
    with pytest.raises(AssertionError, match=what):
        run(24, 8, 3, 4, 0, prefer, drop=wait)
    run(24, 8, 3, 4, 0, prefer)
