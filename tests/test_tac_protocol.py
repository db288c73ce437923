"""A model of the barrier protocol of the streaming tensor-core TAC kernel
(tac_stream_kernel, csrc/tac.cu) under random and starving interleavings
of its three roles.

A CTA takes a contiguous run of (block, token tile) jobs, at most two
blocks per run. The TMA warp loads M_b's halves once per block (for the
second block only after the MMA warp's commit on `mempty`: the first
block's MMAs are done with M) and the Z tiles through a ring of ZS stages
(`zfull` / `zempty`); the MMA warp multiplies each tile into one of two
TMEM accumulators (`accfull` / `accempty`); the epilogue warps read an
accumulator, free it and store. The model replays the kernel's waits and
parities and checks, for many job counts, block splits and ring depths:

- no schedule deadlocks;
- every wait sees the completed-phase count it means;
- the MMAs of a job read the Z stage holding that job and the M of its
  block; a Z stage or M is reloaded only after the MMAs that read it
  completed; an accumulator is written only after it was drained, and the
  epilogue reads the job that was written into it.
"""

import random

import pytest


def run(blocks, zs, seed, prefer=None, drop=None):
    """blocks: the block of each job of the CTA (non-decreasing). `drop`
    removes one wait ("mempty", "zempty" or "accempty")."""
    n = len(blocks)
    phases = {}
    W = lambda name, want: ("wait", name, want)      # completed phases >= want
    A = lambda name: ("arrive", name)
    state = {"M": None, "mma_jobs": 0}
    zstage = {}                                      # stage -> job it holds
    zread = {}                                       # stage -> uses read by MMAs
    acc_job, acc_drained = [None, None], [True, True]

    def tma():
        mb, mloads = None, 0
        for i in range(n):
            b = blocks[i]
            if b != mb:
                if mloads > 0 and drop != "mempty":
                    yield W("mempty", mloads)        # parity (mloads - 1) & 1
                first = blocks.index(mb) if mb is not None else 0
                done_old = state["mma_jobs"] >= first + blocks.count(mb) if mb is not None else True
                assert done_old, "M reloaded while MMAs of the previous block may still read it"
                state["M"] = b
                yield A("mfull")
                mb, mloads = b, mloads + 1
            k = i % zs
            if drop != "zempty":
                yield W(("zempty", k), i // zs)       # parity ((i / zs) & 1) ^ 1
            assert zread.get(k, 0) == i // zs, "Z stage refilled before its MMAs completed"
            zstage[k] = i
            yield A(("zfull", k))
        for i in range(max(n - zs, 0), n):
            yield W(("zempty", i % zs), i // zs + 1)

    def mma():
        mb, mloads = None, 0
        for i in range(n):
            b = blocks[i]
            if b != mb:
                if mloads > 0:
                    yield A("mempty")                # commit: the previous block's MMAs are done
                yield W("mfull", mloads + 1)         # parity mloads & 1
                mb, mloads = b, mloads + 1
            k, acc = i % zs, i & 1
            yield W(("zfull", k), i // zs + 1)       # parity (i / zs) & 1
            if drop != "accempty":
                yield W(("accempty", acc), i >> 1)   # parity ((i >> 1) & 1) ^ 1
            assert zstage.get(k) == i and state["M"] == b, "MMA operands are not this job's"
            assert acc_drained[acc], "accumulator overwritten before it was drained"
            acc_job[acc], acc_drained[acc] = i, False
            zread[k] = zread.get(k, 0) + 1
            state["mma_jobs"] = i + 1
            yield A(("zempty", k))
            yield A(("accfull", acc))
        if n:
            yield W(("accfull", (n - 1) & 1), ((n - 1) >> 1) + 1)

    def epilogue():
        for i in range(n):
            acc = i & 1
            yield W(("accfull", acc), (i >> 1) + 1)   # parity (i >> 1) & 1
            assert acc_job[acc] == i and not acc_drained[acc], "epilogue read another job's accumulator"
            acc_drained[acc] = True
            yield A(("accempty", acc))

    rng = random.Random(seed)
    roles = {"tma": tma(), "mma": mma(), "epi": epilogue()}
    cur = {k: next(v, None) for k, v in roles.items()}

    def ready(step):
        return step[0] == "arrive" or phases.get(step[1], 0) >= step[2]

    while any(c is not None for c in cur.values()):
        live = [k for k, c in cur.items() if c is not None and ready(c)]
        assert live, f"deadlock at {cur}"
        k = next((r for r in prefer or () if r in live), None) or rng.choice(live)
        step = cur[k]
        if step[0] == "arrive":
            phases[step[1]] = phases.get(step[1], 0) + 1
        else:
            assert phases.get(step[1], 0) in (step[2], step[2] + 1), \
                f"{k} waits for {step[2]} phases of {step[1]}, which has {phases.get(step[1], 0)}"
        cur[k] = next(roles[k], None)
    assert all(acc_drained)


ORDERS = (None, ("tma", "mma"), ("mma", "tma"), ("epi",), ("tma", "epi"), ("mma", "epi"))
SPLITS = [[0], [0, 0, 0], [0] * 8, [0, 1], [0] * 5 + [1] * 3, [0] + [1] * 6, [3] * 4 + [4] * 4]


@pytest.mark.parametrize("blocks", SPLITS, ids=lambda b: "-".join(map(str, b)))
@pytest.mark.parametrize("zs", [2, 3])
def test_tac_stream_barrier_protocol(blocks, zs):
    for prefer in ORDERS:
        for seed in range(4):
            run(blocks, zs, seed, prefer)


@pytest.mark.parametrize("wait,prefer,what", [("mempty", ("tma", "mma"), "M reloaded"),
                                              ("zempty", ("tma", "mma"), "Z stage refilled"),
                                              ("accempty", ("mma", "tma"), "accumulator overwritten")])
def test_model_catches_a_missing_wait(wait, prefer, what):
    """Each of the producer-side waits, taken out, lets a schedule that runs
    the producer ahead trip the matching hazard check."""
    blocks = [0] * 5 + [1] * 5
    with pytest.raises(AssertionError, match=what):
        run(blocks, 2, 0, prefer, drop=wait)
    run(blocks, 2, 0, prefer)
