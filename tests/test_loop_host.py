"""Host-side checks of the double-buffered decode loop's schedule (no GPU).

The schedule is replayed on a model of two CUDA streams and their events: an operation on a
stream happens after every earlier operation on that stream and after everything an event it
waited for had seen when it was recorded. Checked for every block: it runs on the buffer set
that holds its own pool block, that set's last refill happens before it, and no refill of a
set starts before the block that last read that set has finished.
"""
import pytest

from paper_2609_33390_gb300 import loop, synth

COPY, RUN = "copy", "run"
STREAM_OF = {"copy_wait": COPY, "copy": COPY, "copy_ready": COPY,
             "run_wait": RUN, "launch": RUN, "run_done": RUN}


def check_schedule(ops, blocks, pool_len):
    known = {COPY: set(), RUN: set()}          # ops known to have happened, per stream
    ready, done = {}, {}                        # event -> ops seen when it was recorded
    content = {0: 0, 1: 1 % pool_len}           # pool block held by each input set
    last_copy = {0: None, 1: None}              # op index of the latest refill of each set
    last_launch = {0: None, 1: None}
    launched = []
    for n, op in enumerate(ops):
        kind, s = op[0], op[1]
        st = STREAM_OF[kind]
        if kind == "copy_wait":
            known[COPY] |= done.get(s, set())
        elif kind == "run_wait":
            known[RUN] |= ready.get(s, set())
        elif kind == "copy_ready":
            ready[s] = set(known[COPY])
        elif kind == "run_done":
            done[s] = set(known[RUN])
        elif kind == "copy":
            prev = last_launch[s]
            assert prev is None or prev in known[COPY], f"op {n}: refill of set {s} may overlap the block reading it"
            content[s] = op[2]
            last_copy[s] = n
        elif kind == "launch":
            t = op[2]
            assert s == t % 2, f"block {t} on set {s}"
            assert content[s] == t % pool_len, f"block {t} would read pool block {content[s]}"
            lc = last_copy[s]
            assert lc is None or lc in known[RUN], f"block {t} may start before its inputs are written"
            last_launch[s] = n
            launched.append(t)
        known[st].add(n)
    assert launched == list(range(blocks))


@pytest.mark.parametrize("blocks", [1, 2, 5, 8])
@pytest.mark.parametrize("pool_len", [1, 2, 3, 4])
def test_schedule_orders_every_refill_and_block(blocks, pool_len):
    check_schedule(loop.double_buffer_schedule(blocks, pool_len), blocks, pool_len)


def test_checker_catches_a_missing_wait():
    """A schedule without the refill's wait on the block that read the set, and one without the
    block's wait on its refill, both fail the check."""
    ops = loop.double_buffer_schedule(5, 3)
    with pytest.raises(AssertionError, match="overlap"):
        check_schedule([o for o in ops if o[0] != "copy_wait"], 5, 3)
    with pytest.raises(AssertionError, match="inputs are written"):
        check_schedule([o for o in ops if o[0] != "run_wait"], 5, 3)


def test_refilled_inputs_are_the_block_inputs_except_the_anchor():
    wl = synth.Workload("loophost", B=1, L=4, V=64, d=16, K=4, r=16)
    blk = synth.make_block(wl, "cpu")
    assert set(loop.BLOCK_INPUTS) == set(blk) - {"x0"}
