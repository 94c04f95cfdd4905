"""Host-side checks of the double-buffered decode loop (no GPU): it refills exactly the inputs a
block carries besides the chained anchor."""
from paper_2609_33390_gb300 import loop, synth


def test_refilled_inputs_are_the_block_inputs_except_the_anchor():
    wl = synth.Workload("loophost", B=1, L=4, V=64, d=16, K=4, r=16)
    blk = synth.make_block(wl, "cpu")
    assert set(loop.BLOCK_INPUTS) == set(blk) - {"x0"}
    assert callable(loop.graph_loop_double_buffered)
