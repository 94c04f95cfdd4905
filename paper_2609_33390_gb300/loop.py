"""Host-side decode loop over captured decode tails (App. F: fused head plus CUDA Graph
replay), with the next block's inputs written while the current block runs. Only streams,
events and graph launches: every step of the tail runs in the library's kernels."""
from __future__ import annotations

BLOCK_INPUTS = ("logits_q", "logits_p", "hidden", "h_c", "u_sel", "u_acc", "u_res")


def graph_loop_double_buffered(tail, pool, sm, vm, stream, blocks, keep=False):
    """Block after block through two captured decode tails (App. F), one per input buffer set,
    the anchor chained on the device through one buffer both graphs share. While block t runs
    on `stream`, a second stream copies block t+1's inputs from `pool` (pre-generated blocks,
    taken in turn) into the other buffer set: the stand-in for the backbone writing the next
    block. Events order the two streams: block t waits for its set to be filled, the refill of
    a set waits for the block that last read it.

    Returns (elapsed ms of the `blocks` replays on `stream`, bytes copied per block, per-block
    output copies if keep else None)."""
    import torch
    anchor = pool[0]["x0"].clone()
    bufs = []
    for j in range(2):
        b = {k: pool[j % len(pool)][k].clone() for k in BLOCK_INPUTS}
        b["x0"] = anchor
        bufs.append(b)
    out = tail.alloc_outputs(full=keep)
    out["next_anchor"] = anchor
    torch.cuda.synchronize()
    graphs = [tail.graph(bufs[j], sm, vm, out=out, chain_anchor=False, stream=stream)
              for j in range(2)]
    prod = torch.cuda.Stream()
    ready = [torch.cuda.Event(), torch.cuda.Event()]
    done = [torch.cuda.Event(), torch.cuda.Event()]
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    nbytes = sum(bufs[0][k].numel() * bufs[0][k].element_size() for k in BLOCK_INPUTS)
    outs = [] if keep else None
    ready[0].record(prod)
    e0.record(stream)
    for t in range(blocks):
        k, nk = t % 2, 1 - t % 2
        with torch.cuda.stream(prod):
            if t >= 1:
                prod.wait_event(done[nk])
            src = pool[(t + 1) % len(pool)]
            for name in BLOCK_INPUTS:
                bufs[nk][name].copy_(src[name], non_blocking=True)
            ready[nk].record(prod)
        stream.wait_event(ready[k])
        graphs[k].launch()
        done[k].record(stream)
        if keep:
            with torch.cuda.stream(stream):
                outs.append({n: v.clone() for n, v in out.items()})
    e1.record(stream)
    stream.synchronize()
    prod.synchronize()
    for g in graphs:
        g.close()
    return e0.elapsed_time(e1), nbytes, outs
