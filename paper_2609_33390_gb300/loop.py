"""Host-side decode loop over captured decode tails (App. F: fused head plus CUDA Graph
replay), with the next block's inputs written while the current block runs. Only streams,
events and graph launches: every step of the tail runs in the library's kernels."""
from __future__ import annotations

BLOCK_INPUTS = ("logits_q", "logits_p", "hidden", "h_c", "u_sel", "u_acc", "u_res")


def double_buffer_schedule(blocks: int, pool_len: int):
    """The operations of the double-buffered loop in issue order, as tuples:

      ("copy_wait", s)      the copy stream waits for `done[s]` (the last block that read set s)
      ("copy", s, j)        the copy stream fills input set s from pool block j
      ("copy_ready", s)     `ready[s]` is recorded on the copy stream
      ("run_wait", s)       the compute stream waits for `ready[s]`
      ("launch", s, t)      block t runs (the graph captured over set s)
      ("run_done", s)       `done[s]` is recorded on the compute stream

    Set s = t % 2 holds block t; it starts out holding pool block s. While block t runs, the
    other set is refilled with pool block (t + 1) % pool_len, after the block that last read it."""
    ops = [("copy_ready", 0)]
    for t in range(blocks):
        k, nk = t % 2, 1 - t % 2
        if t >= 1:
            ops.append(("copy_wait", nk))
        ops.append(("copy", nk, (t + 1) % pool_len))
        ops.append(("copy_ready", nk))
        ops.append(("run_wait", k))
        ops.append(("launch", k, t))
        ops.append(("run_done", k))
    return ops


def graph_loop_double_buffered(tail, pool, sm, vm, stream, blocks, keep=False):
    """Block after block through two captured decode tails (App. F), one per input buffer set,
    the anchor chained on the device through one buffer both graphs share. While block t runs
    on `stream`, a second stream copies block t+1's inputs from `pool` (pre-generated blocks,
    taken in turn) into the other buffer set: the stand-in for the backbone writing the next
    block. Events order the two streams as `double_buffer_schedule` lists.

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
    ops = double_buffer_schedule(blocks, len(pool))
    e0.record(stream)
    for op in ops:
        kind, s = op[0], op[1]
        if kind == "copy_wait":
            prod.wait_event(done[s])
        elif kind == "copy":
            with torch.cuda.stream(prod):
                src = pool[op[2]]
                for name in BLOCK_INPUTS:
                    bufs[s][name].copy_(src[name], non_blocking=True)
        elif kind == "copy_ready":
            ready[s].record(prod)
        elif kind == "run_wait":
            stream.wait_event(ready[s])
        elif kind == "launch":
            graphs[s].launch()
            if keep:
                with torch.cuda.stream(stream):
                    outs.append({n: v.clone() for n, v in out.items()})
        elif kind == "run_done":
            done[s].record(stream)
    e1.record(stream)
    stream.synchronize()
    prod.synchronize()
    for g in graphs:
        g.close()
    return e0.elapsed_time(e1), nbytes, outs
