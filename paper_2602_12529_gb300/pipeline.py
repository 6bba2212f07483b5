"""Host-fed step pipeline: runs one device step per host-resident batch with
the host-to-device copies of batch k + 1 and the device-to-host copies of
batch k's results on a side stream, so both overlap batch k's kernels.

A rollout service receives its batches (initial noise, text embeddings,
times, rewards) in host memory and hands its results (x_next, log-probs,
loss) back there; with the copies on the compute stream every batch pays
them in series.  Here the device holds two input sets and two output sets:
batch k computes on set k % 2 while the copy stream fills set (k + 1) % 2
and drains the results of batch k - 1.  Events order the two streams:
  up[s]    inputs of set s landed (copy stream)      -> compute may start
  done[s]  the step on set s finished (compute)      -> its results may be
           copied out, and set s may take new inputs
  down[s]  results of set s copied out (copy stream) -> set s's outputs may
           be overwritten
The step itself is any sequence of library calls on the current stream.
"""
from __future__ import annotations


class HostFedPipeline:
    def __init__(self, device, inputs: dict, outputs: dict, step):
        """inputs / outputs: {name: device tensor} shaped like one batch's
        input / result (two device copies of each are made); step(ins, outs)
        enqueues one batch's work on the current stream, reading the tensors
        of ins and writing those of outs."""
        import torch
        self.dev = device
        self.ins = [{k: torch.empty_like(v) for k, v in inputs.items()} for _ in range(2)]
        self.outs = [{k: torch.empty_like(v) for k, v in outputs.items()} for _ in range(2)]
        self.copy = torch.cuda.Stream(device)
        self.step = step
        self.up = [torch.cuda.Event() for _ in range(2)]
        self.done = [torch.cuda.Event() for _ in range(2)]
        self.down = [torch.cuda.Event() for _ in range(2)]

    def run(self, host_inputs, host_outputs):
        """host_inputs[k]: {name: pinned host tensor} of batch k;
        host_outputs[k]: {name: pinned host tensor} its results land in.
        Everything is enqueued behind the work already on the current stream,
        and the current stream waits for the last copy out, so an event
        recorded on it afterwards (or a synchronise) covers the whole run."""
        import torch
        n = len(host_inputs)
        if n == 0:
            return
        comp, copy = torch.cuda.current_stream(self.dev), self.copy
        start = torch.cuda.Event()
        start.record(comp)
        copy.wait_event(start)

        def upload(k):
            s = k % 2
            with torch.cuda.stream(copy):
                if k >= 2:
                    copy.wait_event(self.done[s])      # batch k - 2 has finished reading set s
                for name, h in host_inputs[k].items():
                    self.ins[s][name].copy_(h, non_blocking=True)
                self.up[s].record(copy)

        upload(0)
        for k in range(n):
            s = k % 2
            if k + 1 < n:
                upload(k + 1)
            comp.wait_event(self.up[s])
            if k >= 2:
                comp.wait_event(self.down[s])          # batch k - 2's results have left set s
            self.step(self.ins[s], self.outs[s])
            self.done[s].record(comp)
            with torch.cuda.stream(copy):
                copy.wait_event(self.done[s])
                for name, h in host_outputs[k].items():
                    h.copy_(self.outs[s][name], non_blocking=True)
                self.down[s].record(copy)
        comp.wait_event(self.down[(n - 1) % 2])
