"""A training step whose inputs arrive from pinned host memory.

The decoupled-loss step reads tens of GB of inputs (both logits tensors, the
token arrays) and the EWMA update reads the new actor parameters.  When those
come from host memory, the host link (~200 GB/s) bounds the step, not HBM.
``HostFedStep`` hides the kernels under the copies. The copies run on a
stream of their own, so step k's loss runs while its parameters are still
copying, and its EWMA update runs while step k+1's logits copy in. Events
order every reuse of a device buffer: step k+1's copies into the loss inputs
wait for step k's loss, and its parameter copy waits for step k's EWMA
update.  Everything is enqueued asynchronously; nothing here synchronises
the host.

This is orchestration of the library's entry points (``occ``) through torch
streams and events; every step of the computation runs in libocc's kernels.
"""

import torch


class HostFedStep:
    """Enqueues loss + EWMA steps whose inputs are copied in from the host.

    ``device_loss_inputs``: device tensors the loss reads (e.g. z_old,
    z_theta, ids, logp_mu, adv, mask); ``device_theta``: the device tensor the
    EWMA update reads as theta.  ``loss_fn()`` and ``ewma_fn()`` enqueue the
    kernels on the current stream and read only those device tensors (and
    their own outputs).  ``step(host_loss_inputs, host_theta)`` copies the
    host tensors (page-locked, same shapes and dtypes, in the same order) into
    the device tensors and enqueues the step; ``after_step()``, if given, runs
    on the compute stream after the EWMA update (e.g. a device-to-host read of
    the loss statistics).
    """

    def __init__(self, device_loss_inputs, device_theta, loss_fn, ewma_fn, after_step=None,
                 stream=None, copy_stream=None):
        self.dev_loss = list(device_loss_inputs)
        self.dev_theta = device_theta
        self.loss_fn, self.ewma_fn, self.after_step = loss_fn, ewma_fn, after_step
        dev = device_theta.device
        self.stream = stream if stream is not None else torch.cuda.current_stream(dev)
        self.copy_stream = copy_stream if copy_stream is not None else torch.cuda.Stream(dev)
        self.loss_done = torch.cuda.Event()
        self.ewma_done = torch.cuda.Event()
        self.loss_done.record(self.stream)
        self.ewma_done.record(self.stream)

    def bytes_per_step(self):
        return sum(t.numel() * t.element_size() for t in self.dev_loss + [self.dev_theta])

    def step(self, host_loss_inputs, host_theta):
        if len(host_loss_inputs) != len(self.dev_loss):
            raise ValueError("one host tensor per device loss input")
        for h, d in zip(list(host_loss_inputs) + [host_theta], self.dev_loss + [self.dev_theta]):
            if h.shape != d.shape or h.dtype != d.dtype or not h.is_pinned():
                raise ValueError("host inputs must be page-locked and match the device tensors")
        inputs_in, theta_in = torch.cuda.Event(), torch.cuda.Event()
        cs = self.copy_stream
        with torch.cuda.stream(cs):
            cs.wait_event(self.loss_done)      # the previous loss has read the loss inputs
            for h, d in zip(host_loss_inputs, self.dev_loss):
                d.copy_(h, non_blocking=True)
            inputs_in.record(cs)
            cs.wait_event(self.ewma_done)      # the previous update has read theta
            self.dev_theta.copy_(host_theta, non_blocking=True)
            theta_in.record(cs)
        with torch.cuda.stream(self.stream):
            self.stream.wait_event(inputs_in)
            self.loss_fn()
            self.loss_done.record(self.stream)
            self.stream.wait_event(theta_in)
            self.ewma_fn()
            self.ewma_done.record(self.stream)
            if self.after_step is not None:
                self.after_step()

    def start_timing(self, event):
        """Makes the copy stream wait for ``event`` (recorded on the compute
        stream), so that a timed region bracketed by events on the compute
        stream also covers the copies."""
        self.copy_stream.wait_event(event)
