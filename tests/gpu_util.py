"""Shared helpers of the GPU parity tests (run the library and the oracle on
the same seeded inputs and compare)."""
from __future__ import annotations

import numpy as np

import oracle
import workloads as WL

# Tolerances on the emitted chunk / buffer (bf16 and fp32 dtypes), on the velocity
# (bf16 internal diagnostic: rel-L2 only) and on the per-layer intermediates.
TOL = {"bf16": dict(max_abs=3e-2, rel_l2=1e-2), "fp32": dict(max_abs=1e-4, rel_l2=1e-4)}
VEL_REL_L2 = {"bf16": 2e-2, "fp32": 1e-4}


def errors(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    max_abs = float(np.abs(got - ref).max()) if got.size else 0.0
    denom = float(np.linalg.norm(ref))
    rel = float(np.linalg.norm(got - ref) / denom) if denom > 0 else float(np.linalg.norm(got))
    return max_abs, rel


def assert_close(got, ref, max_abs=None, rel_l2=None, what=""):
    ma, rl = errors(got, ref)
    msg = f"{what}: max_abs={ma:.3e} rel_l2={rl:.3e}"
    print(msg)  # the measured errors, shown with pytest -s / -rP
    if max_abs is not None:
        assert ma <= max_abs, msg
    if rel_l2 is not None:
        assert rl <= rel_l2, msg
    return ma, rl


class Case:
    """A workload with its seeded inputs, a loaded Decoder and device buffers."""

    def __init__(self, wl, recipe="unit_gate", flags=0, weights_on_device=False, max_batch=None,
                 max_prefix=None, noise_seed=0):
        import torch
        from paper_2608_27384_gb300.harness import Decoder
        self.wl = wl
        self.w = WL.make_weights(wl, recipe=recipe)
        self.prefix = WL.make_prefix_kv(wl)
        self.buf = WL.make_buffer(wl)
        self.tau = WL.make_noise_levels(wl)
        self.dec = Decoder(wl, WL.flat_weights(wl, self.w), self.prefix, max_batch=max_batch,
                           max_prefix=max_prefix, flags=flags, noise_seed=noise_seed,
                           weights_on_device=weights_on_device)
        self.torch = torch

    @property
    def handle(self):
        return self.dec.handle

    def dev(self, a):
        return self.torch.from_numpy(np.ascontiguousarray(a)).cuda()

    def run(self, buf=None, tau=None, fresh=None, want_vel=True, trace_layer=-1, batch=None,
            n_valid=None, reuse_film=False, serial_film=False):
        """One GPU step.  Returns dict(out, buffer, vel[, trace]) as numpy arrays."""
        import paper_2608_27384_gb300 as fva
        torch = self.torch
        wl = self.wl
        B = batch or wl.batch
        buf = self.buf if buf is None else buf
        tau = self.tau if tau is None else tau
        d_buf = self.dev(buf[:B])
        d_out = torch.full((B, wl.chunk_tokens, wl.action_dim), float("nan"), device="cuda")
        d_vel = torch.empty((B, wl.n_chunks, wl.chunk_tokens, wl.action_dim), device="cuda") \
            if want_vel else None
        d_fresh = self.dev(fresh[:B]) if fresh is not None else None
        d_tr = None
        if trace_layer >= 0:
            d_tr = torch.empty(fva.fva_trace_floats(self.handle, B), device="cuda")
        fva.fva_step_ex(self.handle, d_buf, tau[:B], d_out, B, fresh_noise=d_fresh,
                        velocity_out=d_vel, trace_layer=trace_layer, trace_out=d_tr,
                        n_valid=None if n_valid is None else list(n_valid)[:B],
                        reuse_film=reuse_film, serial_film=serial_film)
        torch.cuda.synchronize()
        res = dict(out=d_out.cpu().numpy(), buffer=d_buf.cpu().numpy())
        if want_vel:
            res["vel"] = d_vel.cpu().numpy()
        if d_tr is not None:
            res["trace"] = d_tr.cpu().numpy()
        return res

    def oracle_step(self, buf=None, tau=None, fresh=None, batch=None, n_valid=None):
        wl = self.wl
        B = batch or wl.batch
        buf = self.buf if buf is None else buf
        tau = self.tau if tau is None else tau
        if fresh is None:
            fresh = np.zeros((B, wl.chunk_tokens, wl.action_dim), np.float32)
        return oracle.stream_step(self.w, wl.as_config(), buf[:B], tau[:B], self.prefix[:B],
                                  fresh[:B], None if n_valid is None else list(n_valid)[:B])

    def close(self):
        self.dec.close()


def split_trace(wl, flat, batch):
    """Views of fva_step_ex's trace buffer, in the documented order."""
    M = batch * wl.tokens
    W, Dq, dh, F = wl.width, wl.n_q_heads * wl.head_dim, wl.head_dim, wl.mlp_dim
    names = [("h_in", W), ("y1", W), ("q", Dq), ("k", dh), ("v", dh), ("attn", Dq),
             ("h_mid", W), ("y2", W), ("mlp", F), ("h_out", W)]
    out, off = {}, 0
    for n, c in names:
        out[n] = flat[off:off + M * c].reshape(M, c)
        off += M * c
    out["cond"] = flat[off:off + batch * wl.n_chunks * W].reshape(batch * wl.n_chunks, W)
    assert off + batch * wl.n_chunks * W == flat.size
    return out
