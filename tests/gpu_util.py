"""Helpers shared by the GPU tests: device buffers for a workload, and the
oracle evaluated on sampled coordinates with host-regenerated residues."""
import numpy as np
import torch

import oracle
from paper_2609_35352_gb300 import fiona as F
from paper_2609_35352_gb300 import workloads as W


def to_device(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int64)).cuda()


def to_host(t: torch.Tensor) -> np.ndarray:
    return t.cpu().numpy().view(np.uint64)


class DeviceLayer:
    """A workload's plan on the GPU with its inputs, plaintexts and outputs."""

    def __init__(self, wl: W.Workload, host_inputs: bool = True, device: int = 0):
        self.wl = wl
        self.ctx = F.Context(wl.N, wl.moduli, device=device)
        self.plan = F.Plan(self.ctx, wl.plan)
        p = wl.plan
        if host_inputs:
            self.X = wl.host_inputs()
            self.P = wl.host_plaintexts()
            self.d_in = to_device(self.X) if self.X.size else torch.zeros(2, dtype=torch.int64, device="cuda")
            self.d_pt = to_device(self.P) if self.P.size else torch.zeros(2, dtype=torch.int64, device="cuda")
        else:
            self.X = self.P = None
            n_in = 2 * p.n_in * wl.L * wl.N
            n_pt = p.n_pt * wl.L * wl.N
            self.d_in = torch.empty(max(n_in, 2), dtype=torch.int64, device="cuda")
            self.d_pt = torch.empty(max(n_pt, 2), dtype=torch.int64, device="cuda")
            mode = 1 if wl.fill == "max" else 0
            F.device_fill(self.d_in, 2 * p.n_in, wl.L, wl.N, wl.moduli, wl.key(W.STREAM_INPUTS), mode)
            F.device_fill(self.d_pt, p.n_pt, wl.L, wl.N, wl.moduli, wl.key(W.STREAM_PLAINTEXTS), mode)
            if wl.const_pts:  # constant raw plaintexts come first
                F.device_fill(self.d_pt, wl.const_pts, wl.L, wl.N, wl.moduli, wl.key(W.STREAM_PLAINTEXTS), 2)
        self.d_out = torch.full((p.n_out * 2 * wl.L * wl.N,), -1, dtype=torch.int64, device="cuda")

    def run(self, stream=None) -> None:
        self.plan.eval(self.d_in, self.d_pt, self.d_out, stream=stream)

    def outputs(self) -> np.ndarray:
        torch.cuda.synchronize()
        wl = self.wl
        return to_host(self.d_out).reshape(wl.plan.n_out, 2, wl.L, wl.N)


def oracle_at(wl: W.Workload, limbs: np.ndarray, coefs: np.ndarray) -> np.ndarray:
    """Oracle outputs [n_out][2][len(samples)] at (limb, coefficient) samples,
    from residues regenerated on the host one by one."""
    p = wl.plan
    out = np.zeros((p.n_out, 2, limbs.shape[0]), dtype=np.uint64)
    for l in np.unique(limbs):
        sel = np.nonzero(limbs == l)[0]
        k = coefs[sel]
        X = wl.input_values(np.arange(p.n_in).reshape(-1, 1, 1), np.arange(2).reshape(1, -1, 1),
                            l, k.reshape(1, 1, -1)).reshape(p.n_in, 2, 1, -1)
        P = wl.plaintext_values(np.arange(p.n_pt).reshape(-1, 1), l, k.reshape(1, -1))
        P = P.reshape(p.n_pt, 1, -1)
        y = oracle.linear_eval(p, [wl.moduli[int(l)]], X, P)
        out[:, :, sel] = y[:, :, 0, :]
    return out
