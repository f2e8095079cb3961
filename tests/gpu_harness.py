"""Drive the CUDA library and the fp64 oracle on the same seeded inputs."""
from __future__ import annotations

import numpy as np

import oracle.malt_ref as ref
from paper_2608_05088_gb300 import inputs

# Tolerances (the first three are the project's stated bars; see test docstrings).
TOL_STATS = 1e-5   # momentum, statistics, ||Mt||: fp32 arithmetic vs fp64
TOL_DIR = 2e-2     # orthogonalised direction O: bf16 NS operands, fp32 accumulation
TOL_W = 5e-3       # final weights, relative Frobenius
TOL_DW = 2e-2      # the update W_0 - W_t: D = L O R, so O's tolerance carries over


def rel(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    nb = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / nb) if nb > 0 else float(np.linalg.norm(a))


def bf16_ulp(x: np.ndarray) -> np.ndarray:
    """Spacing of bf16 numbers at |x| (8 significant bits)."""
    x = np.abs(np.asarray(x, dtype=np.float64))
    _, e = np.frexp(np.where(x > 0, x, 1e-38))
    return np.ldexp(1.0, np.maximum(e - 8, -133))


class Run:
    """One optimizer state on the GPU plus oracle states for `check` matrices."""

    def __init__(self, wl: inputs.Workload, check=None, g_dtype="f32", w_dtypes=None,
                 variant=None, device="cuda:0", ns_coeffs=ref.DEFAULT_NS_COEFFS, **hyper):
        import torch
        import paper_2608_05088_gb300.malt as malt
        self.torch, self.malt = torch, malt
        self.wl = wl
        self.variant = variant or wl.variant
        self.dev = torch.device(device)
        n = len(wl.shapes)
        self.check = list(range(n)) if check is None else list(check)
        self.g_dtype = g_dtype
        self.w_dtypes = w_dtypes or [wl.weight_dtype] * n
        tdt = {"f32": torch.float32, "bf16": torch.bfloat16}
        self.W0 = {}
        self.W, self.G, self.M, self.l, self.r = [], [], [], [], []
        for i, (m, c) in enumerate(wl.shapes):
            w0 = inputs.initial_weight(wl, i)
            if self.w_dtypes[i] == "bf16":
                w0 = inputs.bf16_representable(w0)
            if i in self.check:
                self.W0[i] = w0.astype(np.float64)
            self.W.append(torch.from_numpy(w0).to(self.dev).to(tdt[self.w_dtypes[i]]))
            self.G.append(torch.zeros((m, c), dtype=tdt[g_dtype], device=self.dev))
            self.M.append(torch.empty((m, c), dtype=torch.float32, device=self.dev))
            self.l.append(torch.empty(m, dtype=torch.float32, device=self.dev))
            self.r.append(torch.empty(c, dtype=torch.float32, device=self.dev))
        self.params = list(zip(self.W, self.G, self.M, self.l, self.r))
        self.opt = malt.MaltOptimizer(self.params)
        # Extra hyperparameters (mu1, mu2, eps, weight_decay, ns_eps) go to both
        # sides.  The library takes its hyperparameters as fp32, so the oracle
        # gets the same fp32 values (1 - 0.999f differs from 1 - 0.999 by 1.3e-5
        # relative, more than the statistics bar).
        f32 = lambda v: float(np.float32(v))
        self.hp_ref = ref.Hyper(lr=f32(wl.lr), ns_steps=wl.ns_steps,
                                ns_coeffs=tuple(f32(c) for c in ns_coeffs),
                                **{k: f32(v) for k, v in hyper.items()})
        self.hp = malt.hparams(lr=wl.lr, ns_steps=wl.ns_steps, ns_coeffs=tuple(ns_coeffs), **hyper)
        # the apply kernel's decay factor, 1 - lr * wd evaluated in fp32
        self.decay_gpu = float(np.float32(1) - np.float32(wl.lr) * np.float32(self.hp_ref.weight_decay))
        self.W_ref = dict(self.W0)
        self.st_ref = {i: ref.State.zeros(*wl.shapes[i]) for i in self.check}
        self.info = {}
        self.steps_done = 0

    def gradient(self, i, step):
        G = inputs.gradient(self.wl, i, step)
        if self.g_dtype == "bf16":
            G = inputs.bf16_representable(G)
        return G

    def step(self, grads=None, oracle=True):
        """One step on the GPU (and the oracle for checked matrices)."""
        s = self.steps_done
        self.W_prev = {i: self.host(self.W[i]) for i in self.check if self.w_dtypes[i] == "bf16"}
        self.W_prev_ref = {i: self.W_ref[i].copy() for i in self.W_prev}
        for i in range(len(self.wl.shapes)):
            G = grads[i] if grads is not None else self.gradient(i, s)
            self.G[i].copy_(self.torch.from_numpy(np.ascontiguousarray(G)))
            if oracle and i in self.check:
                # Muon through the same engine = MALT with identity preconditioners
                self.W_ref[i], self.info[i] = ref.malt_step_ref(
                    self.W_ref[i], G.astype(np.float64), self.st_ref[i], self.hp_ref,
                    variant="malt" if self.variant == "muon" else self.variant,
                    weight_dtype=self.w_dtypes[i], force_identity=(self.variant == "muon"))
        self.opt.step(self.hp, malter=(self.variant == "malter"), muon=(self.variant == "muon"))
        self.steps_done += 1

    def status(self):
        return self.opt.check()

    def host(self, t):
        return t.double().cpu().numpy()

    def compare(self, i):
        """Errors of matrix i against the oracle after the last step."""
        st = self.st_ref[i]
        info = self.info[i]
        W = self.host(self.W[i])
        O = self.host(self.opt.direction(i))
        sc = self.opt.debug_scalars()[i]
        if self.w_dtypes[i] == "bf16":
            # bf16 rounding decides most entries of W_0 - W_t, so compare the
            # pre-rounding update rebuilt from the GPU's own l, r, O and scale.
            eps = self.hp_ref.eps
            if self.variant == "muon":
                Lg, Rg = np.ones(W.shape[0]), np.ones(W.shape[1])
            else:
                Lg = (self.host(self.l[i]) + eps) ** -0.125
                Rg = (self.host(self.r[i]) + eps) ** -0.125
            dW = float(sc[6]) * Lg[:, None] * O * Rg[None, :]
            dW_ref = info["delta"]
            # the GPU's own pre-rounding value, decoupled decay included
            W_pre = self.decay_gpu * self.W_prev[i] - dW
            hp = self.hp_ref
            W_pre_ref = (1.0 - hp.lr * hp.weight_decay) * self.W_prev_ref[i] - dW_ref
        else:
            dW = self.W0[i] - W
            dW_ref = self.W0[i] - self.W_ref[i]
        stats_used = self.variant != "muon"      # Muon leaves l and r untouched
        return dict(
            M=rel(self.host(self.M[i]), st.M),
            l=float(np.max(np.abs(self.host(self.l[i]) - st.l) / np.maximum(st.l, 1e-30)))
            if stats_used else 0.0,
            r=float(np.max(np.abs(self.host(self.r[i]) - st.r) / np.maximum(st.r, 1e-30)))
            if stats_used else 0.0,
            O=rel(O, info["O"]),
            W=rel(W, self.W_ref[i]),
            dW=rel(dW, dW_ref),
            norm_mt=abs(sc[2] - info["norm_Mt"]) / max(info["norm_Mt"], 1e-30),
            norm_o=abs(sc[0] - info["norm_O"]) / max(info["norm_O"], 1e-30),
            norm_d=abs(sc[1] - info["norm_D"]) / max(info["norm_D"], 1e-30),
            alpha=abs(sc[5] - info["alpha"]) / max(abs(info["alpha"]), 1e-30),
            nu=(abs(sc[4] - info["nu"]) / max(info["nu"], 1e-30)) if self.variant == "malter" else 0.0,
            W_gpu=W,
            W_pre=W_pre if self.w_dtypes[i] == "bf16" else None,
            W_pre_ref=W_pre_ref if self.w_dtypes[i] == "bf16" else None,
        )

    def assert_close(self, i, ctx=""):
        e = self.compare(i)
        msg = f"{ctx} matrix {i} {self.wl.shapes[i]}: " + ", ".join(
            f"{k}={v:.3g}" for k, v in e.items() if k not in ("W_gpu", "W_pre", "W_pre_ref"))
        assert e["M"] < TOL_STATS and e["l"] < TOL_STATS and e["r"] < TOL_STATS, msg
        assert e["norm_mt"] < TOL_STATS, msg
        assert e["O"] < TOL_DIR and e["norm_o"] < TOL_DIR and e["norm_d"] < TOL_DIR, msg
        assert e["W"] < TOL_W and e["dW"] < TOL_DW, msg
        if self.variant == "malter":
            assert e["nu"] < 1e-4 and e["alpha"] < 1e-4, msg
        if self.w_dtypes[i] == "bf16":
            # Rounding x and y to nearest bf16 moves them apart by at most
            # |x - y| + one ulp, with x, y the GPU's and the oracle's
            # pre-rounding values; and the stored W is the round-to-nearest-
            # even of the GPU's own pre-rounding value (fp32 arithmetic decides
            # a few near-ties).
            Wr = self.W_ref[i]
            diff = np.abs(e["W_gpu"] - Wr)
            gap = np.abs(e["W_pre"] - e["W_pre_ref"])
            ulp = bf16_ulp(np.maximum(np.abs(e["W_pre"]), np.abs(e["W_pre_ref"])))
            assert np.all(diff <= gap * 1.001 + ulp * 1.0001), msg
            own = ref.round_to_bf16(e["W_pre"])
            assert np.mean(own != e["W_gpu"]) < 5e-3, msg + f", rne mismatch={np.mean(own != e['W_gpu']):.3g}"
        return e

    def close(self):
        self.opt.close()
