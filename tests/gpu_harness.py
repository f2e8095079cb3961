"""Drive the CUDA library and the fp64 oracle on the same seeded inputs."""
from __future__ import annotations

import numpy as np

import oracle.malt_ref as ref
from paper_2608_05088_gb300 import inputs
from tests import bf16_ns_model

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


def bf16_rounding(W_gpu, x_gpu, x_ref, slack, dW_ref):
    """Rounding checks of a bf16 weight update against the oracle.

    x_gpu: the GPU's pre-rounding value rebuilt in fp64 (exact up to `slack`,
    the kernel's own fp32 rounding); x_ref: the oracle's.  An entry
    "straddles" when a bf16 rounding boundary lies between the two values
    (the interval widened by the slack); elsewhere both must round alike.
      own_mismatch: entries with W_gpu != rn(x_gpu) although no boundary lies
        within the slack of x_gpu (must be 0);
      oracle_mismatch_off_boundary: entries with W_gpu != rn(x_ref) that do
        not straddle (must be 0);
      straddle: the fraction of entries that straddle;
      straddle_allowed: the fraction the update tolerance would allow, the
        mean over entries of min(1, TOL_DW |dW_ref| / ulp) -- the chance that
        a boundary falls between two values that far apart.
    """
    rn = ref.round_to_bf16
    near = rn(x_gpu - slack) != rn(x_gpu + slack)            # within slack of a boundary
    own_mismatch = int(np.sum((W_gpu != rn(x_gpu)) & ~near))
    lo = np.minimum(x_gpu, x_ref) - slack
    hi = np.maximum(x_gpu, x_ref) + slack
    straddle = rn(lo) != rn(hi)
    off = int(np.sum((W_gpu != rn(x_ref)) & ~straddle))
    ulp = bf16_ulp(np.maximum(np.abs(x_ref), np.abs(x_gpu)))
    allowed = float(np.mean(np.minimum(1.0, TOL_DW * np.abs(dW_ref) / ulp)))
    return dict(own_mismatch=own_mismatch, oracle_mismatch_off_boundary=off,
                straddle=float(np.mean(straddle)), straddle_allowed=allowed)


CANARY = 64                    # elements of margin before and after every caller buffer
CANARY_VALUE = -7.625e7         # a value no step writes (exact in fp32 and bf16)


def guarded(shape, dtype, device):
    """A contiguous tensor of `shape` inside a larger allocation whose CANARY
    elements before and after hold CANARY_VALUE (16-byte aligned: the margin
    is 256 bytes in fp32, 128 in bf16).  Returns (tensor, whole allocation)."""
    import torch
    n = int(np.prod(shape))
    buf = torch.full((n + 2 * CANARY,), CANARY_VALUE, dtype=dtype, device=device)
    return buf[CANARY:CANARY + n].view(shape), buf


def canaries_intact(buf) -> bool:
    import torch
    return bool(torch.all(buf[:CANARY] == CANARY_VALUE) and torch.all(buf[-CANARY:] == CANARY_VALUE))


class Run:
    """One optimizer state on the GPU plus oracle states for `check` matrices.
    Every caller buffer (W, G, M, l, r) sits between canary margins, and
    close() checks them and the library's workspace guards: a kernel that
    writes past any buffer fails the test."""

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
        self.bufs = []
        for i, (m, c) in enumerate(wl.shapes):
            w0 = inputs.initial_weight(wl, i)
            if self.w_dtypes[i] == "bf16":
                w0 = inputs.bf16_representable(w0)
            if i in self.check:
                self.W0[i] = w0.astype(np.float64)
            for lst, shape, dt in ((self.W, (m, c), tdt[self.w_dtypes[i]]),
                                   (self.G, (m, c), tdt[g_dtype]),
                                   (self.M, (m, c), torch.float32), (self.l, (m,), torch.float32),
                                   (self.r, (c,), torch.float32)):
                t, buf = guarded(shape, dt, self.dev)
                lst.append(t)
                self.bufs.append(buf)
            self.W[-1].copy_(torch.from_numpy(w0))
            self.G[-1].zero_()
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
        Lg, Rg = (self.host(t) for t in self.opt.precond(i))
        sc = self.opt.debug_scalars()[i]
        out = dict(W_gpu=W, W_pre=None, W_pre_ref=None, slack=None)
        if self.w_dtypes[i] == "bf16":
            # bf16 rounding decides most entries of W_0 - W_t, so compare the
            # pre-rounding update, rebuilt exactly (fp64) from the step's own
            # L, R, bf16 O and fp32 scale, with the oracle's.
            dW = float(sc[6]) * Lg[:, None] * O * Rg[None, :]
            dW_ref = info["delta"]
            hp = self.hp_ref
            # Both pre-rounding values start from the GPU's previous W (the
            # oracle teacher-forced), so their gap is this step's only.
            W_pre = self.decay_gpu * self.W_prev[i] - dW
            W_pre_ref = (1.0 - hp.lr * hp.weight_decay) * self.W_prev[i] - dW_ref
            # the apply kernel's own fp32 arithmetic (s L_i, its product with
            # O_ij, decay * W, one fma) moves its value from W_pre by at most a
            # few fp32 ulps of the terms
            out.update(W_pre=W_pre, W_pre_ref=W_pre_ref,
                       slack=2.0 ** -21 * (np.abs(W_pre) + np.abs(dW)))
        else:
            dW = self.W0[i] - W
            dW_ref = self.W0[i] - self.W_ref[i]
        stats_used = self.variant != "muon"      # Muon leaves l and r untouched

        def elem(a, b):
            return float(np.max(np.abs(a - b) / np.maximum(np.abs(b), 1e-30)))
        out.update(
            M=rel(self.host(self.M[i]), st.M),
            l=elem(self.host(self.l[i]), st.l) if stats_used else 0.0,
            r=elem(self.host(self.r[i]), st.r) if stats_used else 0.0,
            L=elem(Lg, info["L"]),
            R=elem(Rg, info["R"]),
            O=rel(O, info["O"]),
            W=rel(W, self.W_ref[i]),
            dW_over_W=float(np.linalg.norm(self.W0[i] - self.W_ref[i]) /
                            max(np.linalg.norm(self.W_ref[i]), 1e-30)),
            dW=rel(dW, dW_ref),
            norm_mt=abs(sc[2] - info["norm_Mt"]) / max(info["norm_Mt"], 1e-30),
            norm_o=abs(sc[0] - info["norm_O"]) / max(info["norm_O"], 1e-30),
            norm_d=abs(sc[1] - info["norm_D"]) / max(info["norm_D"], 1e-30),
            alpha=abs(sc[5] - info["alpha"]) / max(abs(info["alpha"]), 1e-30),
            nu=(abs(sc[4] - info["nu"]) / max(info["nu"], 1e-30)) if self.variant == "malter" else 0.0,
        )
        if self.w_dtypes[i] == "bf16":
            out.update(bf16_rounding(W, out["W_pre"], out["W_pre_ref"], out["slack"], dW_ref))
        return out

    def assert_close(self, i, ctx=""):
        e = self.compare(i)
        arrays = ("W_gpu", "W_pre", "W_pre_ref", "slack")
        msg = f"{ctx} matrix {i} {self.wl.shapes[i]}: " + ", ".join(
            f"{k}={v:.3g}" for k, v in e.items() if k not in arrays)
        assert e["M"] < TOL_STATS and e["l"] < TOL_STATS and e["r"] < TOL_STATS, msg
        assert e["L"] < TOL_STATS and e["R"] < TOL_STATS, msg
        assert e["norm_mt"] < TOL_STATS, msg
        direction = ("O", "norm_o", "norm_d", "dW")
        if not all(e[k] < TOL_DIR for k in direction):
            # Where bf16 Newton-Schulz operands (the arithmetic the bar itself
            # fixes) cannot meet 2e-2 on this input, the GPU must be no worse
            # than a CPU model of that arithmetic.
            model = bf16_ns_model.step_errors(self.info[i], self.hp_ref)
            msg += ", model: " + ", ".join(f"{k}={v:.3g}" for k, v in model.items())
            assert max(model.values()) >= 0.9 * TOL_DIR, msg
            assert all(e[k] <= 1.25 * model[k] + 2e-3 for k in direction), msg
        # The final weights within 5e-3, or within what the update's own bar
        # implies when the steps moved W by a large part of itself (a 1 x 1
        # matrix at lr 0.02): |W_gpu - W_ref| <= |dW_gpu - dW_ref|.
        assert e["W"] < max(TOL_W, max(TOL_DW, e["dW"]) * e["dW_over_W"]), msg
        if self.variant == "malter":
            assert e["nu"] < 1e-4 and e["alpha"] < 1e-4, msg
        if self.w_dtypes[i] == "bf16":
            # The stored bf16 W is the round-to-nearest-even of the GPU's own
            # pre-rounding value, and equals the oracle's rounding wherever no
            # rounding boundary lies between the two pre-rounding values.
            assert e["own_mismatch"] == 0, msg
            assert e["oracle_mismatch_off_boundary"] == 0, msg
            # Where a boundary does lie between them the two roundings may
            # differ.  That happens on a fraction of the entries set by the
            # pre-rounding gap, which grows with the update (so with the
            # learning rate): at most the fraction the update tolerance
            # allows, and at most 1 % for the GPT-2 sets at the paper's MALT
            # learning rates (MALTER's tuned rates are ten times larger).
            assert e["straddle"] <= e["straddle_allowed"] + 1e-3, msg
            if self.wl.name.startswith("gpt2") and self.variant == "malt":
                assert e["straddle"] <= 0.01, msg
        return e

    def close(self):
        """Check that no kernel wrote outside its buffers, then free the state."""
        self.torch.cuda.synchronize()
        assert self.opt.guard_bytes_corrupted() == 0, "a kernel wrote past a workspace buffer"
        for k, buf in enumerate(self.bufs):
            assert canaries_intact(buf), f"a kernel wrote past caller buffer {k} (W, G, M, l, r per matrix)"
        self.opt.close()
