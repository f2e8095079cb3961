"""The whole-optimizer step (Section 5.1 parameter grouping): MALT on the 2-D
weight matrices with fp32 master weights, their bf16 copies and decoupled
weight decay 0.1 (appendix table), and AdamW on every other tensor, against
the fp64 oracles.

Bars (fp32 arithmetic against fp64): AdamW moments within 1e-5 relative
(Frobenius, per tensor); each element of the update w_t - w_{t-1} within 1e-5
of the oracle's step (teacher-forced on the GPU's w_{t-1}) and of the step its
moment terms would give without cancellation, plus two fp32 ulps of w, the
resolution at which an fp32 master can move; master weights within
1e-6 (|w| + lr) elementwise; every bf16 copy equal, bit for bit, to the
round-to-nearest-even of the GPU's own fp32 master (integer-exact work)."""
import dataclasses

import numpy as np
import pytest

import oracle.adamw_ref as aref
import oracle.malt_ref as ref
import paper_2608_05088_gb300.malt as malt
from paper_2608_05088_gb300 import inputs
from tests.gpu_harness import Run, canaries_intact, guarded

pytestmark = pytest.mark.gpu

TOL_MOMENT = 1e-5
TOL_UPDATE = 1e-5
TOL_MASTER = 1e-6


def _host(t):
    return t.double().cpu().numpy()


def _rel(a, b):
    nb = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / nb) if nb > 0 else float(np.linalg.norm(a))


class AdamRun:
    """AdamW tensors on the GPU and their fp64 oracle states."""

    def __init__(self, shapes, wds, lr, seed, g_dtype="f32", copies=True, stream=None):
        import torch
        self.torch = torch
        dev = torch.device("cuda:0")
        self.rng = np.random.default_rng(seed)
        self.shapes, self.wds, self.lr, self.g_dtype = shapes, wds, lr, g_dtype
        gdt = torch.float32 if g_dtype == "f32" else torch.bfloat16
        self.w0 = [(self.rng.standard_normal(s) * 0.02).astype(np.float32) for s in shapes]
        # every buffer between canary margins (checked by close())
        self.bufs = []

        def buf(shape, dt):
            t, b = guarded(shape, dt, dev)
            self.bufs.append(b)
            return t
        self.w = [buf(s, torch.float32) for s in shapes]
        for t, x in zip(self.w, self.w0):
            t.copy_(torch.from_numpy(x))
        self.wc = [buf(s, torch.bfloat16) if copies else None for s in shapes]
        self.g = [buf(s, gdt).zero_() for s in shapes]
        self.m = [buf(s, torch.float32) for s in shapes]
        self.v = [buf(s, torch.float32) for s in shapes]
        self.params = list(zip(self.w, self.wc, self.g, self.m, self.v, wds))
        self.opt = malt.AdamW(self.params, stream)
        f32 = lambda x: float(np.float32(x))
        self.hp = malt.adamw_hparams(lr=lr)
        self.hp_ref = aref.AdamWHyper(lr=f32(lr), beta1=f32(0.9), beta2=f32(0.95), eps=f32(1e-8))
        self.w_ref = [x.astype(np.float64) for x in self.w0]
        self.st_ref = [aref.AdamWState.zeros(s) for s in shapes]

    def close(self):
        self.torch.cuda.synchronize()
        for k, b in enumerate(self.bufs):
            assert canaries_intact(b), f"a kernel wrote past AdamW buffer {k}"
        self.opt.close()

    def draw(self):
        gs = []
        for i, s in enumerate(self.shapes):
            g = (self.rng.standard_normal(s) * np.exp(self.rng.standard_normal(s))).astype(np.float32)
            if self.g_dtype == "bf16":
                g = inputs.bf16_representable(g)
            gs.append(g)
        return gs

    def step(self, grads, stream=None):
        for i, g in enumerate(grads):
            self.g[i].copy_(self.torch.from_numpy(g))
        self.w_prev = [_host(w) for w in self.w]
        self.m_prev_ref = [st.m.copy() for st in self.st_ref]
        self.g_last = [g.astype(np.float64) for g in grads]
        self.opt.step(self.hp, stream=stream)
        for i, g in enumerate(grads):
            self.w_ref[i], _ = aref.adamw_step_ref(self.w_ref[i], g.astype(np.float64), self.st_ref[i],
                                                   self.hp_ref, weight_decay=float(np.float32(self.wds[i])))

    def check(self, i, ctx=""):
        w = _host(self.w[i])
        msg = f"{ctx} tensor {i} {self.shapes[i]}"
        st = self.st_ref[i]
        assert _rel(_host(self.m[i]), st.m) < TOL_MOMENT, msg
        assert _rel(_host(self.v[i]), st.v) < TOL_MOMENT, msg
        # this step's update, the oracle teacher-forced on the GPU's previous w
        wd = float(np.float32(self.wds[i]))
        lr = self.hp_ref.lr
        t = st.t
        m_hat = st.m / (1 - self.hp_ref.beta1 ** t)
        v_hat = st.v / (1 - self.hp_ref.beta2 ** t)
        step_ref = (1 - lr * wd) * self.w_prev[i] - lr * m_hat / (np.sqrt(v_hat) + self.hp_ref.eps)
        # Elementwise: the step within 1e-5 of the size of the terms it is
        # computed from (m sums beta1 m and (1 - beta1) g, which can cancel,
        # so its fp32 error scales with those terms, not with m), plus the fp32
        # resolution of w itself (the decay product, the fused update and the
        # store each round w to fp32: at most two ulps of w together).
        hpr = self.hp_ref
        terms = hpr.beta1 * np.abs(self.m_prev_ref[i]) + (1 - hpr.beta1) * np.abs(self.g_last[i])
        scale = lr / (1 - hpr.beta1 ** t) * terms / (np.sqrt(v_hat) + hpr.eps)
        d_gpu, d_ref = w - self.w_prev[i], step_ref - self.w_prev[i]
        ulp = np.spacing(np.maximum(np.abs(w), np.abs(self.w_prev[i])).astype(np.float32))
        bound = TOL_UPDATE * (np.abs(d_ref) + scale) + 2.0 * ulp
        assert np.all(np.abs(d_gpu - d_ref) <= bound), (msg, float(np.max(np.abs(d_gpu - d_ref) / bound)))
        err = np.abs(w - self.w_ref[i])
        assert np.all(err <= TOL_MASTER * (np.abs(self.w_ref[i]) + lr)), (msg, float(err.max()))
        if self.wc[i] is not None:
            want = ref.round_to_bf16(w)
            assert np.array_equal(_host(self.wc[i]), want), msg


def test_adamw_against_oracle_ragged_sizes():
    """Tensors of every size class: sizes not a multiple of 4 (scalar tail),
    one element, runs over several 4096-element blocks, 2-D embeddings; with
    and without decay; 4 steps, every element checked."""
    shapes = [(1,), (3,), (7,), (768,), (2304,), (8195,), (40000,), (97, 131), (1024, 768)]
    wds = [0.0, 0.1, 0.0, 0.0, 0.1, 0.0, 0.1, 0.1, 0.1]
    run = AdamRun(shapes, wds, lr=0.01, seed=70)
    for s in range(4):
        run.step(run.draw())
        run.torch.cuda.synchronize()
        for i in range(len(shapes)):
            run.check(i, f"step {s}")
    assert run.opt.get_step() == 4
    run.close()


def test_adamw_bf16_gradients_without_copies():
    shapes = [(4096,), (300, 257), (5,)]
    run = AdamRun(shapes, [0.0, 0.1, 0.1], lr=3e-3, seed=71, g_dtype="bf16", copies=False)
    for s in range(3):
        run.step(run.draw())
        run.torch.cuda.synchronize()
        for i in range(len(shapes)):
            run.check(i, f"step {s}")
    run.close()


def test_adamw_zero_gradient_is_pure_decay():
    """g = 0: m and v stay 0 and each step multiplies w by (1 - lr wd) in fp32."""
    import torch
    shapes = [(1000,), (64, 48)]
    run = AdamRun(shapes, [0.1, 0.1], lr=0.02, seed=72)
    zeros = [np.zeros(s, np.float32) for s in shapes]
    for _ in range(3):
        run.step(zeros)
    torch.cuda.synchronize()
    decay = np.float32(1) - np.float32(0.02) * np.float32(0.1)
    for i, s in enumerate(shapes):
        want = run.w0[i]
        for _ in range(3):
            want = (want * decay).astype(np.float32)
        assert np.array_equal(run.w[i].cpu().numpy(), want)
        assert not torch.any(run.m[i]) and not torch.any(run.v[i])
    run.close()


def test_adamw_checkpoint_and_graph_replay():
    """Three eager steps equal one step, a save and restore of (w, m, v, t)
    into a fresh state, and two steps replayed from a CUDA graph, bitwise."""
    import torch
    shapes = [(5000,), (128, 96)]
    a = AdamRun(shapes, [0.0, 0.1], lr=0.01, seed=73)
    b = AdamRun(shapes, [0.0, 0.1], lr=0.01, seed=73)
    grads = a.draw()
    for r in (a, b):
        for i, g in enumerate(grads):
            r.g[i].copy_(torch.from_numpy(g))
    torch.cuda.synchronize()
    for _ in range(3):
        a.opt.step(a.hp)
    b.opt.step(b.hp)
    t = b.opt.get_step()
    saved = [[x.clone() for x in (b.w[i], b.m[i], b.v[i])] for i in range(2)]
    b.opt.close()
    c = AdamRun(shapes, [0.0, 0.1], lr=0.01, seed=73)
    for i in range(2):
        c.g[i].copy_(torch.from_numpy(grads[i]))
        for dst, src in zip((c.w[i], c.m[i], c.v[i]), saved[i]):
            dst.copy_(src)
    c.opt.set_step(t)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        with torch.cuda.graph(graph, stream=s):
            c.opt.step(c.hp, stream=s)
    torch.cuda.synchronize()
    for _ in range(2):
        graph.replay()
    torch.cuda.synchronize()
    assert a.opt.get_step() == c.opt.get_step() == 3
    for i in range(2):
        for x, y in ((a.w[i], c.w[i]), (a.m[i], c.m[i]), (a.v[i], c.v[i]), (a.wc[i], c.wc[i])):
            assert torch.equal(x, y)
    a.close()
    c.close()


def test_adamw_rejects_changed_sizes():
    import torch
    run = AdamRun([(100,), (64,)], [0.0, 0.0], lr=0.01, seed=74)
    with pytest.raises(malt.MaltError):
        run.opt.step(run.hp, params=run.params[:1])
    other = [(run.w[0][:50], None, run.g[0][:50], run.m[0][:50], run.v[0][:50], 0.0), run.params[1]]
    with pytest.raises(malt.MaltError):
        run.opt.step(run.hp, params=other)
    torch.cuda.synchronize()
    run.close()


def test_whole_optimizer_gpt2_small():
    """One model's whole step, GPT-2 Small (124M parameters): MALT on the 48
    matrices with fp32 master weights, bf16 copies and weight decay 0.1 at
    the MALT learning rate; AdamW on the 100 other tensors (tied embedding
    and head, position embedding, LayerNorms and biases) at the AdamW
    learning rate.  Two steps on one stream.  Every AdamW tensor is checked in
    full; one matrix of each shape against the MALT oracle, and every
    matrix's copy against its master."""
    import torch
    wl = inputs.WORKLOADS["gpt2_small"]
    wl32 = dataclasses.replace(wl, weight_dtype="f32")
    aset = inputs.ADAMW_SETS["gpt2_small"]
    check = [0, 1, 2, 3]
    mats = Run(wl32, check=check, weight_decay=0.1)
    copies = [torch.empty(s, dtype=torch.bfloat16, device="cuda:0") for s in wl.shapes]
    mats.opt.set_weight_copies(copies)
    shapes = [shape for _, shape, _ in aset.tensors]
    adam = AdamRun(shapes, [wd for _, _, wd in aset.tensors], lr=aset.lr, seed=75)
    # the set's own initial values and gradients
    for i in range(len(shapes)):
        adam.w0[i] = inputs.adamw_initial(aset, i)
        adam.w[i].copy_(torch.from_numpy(adam.w0[i]))
        adam.w_ref[i] = adam.w0[i].astype(np.float64)
    for s in range(2):
        mats.step()
        adam.step([inputs.adamw_gradient(aset, i, s) for i in range(len(shapes))])
        assert mats.status() == malt.MALT_OK
        torch.cuda.synchronize()
        for i in range(len(shapes)):
            adam.check(i, f"step {s}")
        for i in check:
            mats.assert_close(i, f"step {s}")
        for i in range(len(wl.shapes)):
            assert torch.equal(copies[i], mats.W[i].to(torch.bfloat16))
    mats.close()
    adam.close()


def test_weight_copies_need_fp32_weights():
    """Copies are written for fp32 weights only; a matrix with odd sizes
    (padded inside the library) gets its copy in the caller's layout."""
    import torch
    wl = inputs.Workload("copies", 76, ((256, 512), (392, 136), (250, 509)), "f32", 1.0, 0.02,
                         "malt", 1)
    run = Run(wl, check=[], w_dtypes=["bf16", "f32", "f32"])
    c = [torch.empty(s, dtype=torch.bfloat16, device="cuda:0") for s in wl.shapes]
    with pytest.raises(malt.MaltError):
        run.opt.set_weight_copies(c)                  # W of matrix 0 is bf16
    run.opt.set_weight_copies([None, c[1], c[2]])
    run.step(oracle=False)
    assert run.status() == malt.MALT_OK
    for i in (1, 2):
        assert torch.equal(c[i], run.W[i].to(torch.bfloat16))
    run.opt.set_weight_copies(None)
    run.close()
