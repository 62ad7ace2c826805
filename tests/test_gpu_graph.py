"""The benchmarked step captured into one CUDA graph and replayed.

gather -> forward keeping the logits -> accepted length -> G from the kept logits -> dH -> dW,
all through the C ABI on the current stream.  Every call only enqueues work (tensor maps are
encoded on the host at capture and travel as kernel parameters), so the graph replays the
device work alone; the kernels are deterministic, so a replay is bit-identical to the eager
run on the same inputs, and after new inputs are copied into the captured buffers a replay
matches an eager run on those inputs."""

import pytest
import torch

from paper_2609_38795_gb300 import alr, build_lib, synthetic

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    build_lib.build()
    alr.lib()
    assert alr.alr_device_supported() == alr.ALR_OK, alr.alr_last_error()


A, B, d, V, S, L = 64, 16, 1024, 8192, 4, 512


def _inputs(seed):
    b = synthetic.rollout_batch(d, V, A, B, S, L, 0.5, dtype=torch.bfloat16, device="cuda",
                                seed=seed)
    b["Ht"] = torch.empty(A * B, d, dtype=torch.bfloat16, device="cuda")
    b["row_valid"] = torch.empty(A * B, device="cuda")
    return b


class _Step:
    def __init__(self, x):
        self.x = x
        self.sl = alr.SlotLoss(A * B, d, V, B, keep_logits=True)
        self.dH = torch.empty(A * B, d, device="cuda")
        self.dW = torch.empty(d, V, device="cuda")

    def run(self):
        x, sl = self.x, self.sl
        alr.alr_gather_ira_blocks(x["F"], x["seq"], x["pos"], B, x["Ht"], x["row_valid"])
        sl.forward(x["Hd"], x["Ht"], x["W"], row_mask=x["row_valid"])
        sl.accept(active=x["row_valid"])
        o = sl.out
        G = sl.G                                            # G is written over z_d
        alr.alr_logit_grad_from_logits(sl.params, sl.Zd, sl.Zt, sl.Zd_ref, sl.Zt_ref, o["weight"],
                                       o["weight_sum"], o["lse_d"], o["lse_t"], G)
        alr.alr_gemm(G, x["W"], self.dH, A * B, d, V)
        self.dW.zero_()
        alr.alr_gemm(x["Hd"], G, self.dW, d, V, A * B, a_mn=True, b_mn=True, accumulate=True)

    def results(self):
        o = self.sl.out
        r = {k: o[k].clone() for k in ("loss_row", "lse_d", "lse_t", "argmax_d", "argmax_t",
                                       "weight", "loss_total", "weight_sum")}
        r.update(acc=self.sl.acc_len.clone(), hist=self.sl.hist.clone(), dH=self.dH.clone(),
                 dW=self.dW.clone(), Ht=self.x["Ht"].clone())
        return r


def _same(a, b):
    for k in a:
        x, y = a[k], b[k]
        if x.dtype.is_floating_point:
            x, y = x.float().view(torch.int32), y.float().view(torch.int32)
        assert torch.equal(x, y), k


def test_step_replays_from_a_cuda_graph():
    x = _inputs(seed=3)
    step = _Step(x)
    step.run()                                           # eager; also loads every kernel form
    torch.cuda.synchronize()
    eager = step.results()
    assert alr.alr_device_status() == alr.ALR_OK

    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step.run()
    graph.replay()
    torch.cuda.synchronize()
    _same(eager, step.results())
    graph.replay()                                       # again: no state left over
    torch.cuda.synchronize()
    _same(eager, step.results())

    # new inputs in the captured buffers: the replay computes on them
    y = _inputs(seed=4)
    for k in ("F", "Hd", "W", "seq", "pos"):
        x[k].copy_(y[k])
    graph.replay()
    torch.cuda.synchronize()
    replayed = step.results()
    fresh = _Step(y)
    fresh.run()
    torch.cuda.synchronize()
    _same(fresh.results(), replayed)
    assert not torch.equal(replayed["dW"], eager["dW"])
    assert alr.alr_device_status() == alr.ALR_OK
