"""The boundary step captured once into a CUDA graph and replayed.

Every call of the library is stream-ordered, allocates nothing and never
synchronises, so the whole step — compress fwd -> pinned-host wire ->
reconstruct fwd, compress bwd -> wire -> recover bwd, projection of W_o, the
wire on its own stream joined by events — is captured as it is (the chained
launches keep their programmatic dependencies as graph edges).  Each replay
gives the eager step's outputs bit for bit, replays pick up inputs changed in
place between them, and a bad id planted between replays is reported by the
error word like in an eager call (Sec. 4.3.1 ids, the error rule of the ABI)."""
import pytest
import torch

from paper_2506_01260_gb300 import workloads as W

pytestmark = pytest.mark.gpu


class Step:
    """The step's buffers and its launch sequence (the wire on its own stream)."""

    def __init__(self, sn, wl, wo_cols=1536):
        self.sn, self.n = sn, wl.seq_len
        wo_shape = (wl.d, wo_cols)
        self.inp = W.generate_on_device(wl, "cuda", grad=True)
        self.basis = sn.Basis(self.inp["U"])
        T, k = wl.T, wl.k
        g = torch.Generator(device="cuda").manual_seed(11)
        self.Wo = (0.02 * torch.randn(*wo_shape, generator=g, device="cuda")).to(torch.bfloat16)
        bf = dict(dtype=torch.bfloat16, device="cuda")
        self.out = {"C": torch.empty(T, k, **bf), "C_rx": torch.empty(T, k, **bf),
                    "Cg": torch.empty(T, k, **bf), "Cg_rx": torch.empty(T, k, **bf),
                    "Xr": torch.empty_like(self.inp["X"]), "Gr": torch.empty_like(self.inp["G"]),
                    "Wp": torch.empty_like(self.Wo)}
        self.ws = torch.empty(max(16, sn.sn_project_weight_workspace(self.basis, torch.bfloat16,
                                                                    wo_shape[1])),
                              dtype=torch.uint8, device="cuda")
        self.wire_f = torch.empty(T * k * 2, dtype=torch.uint8, pin_memory=True)
        self.wire_b = torch.empty(T * k * 2, dtype=torch.uint8, pin_memory=True)
        self.wire_stream = torch.cuda.Stream()
        self.ev = [torch.cuda.Event() for _ in range(4)]

    def poison(self):
        for t in self.out.values():
            t.view(torch.int16).fill_(0x7FBF)

    def run(self):
        sn, o, i, n = self.sn, self.out, self.inp, self.n
        s, ws = torch.cuda.current_stream(), self.wire_stream
        sn.sn_compress_fwd(self.basis, i["X"], i["ids"], i["tok_emb"], n, pos_emb=i["pos_emb"],
                           out=o["C"])
        self.ev[0].record(s)
        ws.wait_event(self.ev[0])
        sn.sn_wire_send(o["C"], self.wire_f, stream=ws)
        sn.sn_wire_recv(self.wire_f, o["C_rx"], stream=ws)
        self.ev[1].record(ws)
        sn.sn_compress_bwd(self.basis, i["G"], out=o["Cg"])
        self.ev[2].record(s)
        ws.wait_event(self.ev[2])
        sn.sn_wire_send(o["Cg"], self.wire_b, stream=ws)
        sn.sn_wire_recv(self.wire_b, o["Cg_rx"], stream=ws)
        self.ev[3].record(ws)
        sn.sn_project_weight(self.basis, self.Wo, out=o["Wp"], workspace=self.ws)
        s.wait_event(self.ev[1])
        sn.sn_decompress_fwd(self.basis, o["C_rx"], i["ids"], i["tok_emb"], n,
                             pos_emb=i["pos_emb"], out=o["Xr"])
        s.wait_event(self.ev[3])
        sn.sn_decompress_bwd(self.basis, o["Cg_rx"], out=o["Gr"])

    def snapshot(self):
        return {name: t.clone() for name, t in self.out.items()}


def _same(a, b):
    return torch.equal(a.view(torch.int16), b.view(torch.int16))


def _capture(step):
    graph = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        with torch.cuda.graph(graph, stream=side, capture_error_mode="thread_local"):
            step.run()
    torch.cuda.current_stream().wait_stream(side)
    return graph


@pytest.mark.parametrize("wname", ["1b", "8b"])
def test_step_graph_replays_eager_bits(sn, wname):
    step = Step(sn, W.WORKLOADS[wname])
    step.run()
    sn.sn_check_errors(step.basis)
    eager = step.snapshot()
    launches0 = sn.sn_launch_count()
    graph = _capture(step)
    captured = sn.sn_launch_count() - launches0
    assert captured >= 5                      # every call launched (recorded, not run)
    for _ in range(3):
        step.poison()
        graph.replay()
        sn.sn_check_errors(step.basis)
        for name, ref in eager.items():
            assert _same(step.out[name], ref), name
    step.basis.destroy()


def test_graph_replay_sees_inputs_changed_in_place(sn):
    step = Step(sn, W.WORKLOADS["1b"])
    graph = _capture(step)
    graph.replay()
    sn.sn_check_errors(step.basis)
    first = step.snapshot()
    # new activations and gradients in the captured buffers: the replay must
    # recompute, and match an eager step on the same inputs
    g = torch.Generator(device="cuda").manual_seed(3)
    step.inp["X"].copy_((step.inp["X"].float() +
                         0.01 * torch.randn(step.inp["X"].shape, generator=g,
                                            device="cuda")).to(torch.bfloat16))
    step.inp["G"].copy_(torch.randn(step.inp["G"].shape, generator=g,
                                    device="cuda").to(torch.bfloat16))
    graph.replay()
    sn.sn_check_errors(step.basis)
    replayed = step.snapshot()
    assert not _same(replayed["C"], first["C"]) and not _same(replayed["Gr"], first["Gr"])
    step.poison()
    step.run()
    sn.sn_check_errors(step.basis)
    for name, ref in step.snapshot().items():
        assert _same(replayed[name], ref), name
    step.basis.destroy()


def test_graph_replay_reports_bad_ids(sn):
    step = Step(sn, W.WORKLOADS["1b"])
    graph = _capture(step)
    ids = step.inp["ids"]
    vocab = step.inp["tok_emb"].shape[0]
    keep = ids[[5, 1000]].clone()
    ids[5] = vocab
    ids[1000] = -1
    step.poison()
    graph.replay()
    with pytest.raises(sn.SNError) as e:
        sn.sn_check_errors(step.basis)
    assert e.value.status == sn.SN_ERR_BAD_ID
    sn.sn_check_errors(step.basis)            # cleared
    for name in ("C", "Xr"):
        rows = step.out[name][[5, 1000]].float()
        assert torch.all(rows == 0), name
    # the backward half and the projection do not read ids
    ids[[5, 1000]] = keep
    graph.replay()
    sn.sn_check_errors(step.basis)
    step.basis.destroy()
