"""Several occam_prune calls in flight at once, as a serving loop runs them:
each call with its own inputs, workspace and outputs on its own stream, the
calls replayed interleaved without synchronizing. Every call's results must
be bit-identical to the same call run alone, and the first of them must
agree with the oracle (the parity rule of tests/gpu_helpers.check_prune).

The three calls take different routes through Stage II ([CLS] Stage I with
4- and 8-CTA clusters; mutual Stage I; samples above the fused kernel's S1
limit on the two-pass path), so their launches overlap on the GPU in every
combination the library's streams allow."""

from __future__ import annotations

import pytest
import torch

from synth import tiny_batch
from tests.gpu_helpers import check_prune, to_device

pytestmark = pytest.mark.gpu

H = dict(H1=16, d1=64, H2=32, d2=128, hidden=256, beta1=2.0, sinks=("count", 1))

CALLS = [
    # (tiny_batch kwargs, lambda1, lambda2)
    (dict(B=3, segs=2, P=(500, 120, 380), R=4, M=(40, 200, 7), seed=71), 0.2, 1.1),
    (dict(B=2, segs=1, P=(900, 300), R=4, M=(150, 60), stage1="mutual", d1=72, query_bias=0.5, seed=72), 0.3, 1.2),
    (dict(B=2, segs=1, P=(3300, 200), R=3, M=(90, 30), seed=73), 0.0, 1.1),
]


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available()


def _call(b, lam1, lam2):
    import paper_2605_29657_gb300 as occ
    d = to_device(b, "cuda")
    layout = occ.BatchLayout.from_batch(b, "cuda")
    if "Q1" in d:
        st1 = dict(mode="mutual", q=d["Q1"], K1=d["K1"])
    else:
        st1 = dict(mode="cls", q=d["q_cls"], k_cls=d["k_cls"], K1=d["K1"])
    call = occ.PruneCall(layout, st1, dict(Q_text=d["Q_text"], K_text=d["K_text"], K2=d["K2"]), lam1, lam2,
                         gather=(d["hidden"], d["K2"].view(d["K2"].shape[0], -1), d["V"]))
    return call


def _snapshot(call):
    out = {k: v.clone() for k, v in call.out.items()}
    out["gathered"] = [t.clone() for t in call.gathered]
    return out


def _same(a, b):
    kept = int(a["out_off"][-1].item())
    for k, v in a.items():
        if k == "gathered":
            for x, y in zip(v, b[k]):
                assert torch.equal(x[:kept], y[:kept]), "gathered rows"
        elif k == "out_index":
            assert torch.equal(v[:kept], b[k][:kept]), k
        else:
            assert torch.equal(v, b[k]), k


@pytest.mark.parametrize("graphs", [False, True], ids=["eager", "graphs"])
def test_calls_in_flight_match_calls_alone(graphs):
    batches = [(tiny_batch(**{**H, **kw}), l1, l2) for kw, l1, l2 in CALLS]
    calls = [_call(b, l1, l2) for b, l1, l2 in batches]
    # each call alone, on the current stream
    alone = []
    for c in calls:
        c()
        torch.cuda.synchronize()
        assert c.status() == 0
        alone.append(_snapshot(c))
    # the first call's results against the oracle (the others are covered by
    # the parity tests of their routes)
    b0, l1, l2 = batches[0]
    gpu0 = {k: v.cpu().numpy() for k, v in calls[0].out.items()}
    gpu0["gathered"] = [t.cpu() for t in calls[0].gathered]
    gpu0["status"] = calls[0].status()
    check_prune(b0, gpu0, l1, l2)

    streams = [torch.cuda.Stream() for _ in calls]
    runners = []
    if graphs:
        for c in calls:
            cap = torch.cuda.Stream()
            cap.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(cap):
                c(cap)  # a warm call on a side stream before capture
            torch.cuda.current_stream().wait_stream(cap)
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                c()
            runners.append(lambda s, g=g: g.replay())
    else:
        runners = [lambda s, c=c: c(s) for c in calls]
    # interleaved, no synchronization between calls: a call's next run on its
    # own stream follows its previous one; calls on different streams overlap
    for s in streams:
        s.wait_stream(torch.cuda.current_stream())
    for i in range(15):
        j = i % len(calls)
        with torch.cuda.stream(streams[j]):
            runners[j](streams[j])
    for s in streams:
        torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    for c, want in zip(calls, alone):
        assert c.status() == 0
        _same(want, _snapshot(c))
