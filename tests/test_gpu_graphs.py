"""A whole GRPO step (group advantages, forward scoring, loss + backward) captured in a CUDA graph
and replayed: the library allocates nothing and never synchronises on this path, so the step can
be captured; replays give bitwise the eager results, also after the inputs change in place."""
import pytest
import torch

from paper_2510_17158_gb300 import grpo as G
from paper_2510_17158_gb300.synthetic import WORKLOADS, make_batch_numpy
from tests.parity_util import oracle_inputs

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,over", [
    ("tiny_f32", {}),
    ("g8_t1k_d2048_v32k", dict(prompts=1, group_sizes=(4,), T=200, len_lo=50, len_hi=200)),
])
def test_step_captured_in_cuda_graph_matches_eager(name, over):
    b = make_batch_numpy(WORKLOADS[name].scaled(**over))
    w = b.workload
    H, W, tok, mask = (t.cuda() for t in (b.H, b.W, b.tokens, b.mask))
    rew, go = b.rewards.cuda(), b.group_offsets.cuda()
    S, T, d = H.shape
    V = W.shape[0]
    old_np, ref_np = oracle_inputs(b)
    old, ref = torch.from_numpy(old_np).cuda(), torch.from_numpy(ref_np).cuda()
    ws = G.Workspace.for_problem(S, T, d, V, H.dtype)
    adv = torch.empty(S, device="cuda")
    fwd = {"logp": torch.empty((S, T), device="cuda"), "lse": torch.empty((S, T), device="cuda"),
           "entropy": torch.empty((S, T), device="cuda"),
           "argmax": torch.empty((S, T), dtype=torch.int32, device="cuda"),
           "valid_count": torch.empty((S,), dtype=torch.int32, device="cuda")}
    bwd = {"loss": torch.empty(1, device="cuda"), "dH": torch.empty_like(H),
           "dW": torch.empty((V, d), device="cuda")}

    def step():
        G.group_advantages(rew, go, ws, adv_out=adv)
        G.grpo_score_fwd(H, W, tok, mask, ws, out=fwd)
        G.grpo_loss_bwd(H, W, tok, mask, fwd["logp"], fwd["lse"], old, ref, adv,
                        fwd["valid_count"], ws, eps_low=w.eps, eps_high=w.eps, beta=w.beta,
                        out=bwd)

    def snapshot():
        return {k: v.clone() for k, v in list(fwd.items()) + list(bwd.items())}

    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        step()                                    # eager, on the capture stream
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    eager = snapshot()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    for _ in range(2):
        for v in list(fwd.values()) + list(bwd.values()):
            v.zero_()
        graph.replay()
        torch.cuda.synchronize()
        got = snapshot()
        for k in eager:
            assert torch.equal(got[k], eager[k]), k
    assert G.grpo_last_device_error(ws)[0] == 0

    # new inputs written in place are picked up by the replay
    H.mul_(0.5)
    with torch.cuda.stream(s):
        step()
    torch.cuda.synchronize()
    eager2 = snapshot()
    graph.replay()
    torch.cuda.synchronize()
    got2 = snapshot()
    for k in eager2:
        assert torch.equal(got2[k], eager2[k]), k
    assert not torch.equal(eager2["logp"], eager["logp"])
