"""rpd_step captured into a CUDA graph: with scratch reserved beforehand the step enqueues no
allocation and no host synchronisation, so it can be captured once and replayed; replays
give the same outputs as eager steps, with one projection pass or two (lazy, or chosen on
the device inside the replay)."""
import pytest
import torch

import workloads as WL

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # collected on CPU machines, never run there
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2609_36452_gb300 as rpd  # noqa: E402


@pytest.mark.parametrize("projection", ["all", "lazy", "auto"])
def test_step_replays_from_cuda_graph(projection):
    dev = torch.device("cuda:0")
    K, N, d, V = 4, 256, 1024, 8192
    W, g = WL.make_head(V, d, 21, w_std=0.08)
    cv = WL.make_hidden(W, K, N, 22, WL.u_profile(N, 0.5, 3.0),
                        WL.calibrated_sigma(V, d, 0.08, 3.0), flip_frac=0.1)
    W, g, hidden = W.to(dev), g.to(dev), cv.hidden.to(dev)
    ctx = rpd.Rpd(d, V, K)
    ctx.set_head(W, g)
    ctx.set_profile("llada")
    ctx.set_projection(projection)
    ctx.reserve(1, N)
    mask0 = torch.ones(N, dtype=torch.uint8, device=dev)

    def outputs():
        return (mask0.clone(), torch.zeros(N, dtype=torch.uint8, device=dev),
                torch.full((N,), -1, dtype=torch.int32, device=dev),
                torch.zeros(rpd.STATS_WORDS, dtype=torch.int32, device=dev))

    # eager reference (also configures the kernels before capture)
    ctx.set_stream(torch.cuda.current_stream(dev))
    m_e, c_e, t_e, s_e = outputs()
    ctx.step(hidden, m_e, 0.9, 1.0, c_e, t_e, s_e)
    torch.cuda.synchronize(dev)

    m_g, c_g, t_g, s_g = outputs()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        ctx.set_stream(torch.cuda.current_stream(dev))
        ctx.step(hidden, m_g, 0.9, 1.0, c_g, t_g, s_g)
    ctx.set_stream(torch.cuda.current_stream(dev))
    for _ in range(3):
        m_g.copy_(mask0)
        c_g.zero_()
        t_g.fill_(-1)
        graph.replay()
        torch.cuda.synchronize(dev)
        assert torch.equal(c_g, c_e) and torch.equal(m_g, m_e)
        assert torch.equal(t_g, t_e) and torch.equal(s_g, s_e)
    assert int(s_g[4]) >= 1 and int(s_g[7]) == 0
    ctx.close()
