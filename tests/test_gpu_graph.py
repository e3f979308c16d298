"""Frozen layouts replayed as CUDA graphs (App. E "Cached metadata and
execution plans"): a decode step captured once (uc_append_next takes each
token's position from the device count) must give the eager step's results
on every later step, while the generated-token segment grows."""
import numpy as np
import pytest
import torch

import synth
from tests import _packed

pytestmark = pytest.mark.gpu
uc = pytest.importorskip("paper_2609_32831_gb300")
from paper_2609_32831_gb300.engine import CacheType, RequestCache  # noqa: E402

DEV = torch.device("cuda")


def _cache(L, B, n_text, n_img, gen):
    types = [CacheType("text", n_text, "full"), CacheType("vit", n_img, "evict_quant", keep_frac=0.5, bits=4)]
    return RequestCache(types, L, B, DEV, gen_capacity=gen)


def _inputs(L, B, N, steps, seed):
    K = torch.stack([synth.torch_kv(seed + l, B, 4, N, DEV)[0] for l in range(L)])
    V = torch.stack([synth.torch_kv(seed + l, B, 4, N, DEV)[1] for l in range(L)])
    Qw = torch.stack([synth.torch_q(seed + 50 + l, B, 28, 32, DEV) for l in range(L)])
    g = torch.Generator(device=DEV)
    g.manual_seed(seed)
    Qd = torch.randn((steps, L, B, 28, 1, 128), generator=g, device=DEV).to(torch.bfloat16)
    Kn = torch.randn((steps, L, B, 4, 128), generator=g, device=DEV).to(torch.bfloat16)
    Vn = torch.randn((steps, L, B, 4, 128), generator=g, device=DEV).to(torch.bfloat16)
    return K, V, Qw, Qd, Kn, Vn


def test_graphed_decode_matches_eager():
    L, B, n_text, n_img, steps = 2, 3, 200, 900, 40
    K, V, Qw, Qd, Kn, Vn = _inputs(L, B, n_text + n_img, steps, 31)
    eager, graphed = _cache(L, B, n_text, n_img, 64), _cache(L, B, n_text, n_img, 64)
    eager.prefill(K, V, Qw)
    graphed.prefill(K, V, Qw)
    graphed.capture_decode(want_lse=True)
    for t in range(steps):
        e_out = eager.decode_step(Qd[t], Kn[t], Vn[t])
        g_out = graphed.decode_step_graph(Qd[t], Kn[t], Vn[t])
        torch.cuda.synchronize()
        for l in range(L):
            err = _packed.attention_error(g_out[l].float().cpu().numpy(), e_out[l].double().cpu().numpy())
            assert err <= 1e-3, (t, l, err)
    graphed.sync_host_counts()
    for l in range(L):
        ge, gg = eager.gen[l], graphed.gen[l]
        assert list(gg.n_kept()) == [steps] * B
        assert torch.equal(ge.tensor("n_kept"), gg.tensor("n_kept"))
        # logical positions and stored rows of the generated tokens: identical
        assert torch.equal(ge.tensor("kept_idx").view(B, 4, -1)[:, :, :steps],
                           gg.tensor("kept_idx").view(B, 4, -1)[:, :, :steps])
        assert torch.equal(ge.tensor("k").view(B, 4, -1, 128)[:, :, :steps],
                           gg.tensor("k").view(B, 4, -1, 128)[:, :, :steps])


def test_prefill_with_a_new_layout_drops_the_graph():
    L, B = 1, 2
    K, V, Qw, Qd, Kn, Vn = _inputs(L, B, 1100, 2, 5)
    c = _cache(L, B, 200, 900, 16)
    c.prefill(K, V, Qw)
    c.capture_decode()
    c.decode_step_graph(Qd[0], Kn[0], Vn[0])
    c.prefill(K, V, Qw)          # same layout: the graph stays
    assert c.graph is not None
    c.types[1].keep_frac = 0.25  # new keep counts: the graph must go
    c.prefill(K, V, Qw)
    assert c.graph is None
    with pytest.raises(RuntimeError):
        c.decode_step_graph(Qd[1], Kn[1], Vn[1])


def test_alternating_input_buffers_reuse_their_captures():
    """Prefills from two input buffers (the text segment is a view, so its
    rows' address is part of the layout): each layout is captured once, and
    a later prefill from the first buffers replays the first capture, whose
    results again match the eager step."""
    L, B, n_text, n_img, steps = 2, 2, 200, 900, 3
    K, V, Qw, Qd, Kn, Vn = _inputs(L, B, n_text + n_img, steps, 41)
    K2, V2 = K.clone(), V.clone()
    c = _cache(L, B, n_text, n_img, 16)
    eager = _cache(L, B, n_text, n_img, 16)
    c.prefill(K, V, Qw)
    c.capture_decode()
    first = c.graphs[0]
    c.decode_step_graph(Qd[0], Kn[0], Vn[0])
    c.prefill(K2, V2, Qw)        # the views move: a new layout
    assert c.graph is None
    c.capture_decode()
    assert c.graphs[0] is not first
    c.decode_step_graph(Qd[0], Kn[0], Vn[0])
    c.prefill(K, V, Qw)          # back to the first buffers: the first capture again
    assert c.graph is first and len(c._captures) == 2
    eager.prefill(K, V, Qw)
    for t in range(steps):
        e_out = eager.decode_step(Qd[t], Kn[t], Vn[t])
        g_out = c.decode_step_graph(Qd[t], Kn[t], Vn[t])
        torch.cuda.synchronize()
        for l in range(L):
            err = _packed.attention_error(g_out[l].float().cpu().numpy(), e_out[l].double().cpu().numpy())
            assert err <= 1e-3, (t, l, err)
