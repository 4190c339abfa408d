"""xpress_accept_noalloc: acceptance without any device allocation.

Callers that cannot allocate device memory (for instance code that runs
while another thread captures a CUDA graph, or behind an allocator that
forbids device allocations after start-up) use xpress_accept_noalloc, which
keeps its scratch in a fixed array inside the library.  This test checks, on
two calls in a row through the C ABI, that its accept lengths and emitted
tokens equal those of xpress_accept on the same inputs (integer outputs, so
the comparison is exact), for a greedy and a sampling batch: first two calls
each followed by a synchronisation, then two calls issued back to back on
one stream with no synchronisation between them (the stream orders them on
the shared array).  It passes when run alone in a fresh process (the first
call then does the one-time address lookup) and after the other tests.
"""
import numpy as np
import pytest

from paper_2608_02438_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def X():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_02438_gb300 import binding, build
    build.build()
    binding.load()
    return binding


def _setup(X, temps, seed):
    cfg = W.tiny_config("noalloc", b=6, B=8, H=128, V=2080, r=256, dtype=W.BF16, temps=temps, seed=seed,
                        logits="gauss4_spike", draft="sample")
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, seed + 1, "strong")
    inp = W.make_inputs(cfg)
    ref = X.Refiner({k: X.to_device(v, X.XPRESS_BF16) for k, v in w.items()}, cfg.H, cfg.V, cfg.r, cfg.B,
                    X.XPRESS_BF16)
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    d = dict(h=X.to_device(inp["h"], X.XPRESS_BF16), s=X.to_device(inp["s"], X.XPRESS_BF16),
             target=X.to_device(inp["target"], X.XPRESS_BF16), draft=dev(inp["draft"]), anchor=dev(inp["anchor"]),
             temperature=dev(inp["temperature"]), seed=dev(inp["seed"].view(np.int64)))
    out = ref.refine_block(d["h"], d["s"], d["draft"], d["anchor"], d["temperature"], d["seed"], inp["offset"],
                           cfg.K_max)
    return cfg, inp, ref, d, out


def _accept_in(X, cfg, inp, d, out):
    return X.XpressAcceptIn(cfg.b, d["target"].data_ptr(), d["s"].data_ptr(), out["tokens"].data_ptr(),
                            out["lse"].data_ptr(), out["logit_sel"].data_ptr(), out["z_final"].data_ptr(),
                            d["temperature"].data_ptr(), d["seed"].data_ptr(), inp["offset"])


def test_noalloc_accept_matches_workspace_accept_on_two_calls(X):
    for temps, seed in (((1.0, 0.0), 71), ((0.0,), 73)):
        cfg, inp, ref, d, out = _setup(X, temps, seed)
        want = ref.accept(d["target"], d["s"], out["tokens"], out["lse"], out["logit_sel"], out["z_final"],
                          d["temperature"], d["seed"], inp["offset"])
        torch.cuda.synchronize()
        want = {k: v.cpu().numpy().copy() for k, v in want.items()}
        for sync_between in (True, False):
            outs = []
            for call in range(2):
                alen = torch.full((cfg.b,), -7, dtype=torch.int32, device="cuda")
                otok = torch.full((cfg.b, cfg.B + 1), -7, dtype=torch.int32, device="cuda")
                X.xpress_accept_noalloc(ref.handle, _accept_in(X, cfg, inp, d, out), alen.data_ptr(),
                                        otok.data_ptr(), ref.stream.cuda_stream)
                if sync_between:
                    torch.cuda.synchronize()
                outs.append((alen, otok))
            torch.cuda.synchronize()
            for call, (alen, otok) in enumerate(outs):
                tag = f"call {call}, {'synchronised' if sync_between else 'back to back'}"
                np.testing.assert_array_equal(alen.cpu().numpy(), want["accept_len"], err_msg=tag)
                np.testing.assert_array_equal(otok.cpu().numpy(), want["out_tokens"], err_msg=tag)
        ref.close()


def test_noalloc_accept_replayed_from_a_cuda_graph(X):
    # the entry point exists for stream capture: one call captured (after a
    # warm-up call that caches the scratch address), then replayed twice
    cfg, inp, ref, d, out = _setup(X, (1.0, 0.0), 83)
    want = ref.accept(d["target"], d["s"], out["tokens"], out["lse"], out["logit_sel"], out["z_final"],
                      d["temperature"], d["seed"], inp["offset"])
    torch.cuda.synchronize()
    want = {k: v.cpu().numpy().copy() for k, v in want.items()}
    alen = torch.full((cfg.b,), -7, dtype=torch.int32, device="cuda")
    otok = torch.full((cfg.b, cfg.B + 1), -7, dtype=torch.int32, device="cuda")
    acc_in = _accept_in(X, cfg, inp, d, out)
    X.xpress_accept_noalloc(ref.handle, acc_in, alen.data_ptr(), otok.data_ptr(), ref.stream.cuda_stream)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):                 # captured on torch's side stream
        X.xpress_accept_noalloc(ref.handle, acc_in, alen.data_ptr(), otok.data_ptr(),
                                torch.cuda.current_stream().cuda_stream)
    for replay in range(2):
        alen.fill_(-7)
        otok.fill_(-7)
        torch.cuda.synchronize()
        graph.replay()
        torch.cuda.synchronize()
        np.testing.assert_array_equal(alen.cpu().numpy(), want["accept_len"], err_msg=f"replay {replay}")
        np.testing.assert_array_equal(otok.cpu().numpy(), want["out_tokens"], err_msg=f"replay {replay}")
    del graph
    ref.close()


def test_noalloc_rejects_a_batch_beyond_its_scratch(X):
    cfg = W.tiny_config("noalloc_big", b=1, B=32, H=64, V=64, r=256, dtype=W.BF16, seed=79)
    w = W.make_weights(cfg.H, cfg.V, cfg.r, cfg.B, cfg.dtype, 80, "paper")
    ref = X.Refiner({k: X.to_device(v, X.XPRESS_BF16) for k, v in w.items()}, cfg.H, cfg.V, cfg.r, cfg.B,
                    X.XPRESS_BF16)
    b = 4096                                   # 4096 * 33 target rows: beyond the fixed scratch
    acc_in = X.XpressAcceptIn(b, 16, 16, 16, 16, 16, 16, 16, 16, 0)   # never dereferenced
    with pytest.raises(X.XpressError) as err:
        X.xpress_accept_noalloc(ref.handle, acc_in, 16, 16, ref.stream.cuda_stream)
    assert err.value.code == X.XPRESS_ERR_UNSUPPORTED
    ref.close()
