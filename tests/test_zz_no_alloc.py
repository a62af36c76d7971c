"""The allocation-free projection entry point.

tda_project_materialized_noalloc serves callers that cannot allocate device
memory where they project gradients (for instance a plugin whose host program
owns all device memory, or a loop that must avoid cudaMalloc's implicit
synchronisation): its scratch is a fixed array inside libtda.so. This test
calls it through the C ABI twice in a row -- the second call on different
inputs, so the array holds the first call's leftovers -- and checks each result
against tda_project with route MATERIALIZE and a caller workspace, within the
tolerances the other parity tests use, and against the oracle; a third call
projects more examples than the array holds at once. It lives in its own
file, collected last, and passes alone in a fresh process as well as after the
other tests.
"""
import numpy as np
import pytest
import torch

import paper_2609_38767_gb300 as tda
from paper_2609_38767_gb300 import build as tbuild
from paper_2609_38767_gb300 import synth

pytestmark = pytest.mark.gpu

TOL = {"f32": 1e-5, "bf16": 2e-2}
TD = {"f32": tda.TDA_F32, "bf16": tda.TDA_BF16}


def _factors(n, T, d_in, d_out, dtype, stream, dev):
    A = synth.factors(synth.SEED_A, stream, n, T, d_in, 1.0, dtype=dtype, mask_p=0.02)
    B = synth.factors(synth.SEED_B, stream, n, T, d_out, 0.1, dtype=dtype, mask_p=0.02)
    if dtype == "bf16":
        return (torch.from_numpy(A.view(np.int16)).view(torch.bfloat16).to(dev),
                torch.from_numpy(B.view(np.int16)).view(torch.bfloat16).to(dev))
    return torch.from_numpy(A).to(dev), torch.from_numpy(B).to(dev)


def _rel(x, ref):
    x, ref = x.double().cpu(), ref.double().cpu()
    return float((x - ref).norm() / ref.norm())


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_noalloc_matches_workspace_route_on_consecutive_calls(dtype, orc):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    tbuild.build()
    dev = torch.device("cuda:0")
    # second call: other sizes; third: 20 examples of 4.3 MB of scratch each, more than the
    # 64 MiB array holds at once, so one call runs the route's chunk loop over the array twice
    shapes = [(6, 45, 256, 192, 32, 16), (4, 130, 512, 256, 16, 32), (20, 24, 1024, 1024, 32, 32)]
    for call, (N, T, di, do, ki, ko) in enumerate(shapes):
        L = tda.LayerDesc(di, do, T, ki, ko, seed=7, layer=call)
        if call == 2:
            assert N * 4 * (do * di + do * ki) > tda.tda_noalloc_scratch_bytes()
        Ah = synth.factors(synth.SEED_A, 20 + call, N, T, di, 1.0, dtype=dtype, mask_p=0.02)
        Bh = synth.factors(synth.SEED_B, 20 + call, N, T, do, 0.1, dtype=dtype, mask_p=0.02)
        A, B = _factors(N, T, di, do, dtype, 20 + call, dev)
        D = ki * ko
        got = torch.full((N, D), float("nan"), device=dev)
        tda.tda_project_materialized_noalloc(L, TD[dtype], A, B, N, got, D)
        wsb = tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, TD[dtype], N, 0, tda.TDA_ROUTE_MATERIALIZE)
        ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
        ref = torch.full((N, D), float("nan"), device=dev)
        tda.tda_project(L, TD[dtype], A, B, N, ref, D, tda.TDA_ROUTE_MATERIALIZE, ws, wsb)
        tda.tda_device_status()
        assert not torch.isnan(got).any()
        assert _rel(got, ref) <= TOL[dtype]
        # and against the oracle's fp64 projection of the same factor bits
        oref = orc.project(synth.to_f64(Ah, dtype), synth.to_f64(Bh, dtype), ki, ko, 7, call).reshape(N, D)
        assert _rel(got, torch.from_numpy(oref)) <= TOL[dtype]


def test_noalloc_rejects_layers_beyond_the_scratch():
    tbuild.build()
    big = tda.LayerDesc(8192, 8192, 16, 64, 64)  # 256 MiB of scratch per example
    assert 4 * (8192 * 8192 + 8192 * 64) > tda.tda_noalloc_scratch_bytes()
    with pytest.raises(tda.TdaError) as e:
        tda.tda_project_materialized_noalloc(big, tda.TDA_BF16, 256, 256, 1, 256, 4096, stream=0)
    assert e.value.status == tda.TDA_ERR_WORKSPACE
    assert "scratch" in str(e.value)
