"""The no-allocation variant of the fused output head + confidence.

Callers that cannot allocate device memory (a host framework that owns all
device allocations, or a latency-critical path that forbids cudaMalloc)
call tadm_head_confidence_static, which keeps its partials in a fixed array
inside the library.  It must give exactly the results of
tadm_head_confidence, which takes caller scratch and runs the same kernels,
on consecutive calls with different inputs: bf16 and fp32 models, and a
vocabulary whose last 128-column half tile holds no column (a partial that
a call failed to write would surface as a stale value from the call
before).  This file is collected last on purpose.
"""
import numpy as np
import pytest

import workloads as wl

torch = pytest.importorskip("torch")


def _mat(shape, seed, std, dtype):
    n = int(np.prod(shape))
    if dtype == 1:
        bits = wl.normal(seed, 97, n, 0.0, std, "bf16").reshape(shape)
        return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).cuda()
    return torch.from_numpy(wl.normal(seed, 97, n, 0.0, std, "f32").reshape(shape)).cuda()


@pytest.mark.gpu
def test_static_scratch_matches_caller_scratch_twice():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()
    from paper_2609_37924_gb300 import tadm
    # (rows, d, V, seed, dtype): V = 4900 leaves the second half of its last 256-column tile empty
    cases = [(300, 768, 32768, 31, 1), (129, 256, 4900, 32, 1), (77, 128, 3000, 33, 0), (300, 768, 32768, 34, 1)]
    for call, (rows, d, V, seed, dt) in enumerate(cases):
        x, w = _mat((rows, d), seed, 1.0, dt), _mat((V, d), seed + 100, 0.05, dt)
        conf_a = torch.empty(rows, dtype=torch.float32, device="cuda")
        tok_a = torch.empty(rows, dtype=torch.int32, device="cuda")
        scratch = torch.empty(tadm.tadm_head_scratch_size(rows, V, dt), dtype=torch.uint8, device="cuda")
        tadm.tadm_head_confidence(x, w, V - 1, conf_a, tok_a, scratch, dt)
        conf_b = torch.full((rows,), -1.0, dtype=torch.float32, device="cuda")
        tok_b = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
        tadm.tadm_head_confidence_static(x, w, V - 1, conf_b, tok_b, dt)
        torch.cuda.synchronize()
        assert np.array_equal(tok_a.cpu().numpy(), tok_b.cpu().numpy()), call
        assert np.array_equal(conf_a.cpu().numpy(), conf_b.cpu().numpy()), call
        assert bool((tok_b >= 0).all()) and bool((tok_b < V - 1).all()), call
    # a request beyond the fixed array is refused before any work
    x, w = _mat((8192, 64), 40, 1.0, 1), _mat((32768, 64), 41, 0.05, 1)
    conf = torch.empty(8192, dtype=torch.float32, device="cuda")
    tok = torch.empty(8192, dtype=torch.int32, device="cuda")
    with pytest.raises(tadm.TadmError):
        tadm.tadm_head_confidence_static(x, w, 32767, conf, tok, 1)
