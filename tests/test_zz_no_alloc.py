"""The no-allocation variant of the fused output head + confidence.

Callers that cannot allocate device memory (a host framework that owns all
device allocations, or a latency-critical path that forbids cudaMalloc)
call tadm_head_confidence_static, which keeps its partials in a fixed array
inside the library.  It must give the results of tadm_head_confidence,
which takes caller scratch, on consecutive calls with different inputs.
This file is collected last on purpose.
"""
import numpy as np
import pytest

import workloads as wl

torch = pytest.importorskip("torch")


def _bf16(shape, seed, std):
    bits = wl.normal(seed, 97, int(np.prod(shape)), 0.0, std, "bf16").reshape(shape)
    return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).cuda()


@pytest.mark.gpu
def test_static_scratch_matches_caller_scratch_twice():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()
    from paper_2609_37924_gb300 import tadm
    for call, (rows, d, V, seed) in enumerate([(300, 768, 32768, 31), (129, 256, 5000, 32)]):
        x, w = _bf16((rows, d), seed, 1.0), _bf16((V, d), seed + 100, 0.05)
        conf_a = torch.empty(rows, dtype=torch.float32, device="cuda")
        tok_a = torch.empty(rows, dtype=torch.int32, device="cuda")
        scratch = torch.empty(tadm.tadm_head_scratch_size(rows, V, 1), dtype=torch.uint8, device="cuda")
        tadm.tadm_head_confidence(x, w, V - 1, conf_a, tok_a, scratch, 1)
        conf_b = torch.full((rows,), -1.0, dtype=torch.float32, device="cuda")
        tok_b = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
        tadm.tadm_head_confidence_static(x, w, V - 1, conf_b, tok_b, 1)
        torch.cuda.synchronize()
        assert np.array_equal(tok_a.cpu().numpy(), tok_b.cpu().numpy()), call
        ca, cb = conf_a.cpu().numpy(), conf_b.cpu().numpy()
        assert np.max(np.abs(cb - ca) / ca) < 4e-6, call
    # a request beyond the fixed array is refused before any work
    x, w = _bf16((8192, 64), 40, 1.0), _bf16((32768, 64), 41, 0.05)
    conf = torch.empty(8192, dtype=torch.float32, device="cuda")
    tok = torch.empty(8192, dtype=torch.int32, device="cuda")
    with pytest.raises(tadm.TadmError):
        tadm.tadm_head_confidence_static(x, w, 32767, conf, tok, 1)
