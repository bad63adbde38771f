"""Full-size parity in the launch configuration bench.py times: the 'small'
workload (batch 16, 1024-position canvas, d_model 768, 8 + 4 layers, vocab
32768, bf16), one refresh and one stale denoising step on the GPU for the
whole batch; the oracle recomputes one sequence and the sampled outputs are
compared."""
import numpy as np
import pytest

import workloads as wl
from oracle import tadm_oracle as O

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def test_small_workload_sampled_sequence(request):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()
    from paper_2609_37924_gb300 import TadmModel, upload_weights
    w = wl.WORKLOADS["small"]
    m, B, R = w.model, w.batch, w.total_len
    host = wl.make_weights(m, seed=w.seed)
    tm = TadmModel(m, upload_weights(m, host), max_batch=B, max_rows=R)
    z0 = wl.random_canvas(w, B, R, 0.9, seed=21, start=w.prompt_len)
    z1 = wl.random_canvas(w, B, R, 0.7, seed=22, start=w.prompt_len)
    cache = tm.new_cache(B, R)
    tm.tadm_reset(B)
    tm.tadm_anchor_forward(torch.from_numpy(z0).cuda(), 128, cache)
    zt = torch.from_numpy(z1).cuda()
    logits = torch.empty((B * R, m.vocab), dtype=torch.float32, device="cuda")
    conf = torch.empty(B * R, dtype=torch.float32, device="cuda")
    tok = torch.empty(B * R, dtype=torch.int32, device="cuda")
    sel = torch.empty((B, 6), dtype=torch.int32, device="cuda")
    tm.tadm_denoise_step(zt, 125, 128, w.gen_len, cache, logits=logits, conf=conf, tok=tok, selected=sel)
    tm.tadm_sync_status()
    b = B - 1                                          # the last sequence: exercises every batch offset
    gl = logits[b * R:(b + 1) * R].cpu().numpy().astype(np.float64)
    gc = conf.cpu().numpy().reshape(B, R)[b]
    gt = tok.cpu().numpy().reshape(B, R)[b]
    gz = zt.cpu().numpy()[b]
    o = O.Oracle(m, host)
    sess = o.new_session(1)
    cache_o = o.anchor_forward(sess, z0[b:b + 1])
    ref = o.denoise_step(sess, z1[b:b + 1], cache_o, 3, 128, w.gen_len)
    rel = np.linalg.norm(gl - ref["logits"][0]) / np.linalg.norm(ref["logits"][0])
    assert rel < 2e-2, rel
    c2, t2 = O.confidence(gl, m.mask_id)
    assert np.array_equal(gt, t2) and np.max(np.abs(gc - c2) / c2) < 4e-6
    p = O.select_topk(z1[b], gc.astype(np.float64), 6, m.mask_id)
    assert list(sel.cpu().numpy()[b]) == list(p)
    masked = z1[b] == m.mask_id
    committed = masked & (gz != m.mask_id)
    assert committed.sum() == 6 and np.array_equal(gz[committed], ref["tok"][0][committed])
    agree = float(np.mean(gt[masked] == ref["tok"][0][masked]))
    assert agree >= 0.95, agree
    print(f"[fullsize small] logits rel-L2 {rel:.3e}, argmax agreement {agree:.4f}, committed 6/6")
