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


def _block_case(m, B, P, bl, seed, T=16):
    """GPU: prefill, refresh + one stale step on block 0; oracle: the last sequence."""
    import __graft_entry__ as g
    g.build()
    from paper_2609_37924_gb300 import TadmModel, upload_weights
    w = wl.Workload("fullsize", m, batch=B, prompt_len=P, gen_len=4 * bl, steps_per_block=T, K=4, block_len=bl,
                    seed=seed)
    host = wl.make_weights(m, seed=seed)
    tm = TadmModel(m, upload_weights(m, host), max_batch=B, max_rows=max(P, bl), max_ctx=P + 4 * bl)
    prompts = wl.make_prompts(w)
    z0 = np.full((B, bl), m.mask_id, np.int32)
    z1 = wl.random_canvas(w, B, bl, 0.6, seed=seed + 1)
    tm.tadm_reset(B)
    tm.tadm_prefill(torch.from_numpy(prompts).cuda())
    cache = tm.new_cache(B, bl)
    tm.tadm_anchor_forward(torch.from_numpy(z0).cuda(), T, cache)
    zt = torch.from_numpy(z1).cuda()
    logits = torch.empty((B * bl, m.vocab), dtype=torch.float32, device="cuda")
    conf = torch.empty(B * bl, dtype=torch.float32, device="cuda")
    tok = torch.empty(B * bl, dtype=torch.int32, device="cuda")
    tm.tadm_denoise_step(zt, T - 1, T, bl, cache, logits=logits, conf=conf, tok=tok)
    tm.tadm_sync_status()
    b = B - 1
    gl = logits[b * bl:(b + 1) * bl].cpu().numpy().astype(np.float64)
    gt = tok.cpu().numpy().reshape(B, bl)[b]
    gz = zt.cpu().numpy()[b]
    del tm, logits
    torch.cuda.empty_cache()
    o = O.Oracle(m, host)
    sess = o.new_session(1)
    o.prefill(sess, prompts[b:b + 1])
    cache_o = o.anchor_forward(sess, z0[b:b + 1])
    ref = o.denoise_step(sess, z1[b:b + 1], cache_o, 1, T, bl)
    rel = np.linalg.norm(gl - ref["logits"][0]) / np.linalg.norm(ref["logits"][0])
    masked = z1[b] == m.mask_id
    committed = masked & (gz != m.mask_id)
    agree = float(np.mean(gt[masked] == ref["tok"][0][masked]))
    return rel, agree, committed, gz, ref


def test_block_workload_full_size_sampled_sequence():
    """'block' workload dims and launch configuration: batch 32, d_model 2048,
    16 + 6 layers, GQA 16/8 heads of 128, vocab 128000, 512-token causal
    prefill, blocks of 32."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    w = wl.WORKLOADS["block"]
    rel, agree, committed, gz, ref = _block_case(w.model, w.batch, w.prompt_len, w.block_len, seed=w.seed)
    assert rel < 2e-2, rel
    assert np.array_equal(gz[committed], ref["tok"][0][committed])
    assert agree >= 0.9, agree
    print(f"[fullsize block] logits rel-L2 {rel:.3e}, argmax agreement {agree:.4f}, committed {committed.sum()}")


def test_posttrain_full_width_reduced_depth():
    """'posttrain' widths (d_model 5376, 32/16 heads of 128, FFN 21504 GeGLU,
    vocab 262144, tied head, paired-attention fusion r = 256) with 1 + 2 + 1
    layers and a 64-token prompt, batch 8."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    m = wl.get_workload("posttrain", model_n_shared=1, model_n_anchor=2, model_n_denoise=1).model
    rel, agree, committed, gz, ref = _block_case(m, 8, 64, 32, seed=3, T=32)
    assert rel < 2e-2, rel
    assert np.array_equal(gz[committed], ref["tok"][0][committed])
    assert agree >= 0.9, agree
    print(f"[fullsize posttrain] logits rel-L2 {rel:.3e}, argmax agreement {agree:.4f}, committed {committed.sum()}")


def test_posttrain_full_depth_one_sequence():
    """'posttrain' at its stated depth (S = embedding + 2 layers, A = 54, D =
    6; d_model 5376, vocab 262144, paired-attention fusion), batch 1, a
    32-token prompt: prefill, refresh and one stale step on the first block
    of 32, against the oracle (weights widened per use, so host memory holds
    only the bf16 model).

    On these random-init weights the logits error of any path with bf16
    tensor-core operands grows with depth past the 2e-2 bound:
    tests/bf16_floor.py --depth runs this very case with the oracle's
    arithmetic rounded to bf16 at every operand (the QKV input exact, as the
    split operand carries it) and stores its rel-L2
    (tests/golden/bf16_posttrain_depth62.json, 4.44e-2).  The GPU must meet
    the bound or sit within 10 % of that bf16 path's own error."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import json
    import os
    import time
    with open(os.path.join(os.path.dirname(__file__), "golden", "bf16_posttrain_depth62.json")) as f:
        gold = json.load(f)
    case = gold["case"]
    w = wl.WORKLOADS["posttrain"]
    m = w.model
    assert case["layers"] == [m.n_shared, m.n_anchor, m.n_denoise] and m.qkv_split
    t0 = time.time()
    rel, agree, committed, gz, ref = _block_case(m, case["batch"], case["prompt_len"], case["block_len"],
                                                 seed=case["seed"], T=case["T"])
    floor = gold["bf16_path_logits_rel_l2"]
    print(f"[fullsize posttrain depth 62] logits rel-L2 {rel:.3e} (bf16-operand path {floor:.3e}), "
          f"argmax agreement {agree:.4f}, committed {committed.sum()}, {time.time() - t0:.0f} s")
    assert rel < 2e-2 or rel <= 1.1 * floor, (rel, floor)
    assert np.array_equal(gz[committed], ref["tok"][0][committed])
