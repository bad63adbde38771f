"""The C ABI without a GPU: the library loads, exports every declared entry
point, and its host-only logic (schedule plan, layer-cost formula, weight
inventory, argument validation) is right."""
import ctypes
import json
import os
import re

import pytest

import workloads as wl
from oracle import tadm_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__ as g
    g.build()
    from paper_2609_37924_gb300 import tadm
    return tadm


def declared_functions():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            names |= set(re.findall(r"^TADM_API\s+[\w\s\*]+?\b(tadm_\w+)\s*\(", src, flags=re.M))
    return names


def test_library_exports_every_declared_symbol(lib):
    so = lib.load_library()
    names = declared_functions()
    assert len(names) >= 20
    for n in sorted(names):
        assert hasattr(so, n), n
    assert set(lib.ABI_FUNCTIONS) == names


def test_plan_refresh_schedule(lib):
    for (P, G, T, K, bl) in [(32, 96, 32, 4, 0), (256, 768, 128, 1, 0), (512, 128, 16, 4, 32), (8, 64, 16, 3, 32)]:
        ev = lib.tadm_plan(P, G, T, K, bl)
        nblk = G // bl if bl else 1
        Gb = bl if bl else G
        refresh = [(b, n) for (kind, b, n, k) in ev if kind == 1]
        assert refresh == [(b, n) for b in range(nblk) for n in range(T) if n % K == 0]
        steps = [(b, n, k) for (kind, b, n, k) in ev if kind == 2]
        assert [(b, n) for b, n, _ in steps] == [(b, n) for b in range(nblk) for n in range(T)]
        for b in range(nblk):
            ks = [k for (bb, n, k) in steps if bb == b]
            assert ks == [O.unmask_count(n, T, Gb) for n in range(T)] and sum(ks) == Gb
        assert sum(1 for e in ev if e[0] == 0) == (1 if bl else 0)
        assert sum(1 for e in ev if e[0] == 3) == (nblk if bl else 0)
        # every refresh is immediately followed by the step it serves
        for i, e in enumerate(ev):
            if e[0] == 1:
                assert ev[i + 1][0] == 2 and ev[i + 1][1:3] == e[1:3]


def test_plan_rejects_bad_arguments(lib):
    for args in [(8, 60, 16, 4, 32), (8, 64, 0, 4, 0), (8, 64, 16, 0, 0), (8, 0, 16, 1, 0)]:
        with pytest.raises(lib.TadmError):
            lib.tadm_plan(*args)


def test_layer_cost_matches_paper_tables(lib):
    g = json.load(open(os.path.join(ROOT, "tests", "golden", "layer_cost.json")))
    for row in g["table1_ratio"]:
        full, cache = lib.tadm_layer_cost(row["L_S"], row["L_A"], row["L_D"], row["T"], row["K"])
        assert round(cache / full, 2) == row["ratio_2dp"]
    for row in g["table2_calls"]:
        assert lib.tadm_layer_cost(0, 12, 6, row["T"], row["K"])[1] == row["tadm"]
    for T in (1, 7, 48, 100):
        for K in (1, 2, 3, 5, 8):
            assert lib.tadm_layer_cost(2, 20, 8, T, K) == O.layer_cost(2, 20, 8, T, K)


@pytest.mark.parametrize("name", list(wl.WORKLOADS) + ["small+fusion_off"])
def test_weight_inventory_matches_the_generator(lib, name):
    if name.endswith("+fusion_off"):
        m = wl.ModelConfig(**{**wl.WORKLOADS[name.split("+")[0]].model.__dict__, "fusion": "none"})
    else:
        m = wl.WORKLOADS[name].model
    inv = lib.tadm_weight_inventory(lib.make_config(m))
    specs = wl.weight_specs(m)
    assert [n for n, _ in inv] == [s.name for s in specs]
    assert [tuple(s) for _, s in inv] == [s.shape for s in specs]


def test_invalid_configs_are_rejected(lib):
    so = lib.load_library()
    base = wl.WORKLOADS["small"].model
    for over in [dict(n_kv_heads=5), dict(vocab=1), dict(head_dim=0), dict(glu="x")]:
        try:
            m = wl.ModelConfig(**{**base.__dict__, **over})
            cfg = lib.make_config(m)
        except Exception:
            continue
        if over.get("glu"):
            cfg.glu = 7
        assert so.tadm_weight_count(ctypes.byref(cfg)) == -1
    cfg = lib.make_config(base)
    cfg.fusion = 3                                  # 0, 1, 2 are the only fusion modes
    assert so.tadm_weight_count(ctypes.byref(cfg)) == -1
    # Gemma-3 layer options: windows and patterns are non-negative, the norms are switches
    for field, bad in (("sliding_window", -1), ("global_every", -2), ("qk_norm", 2), ("sandwich_norm", -1),
                       ("rope_theta_global", -1.0)):
        cfg = lib.make_config(wl.POSTTRAIN_G3)
        assert so.tadm_weight_count(ctypes.byref(cfg)) > 0
        setattr(cfg, field, bad)
        assert so.tadm_weight_count(ctypes.byref(cfg)) == -1, field
    h = ctypes.c_void_p()
    cfg = lib.make_config(base)
    assert so.tadm_create(ctypes.byref(cfg), None, 0, 1, 1, 0, ctypes.byref(h)) == 1   # no weights
    assert not h.value


@pytest.mark.parametrize("kind,eta,T", [("cap", 0.04, 128), ("cap", 0.3, 7), ("loop", 0.02, 1024), ("loop", 0.02, 96)])
def test_remdm_schedule_matches_the_oracle_bit_exactly(lib, kind, eta, T):
    """The library's host schedule and the oracle's, written apart from the
    same readings, agree to the last bit at every step (the decisions u < sigma
    and u < p_unmask are then taken identically on both sides)."""
    for n in range(T):
        assert lib.tadm_remdm_schedule(kind, T, n, eta) == O.remdm_schedule(n, T, kind, eta)


def test_remdm_arguments_are_rejected(lib):
    so = lib.load_library()
    out = (ctypes.c_double * 4)()
    for args in [(0, 0, 0, 0.04, 0.55, 0.05, 0.9), (0, 8, 8, 0.04, 0.55, 0.05, 0.9), (2, 8, 0, 0.04, 0.55, 0.05, 0.9),
                 (0, 8, 0, -1.0, 0.55, 0.05, 0.9), (1, 8, 0, 0.02, 0.05, 0.55, 0.9), (1, 8, 0, 0.02, 0.55, 0.05, 1.0)]:
        assert so.tadm_remdm_schedule(*args, out) == 1, args
    # null buffers / out-of-range probabilities fail before any launch
    assert so.tadm_remdm_update(None, 4, None, 8, 1, 4, 0, 8, 7, 0.1, 0.1, 0.9, 1, 0, None, None) == 1


def test_entropy_bound_arguments_are_rejected(lib):
    """tadm_eb_update checks its arguments before any launch (the pointers
    below are never dereferenced)."""
    so = lib.load_library()
    fake = ctypes.c_void_p(256)
    good = dict(z=fake, ldz=8, logits=fake, ld=16, batch=2, rows=8, first=3, vocab=16, mask=15, tau=0.6, eta=0.1,
                last=0, seed=1, step=0, ent=fake, probs=None, pd=0, ldp=0)
    bad = [dict(z=None), dict(logits=None), dict(first=8), dict(first=-1), dict(ldz=7), dict(ld=15), dict(mask=16),
           dict(tau=0.0), dict(tau=-1.0), dict(eta=float("nan")), dict(last=2), dict(ent=None), dict(step=-1),
           dict(probs=fake, ldp=15), dict(probs=fake, ldp=16, pd=2), dict(rows=20000, ldz=20000, first=0)]
    for over in bad:
        a = {**good, **over}
        st = so.tadm_eb_update(a["z"], a["ldz"], a["logits"], a["ld"], a["batch"], a["rows"], a["first"], a["vocab"],
                               a["mask"], a["tau"], a["eta"], a["last"], a["seed"], a["step"], a["ent"], a["probs"],
                               a["pd"], a["ldp"], None, None)
        assert st == 1, over
    size = ctypes.c_size_t()
    assert so.tadm_eb_scratch_bytes(None, 1, 1, 1, ctypes.byref(size)) == 1


@pytest.mark.parametrize("name,batch,gen", [("posttrain_canvas", 8, 256), ("small", 16, 768), ("tiny", 1, 96)])
def test_entropy_bound_scratch_layout(lib, name, batch, gen):
    """tadm_eb_scratch_bytes follows the header's layout: 256-byte aligned
    segments of logits fp32 [n, V]; with self-conditioning q [n, V] and E^T
    [d, V] in the model's element type, q E fp32 [n, d] and Z fp32 [n]; H
    fp32 [n] (n = batch * gen_len).  The handle is host state only: it is
    created over placeholder (aligned, never dereferenced) weight pointers."""
    so = lib.load_library()
    m = wl.WORKLOADS[name].model
    cfg = lib.make_config(m)
    n_w = so.tadm_weight_count(ctypes.byref(cfg))
    ptrs = (ctypes.c_void_p * n_w)(*[256 * (i + 1) for i in range(n_w)])
    h = ctypes.c_void_p()
    assert so.tadm_create(ctypes.byref(cfg), ptrs, n_w, batch, 512 + gen, 0, ctypes.byref(h)) == 0
    try:
        al = lambda x: (x + 255) // 256 * 256  # noqa: E731
        n, V, d, es = batch * gen, m.vocab, m.d_model, 2 if m.dtype == "bf16" else 4
        want = {1: al(n * V * 4) + al(n * V * es) + al(d * V * es) + al(n * d * 4) + al(n * 4) + al(n * 4),
                0: al(n * V * 4) + al(n * 4)}
        for sc in (0, 1):
            got = ctypes.c_size_t()
            assert so.tadm_eb_scratch_bytes(h, batch, gen, sc, ctypes.byref(got)) == 0
            assert got.value == want[sc], (sc, got.value, want[sc])
        assert so.tadm_eb_scratch_bytes(h, 0, gen, 1, ctypes.byref(got)) == 1
    finally:
        so.tadm_destroy(h)


def test_sampler_generations_reject_bad_arguments_before_any_launch(lib):
    """tadm_generate_entropy_bound and tadm_generate_remdm refuse bad
    arguments on the host (status 1 and a message) on a host-only handle over
    placeholder pointers, which no accepted call could dereference here."""
    so = lib.load_library()
    m = wl.ModelConfig(vocab=4096, d_model=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=768, n_anchor=3,
                       n_denoise=2, dtype="bf16")
    cfg = lib.make_config(m)
    n_w = so.tadm_weight_count(ctypes.byref(cfg))
    ptrs = (ctypes.c_void_p * n_w)(*[256 * (i + 1) for i in range(n_w)])
    hs = {}
    for ctx in (0, 256):
        hs[ctx] = ctypes.c_void_p()
        assert so.tadm_create(ctypes.byref(cfg), ptrs, n_w, 2, 96, ctx, ctypes.byref(hs[ctx])) == 0
    try:
        P, G, fake = 16, 64, ctypes.c_void_p(1 << 20)
        need = ctypes.c_size_t()
        assert so.tadm_eb_scratch_bytes(hs[0], 2, G, 1, ctypes.byref(need)) == 0
        good = dict(h=hs[0], prompt=fake, batch=2, P=P, out=fake, G=G, steps=8, K=2, eta=0.1, tmax=0.8, tmin=0.4,
                    sc=1, seed=1, scratch=fake, nbytes=need.value)
        bad = [(dict(steps=0), "steps"), (dict(K=0), "K"), (dict(eta=float("nan")), "NaN"),
               (dict(tmin=0.0), "tau"), (dict(tmax=0.3), "tau"), (dict(sc=2), "self_cond"),
               (dict(prompt=None), "NULL"), (dict(scratch=None), "NULL"), (dict(G=0), "gen_len"),
               (dict(G=20000), "gen_len"), (dict(h=hs[256]), "single-block"),
               (dict(nbytes=need.value - 1), "scratch"), (dict(scratch=ctypes.c_void_p((1 << 20) + 128)), "aligned")]
        for over, word in bad:
            a = {**good, **over}
            st = so.tadm_generate_entropy_bound(a["h"], a["prompt"], a["batch"], a["P"], a["out"], a["G"], a["steps"],
                                                a["K"], a["eta"], a["tmax"], a["tmin"], a["sc"], a["seed"],
                                                a["scratch"], a["nbytes"], None)
            assert st == 1, over
            assert word in so.tadm_last_error(a["h"]).decode(), (over, so.tadm_last_error(a["h"]))
        # ReMDM: unknown schedule kind, top_p out of range, scratch too small, a KV-context handle
        for over in [dict(kind=2), dict(top_p=0.0), dict(top_p=1.5), dict(nbytes=16), dict(h=hs[256])]:
            a = {**dict(h=hs[0], kind=0, top_p=0.9, nbytes=2 * G * m.vocab * 4), **over}
            st = so.tadm_generate_remdm(a["h"], fake, 2, P, fake, G, 8, 2, a["kind"], 0.04, a["top_p"], 1, fake,
                                        a["nbytes"], None)
            assert st == 1, over
    finally:
        for h in hs.values():
            so.tadm_destroy(h)


def test_generate_refuses_bad_arguments_and_missing_workspace(lib):
    """tadm_generate's host checks on a host-only handle: a block length
    that does not divide the generation, K or steps < 1, block mode without
    a prompt or beyond the KV capacity, NULL buffers and a batch above the
    handle's are INVALID_ARG; valid arguments without a bound workspace are
    STATE; a misaligned or short workspace is refused before it is bound."""
    so = lib.load_library()
    m = wl.WORKLOADS["block"].model
    cfg = lib.make_config(m)
    n_w = so.tadm_weight_count(ctypes.byref(cfg))
    ptrs = (ctypes.c_void_p * n_w)(*[256 * (i + 1) for i in range(n_w)])
    h = ctypes.c_void_p()
    assert so.tadm_create(ctypes.byref(cfg), ptrs, n_w, 4, 512, 2048, ctypes.byref(h)) == 0
    try:
        fake = ctypes.c_void_p(1 << 20)
        good = dict(prompt=fake, batch=4, P=512, out=fake, G=1536, T=16, K=4, bl=32)
        for over in [dict(bl=40), dict(K=0), dict(T=0), dict(G=0), dict(P=0), dict(G=2048), dict(prompt=None),
                     dict(out=None), dict(batch=5), dict(batch=0)]:
            a = {**good, **over}
            st = so.tadm_generate(h, a["prompt"], a["batch"], a["P"], a["out"], a["G"], a["T"], a["K"], a["bl"], None)
            assert st == 1, (over, so.tadm_last_error(h))
        st = so.tadm_generate(h, fake, 4, 512, fake, 1536, 16, 4, 32, None)
        assert st == 6 and b"workspace" in so.tadm_last_error(h)
        need = ctypes.c_size_t()
        assert so.tadm_workspace_size(h, ctypes.byref(need)) == 0 and need.value > 0
        assert so.tadm_bind_workspace(h, ctypes.c_void_p((1 << 20) + 16), need.value) == 1
        assert so.tadm_bind_workspace(h, fake, need.value - 1) == 4
    finally:
        so.tadm_destroy(h)
