"""CPU checks of the C-ABI library: it loads, exports every declared symbol, and its
host mask compiler matches the oracle's bit for bit (no GPU work)."""
import ctypes
import dataclasses
import os
import re

import numpy as np
import pytest

import synth
from oracle import ledger, maskc

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_29499_gb300 import build
    build.build()
    from paper_2609_29499_gb300 import tasp
    return tasp


def _declared_symbols():
    src = open(os.path.join(ROOT, "include", "tasp.h")).read()
    return sorted(set(re.findall(r"^\s*(?:int|const char\*)\s+(tasp_\w+)\s*\(", src, re.M)))


def test_exports_every_declared_symbol(lib):
    names = _declared_symbols()
    assert len(names) >= 15
    so = ctypes.CDLL(lib.LIB_PATH)
    for n in names:
        assert hasattr(so, n), n
    assert set(names) == set(lib.EXPORTED)
    assert "sm_103a" in lib.version()


CASES = [(synth.LAYER1, (1000, 1001, 77)), (synth.LLAMA3_8B, synth.MASK_SEEDS), (synth.LLAMA3_70B, synth.MASK_SEEDS),
         (synth.tiny_shape(L=7), (3, 4, 5))]


@pytest.mark.parametrize("shape,seeds", CASES)
def test_host_mask_compiler_matches_oracle(lib, shape, seeds):
    for seed in seeds:
        sc = synth.mask_scores_u32(seed, shape.L, shape.n_units)
        tg = synth.layer_target_u24(seed, shape.L)
        want = maskc.compile_mask(shape, sc, tg, 0.57, 0.35, 0.85)
        groups, units, fl = lib.mask_select(shape, lib.greedy_mask(sc, tg, 0.57, 0.35, 0.85))
        assert groups == want.keep_groups
        assert units == want.keep_units
        assert fl[:shape.L].tolist() == want.info["layer_flops"]
        assert fl[shape.L] == want.info["total_flops"]
        assert fl[shape.L + 1] == want.info["budget_flops"]
        assert fl[shape.L + 2] == shape.L * ledger.dense_layer_flops(shape)


def test_other_budgets_match_oracle(lib):
    sh = synth.LLAMA3_8B
    for budget, lo, hi in ((0.3, 0.2, 0.5), (0.7, 0.5, 0.9), (0.57, 0.57, 0.57)):
        sc = synth.mask_scores_u32(9, sh.L, sh.n_units)
        tg = synth.layer_target_u24(9, sh.L)
        want = maskc.compile_mask(sh, sc, tg, budget, lo, hi)
        groups, units, _ = lib.mask_select(sh, lib.greedy_mask(sc, tg, budget, lo, hi))
        assert groups == want.keep_groups and units == want.keep_units


def test_explicit_and_all_keep(lib):
    sh = synth.tiny_shape(L=2)
    g = [[0], [1]]
    u = [[0, 3, 5], [2]]
    groups, units, fl = lib.mask_select(sh, lib.explicit_mask(g, u))
    assert groups == g and units == u
    m = maskc.explicit(sh, g, u)
    assert fl[sh.L] == ledger.mask_flops(sh, m.keep_groups, m.keep_chans)
    groups, units, fl = lib.mask_select(sh, lib.all_keep_mask())
    assert groups == [list(range(sh.Hkv))] * sh.L
    assert fl[sh.L] == fl[sh.L + 2]


def test_invalid_requests_are_rejected(lib):
    sh = synth.tiny_shape(L=2)
    with pytest.raises(lib.TaspError) as e:
        lib.mask_select(sh, lib.explicit_mask([[1, 0], [0]], [[0], [0]]))  # not ascending
    assert e.value.code == lib.EINVAL
    with pytest.raises(lib.TaspError) as e:
        lib.mask_select(sh, lib.explicit_mask([[0], [5]], [[0], [0]]))  # group out of range
    assert e.value.code == lib.EINVAL
    sc = synth.mask_scores_u32(1, sh.L, sh.n_units)
    with pytest.raises(lib.TaspError) as e:
        lib.mask_select(sh, lib.greedy_mask(sc, synth.layer_target_u24(1, sh.L), budget=1.5))
    assert e.value.code == lib.EINVAL
    bad = synth.tiny_shape(d=100)  # d not a multiple of 16
    with pytest.raises(lib.TaspError) as e:
        lib.mask_select(bad, lib.all_keep_mask())
    assert e.value.code == lib.EINVAL
    assert "multiples of 16" in str(e.value)


def test_union_step_argument_checks_need_no_gpu(lib):
    # the union entry rejects a null session list, a null input and a session count outside
    # 1..16 before it touches a session or the device
    so = lib.load()
    P = ctypes.c_void_p
    arr = (P * 17)()
    x = ctypes.c_void_p(16)  # never dereferenced: the count is rejected first
    assert so.tasp_decode_step_union(None, 1, x, None, None, None) == lib.EINVAL
    assert so.tasp_decode_step_union(arr, 1, None, None, None, None) == lib.EINVAL
    for n in (0, 17, -1):
        assert so.tasp_decode_step_union(arr, n, x, None, None, None) == lib.EINVAL
    assert "16 sessions" in so.tasp_last_error().decode()
    assert so.tasp_union_status(None, 1, None, None) == lib.EINVAL


# ---------------------------------------------------------------------------
# Query-head candidates (Sec. 3.3, Table 1): the library's heap-based greedy against the
# oracle's plain rescans, bit for bit.
# ---------------------------------------------------------------------------

QHEAD_CASES = [(synth.LAYER1, (1000, 1001)), (synth.LLAMA3_8B, synth.MASK_SEEDS), (synth.LLAMA3_70B, (1000, 1004)),
               (synth.tiny_shape(L=7), (3, 4, 5)),
               (synth.ModelShape(L=5, d=128, Hq=8, Hkv=2, dh=32, df=256, vocab=0, chan_unit=16), (21, 22))]


@pytest.mark.parametrize("shape,seeds", QHEAD_CASES)
def test_host_qhead_compiler_matches_oracle(lib, shape, seeds):
    for seed in seeds:
        for budget, lo, hi in ((0.57, 0.35, 0.85), (0.3, 0.2, 0.5)):
            sc = synth.mask_scores_u32(seed, shape.L, shape.Hq + shape.n_chan_units)
            tg = synth.layer_target_u24(seed, shape.L)
            want = maskc.compile_mask_qheads(shape, sc, tg, budget, lo, hi)
            qh, groups, units, fl = lib.mask_select_qheads(shape, lib.greedy_qhead_mask(sc, tg, budget, lo, hi))
            assert qh == want.keep_qheads
            assert groups == want.keep_groups
            assert units == want.keep_units
            assert fl[:shape.L].tolist() == want.info["layer_flops"]
            assert fl[shape.L] == want.info["total_flops"]
            assert fl[shape.L + 1] == want.info["budget_flops"]


def test_host_qhead_hand_cases_match_oracle(lib):
    # single-layer cases shaped like the oracle's hand-derived pins (4 channel units of 4
    # channels, as the library wants df a multiple of 16), with ratio and score ties
    sh = synth.ModelShape(L=1, d=64, Hq=4, Hkv=2, dh=16, df=16, vocab=0, chan_unit=4)
    for q, ch, r in (([100, 60, 95, 0], [1, 0, 0, 0], 0.75), ([10**6, 4096, 0, 0], [10**5, 1536, 0, 0], 0.49),
                     ([7, 7, 7, 7], [7, 7, 7, 7], 0.6), ([0, 0, 0, 0], [0, 0, 0, 0], 0.9)):
        sc = np.array([q + ch], dtype=np.uint32)
        want = maskc.compile_mask_qheads(sh, sc, [0], r, r, r)
        qh, groups, units, fl = lib.mask_select_qheads(sh, lib.greedy_qhead_mask(sc, [0], r, r, r))
        assert (qh, groups, units) == (want.keep_qheads, want.keep_groups, want.keep_units)
        assert fl[sh.L] == want.info["total_flops"]


def test_explicit_qhead_masks_and_group_kinds(lib):
    sh = synth.tiny_shape(L=3)
    q, u = [[1, 2, 3], [3], [0, 2]], [[0, 3], [2], [1, 4]]
    qh, groups, units, fl = lib.mask_select_qheads(sh, lib.explicit_qhead_mask(q, u))
    want = maskc.explicit_qheads(sh, q, u)
    assert qh == q and groups == want.keep_groups == [[0, 1], [1], [0, 1]] and units == u
    assert fl[sh.L] == ledger.mask_flops(sh, want.keep_groups, want.keep_chans, want.keep_qheads)
    # group kinds report every head of each kept group
    qh, groups, _, _ = lib.mask_select_qheads(sh, lib.explicit_mask([[1], [0, 1], [0]], [[0], [0], [0]]))
    assert groups == [[1], [0, 1], [0]] and qh == [[2, 3], [0, 1, 2, 3], [0, 1]]
    with pytest.raises(lib.TaspError) as e:
        lib.mask_select_qheads(sh, lib.explicit_qhead_mask([[2, 1], [0], [0]], u))  # not ascending
    assert e.value.code == lib.EINVAL
    with pytest.raises(lib.TaspError) as e:
        lib.mask_select_qheads(sh, lib.explicit_qhead_mask([[4], [0], [0]], u))  # head out of range
    assert e.value.code == lib.EINVAL


def test_binding_rejects_host_or_mistyped_buffers_before_any_call(lib):
    # the library takes raw device pointers it cannot check: every wrapper refuses host
    # tensors, wrong dtypes and short buffers before anything reaches the library
    import torch
    sh = synth.tiny_shape(L=1)

    class FakePlan:
        shape = sh
        handle = ctypes.c_void_p(16)

    sess = lib.Session(FakePlan(), 0, handle=ctypes.c_void_p(16))  # never dereferenced
    x_host = torch.zeros((1, sh.d), dtype=torch.bfloat16)
    f_host = torch.zeros(sh.d, dtype=torch.float32)
    with pytest.raises(ValueError, match="GPU"):
        lib.decode_step([sess], x_host)
    with pytest.raises(ValueError, match="GPU"):
        lib.decode_step_static(sess, x_host)
    with pytest.raises(ValueError, match="GPU"):
        lib.decode_step_union([sess], x_host)
    with pytest.raises(ValueError, match="GPU"):
        lib.profile_step([sess], x_host)
    with pytest.raises(ValueError, match="layer residual"):
        sess.layer_step(0, f_host, f_host)
    with pytest.raises(ValueError, match="prompt"):
        lib.Session.prefill(FakePlan(), torch.zeros((4, sh.d), dtype=torch.bfloat16), 8)
    with pytest.raises(ValueError, match="prompt"):
        sess.prefill_into(torch.zeros((4, sh.d + 1), dtype=torch.bfloat16))
    with pytest.raises(ValueError, match="host"):  # the host-buffer entry wants host tensors of the right type
        lib.decode_step_host([sess], torch.zeros((1, sh.d), dtype=torch.float32))
    with pytest.raises(ValueError):
        lib.decode_step_host([sess], torch.zeros((1, sh.d - 1), dtype=torch.bfloat16))


def test_misaligned_device_buffers_are_refused_before_any_work(lib):
    # element-size alignment is checked first, before the handles are even looked at
    so = lib.load()
    P = ctypes.c_void_p
    none = (P * 1)()
    odd = ctypes.c_void_p(0x1001)       # not 2-byte aligned
    half = ctypes.c_void_p(0x1002)      # 2- but not 4-byte aligned
    ok2 = ctypes.c_void_p(0x1000)
    assert so.tasp_decode_step(none, 1, odd, None, None, None) == lib.EINVAL
    assert "aligned" in so.tasp_last_error().decode()
    assert so.tasp_decode_step(none, 1, ok2, half, None, None) == lib.EINVAL
    assert "4 bytes" in so.tasp_last_error().decode()
    assert so.tasp_decode_step(none, 1, ok2, None, half, None) == lib.EINVAL
    assert so.tasp_decode_step_union(none, 1, odd, None, None, None) == lib.EINVAL
    assert so.tasp_decode_step_static(None, odd, None, None, None) == lib.EINVAL
    assert "aligned" in so.tasp_last_error().decode()
    out = ctypes.c_void_p()
    assert so.tasp_prefill(None, odd, 4, 0, None, ctypes.byref(out), None) == lib.EINVAL
    assert so.tasp_session_prefill(None, ok2, 4, None, half) == lib.EINVAL
    assert so.tasp_layer_step(None, 0, half, ok2, None) == lib.EINVAL
    assert "aligned" in so.tasp_last_error().decode()
    # aligned buffers get past the check and meet the handle check instead
    assert so.tasp_decode_step(none, 1, ok2, None, None, None) == lib.EINVAL
    assert "aligned" not in so.tasp_last_error().decode()


def test_memory_limit_fails_cleanly_before_allocating(lib):
    # a cap below the store's size makes plan compilation fail with ENOMEM before any device
    # allocation, and leaves nothing held
    assert lib.memory_in_use() == 0
    lib.set_memory_limit(1 << 20)
    try:
        with pytest.raises(lib.TaspError) as e:
            lib.Plan(synth.LAYER1, lib.all_keep_mask())
        assert e.value.code == lib.ENOMEM
        assert "memory limit" in str(e.value)
        assert lib.memory_in_use() == 0
    finally:
        lib.set_memory_limit(0)
    with pytest.raises(lib.TaspError) as e:
        lib.set_memory_limit(-1)
    assert e.value.code == lib.EINVAL


def test_host_compilers_match_oracle_on_random_shapes_with_ties(lib):
    # seeded random shapes, budgets and retention ranges, with scores drawn from a handful of
    # values so that exact ratio ties are common: both greedy kinds agree bit for bit
    rng = np.random.default_rng(20240611)
    cases = 0
    while cases < 60:
        Hkv = int(rng.choice([1, 2, 4]))
        g = int(rng.choice([1, 2, 4, 8]))
        dh = int(rng.choice([16, 32, 64]))
        cu = int(rng.choice([16, 32, 64]))
        sh = synth.ModelShape(L=int(rng.integers(1, 6)), d=16 * int(rng.integers(2, 12)), Hq=Hkv * g, Hkv=Hkv,
                              dh=dh, df=cu * int(rng.integers(1, 9)), vocab=0, chan_unit=cu)
        lo = float(rng.uniform(0.05, 0.5))
        budget = float(rng.uniform(lo, 0.95))
        hi = float(rng.uniform(budget, 1.0))
        tg = synth.layer_target_u24(int(rng.integers(1 << 30)), sh.L)
        top = int(rng.choice([3, 50, 1 << 32]))
        for kind in ("groups", "qheads"):
            n = (sh.Hkv if kind == "groups" else sh.Hq) + sh.n_chan_units
            sc = rng.integers(0, top, size=(sh.L, n), dtype=np.uint64).astype(np.uint32)
            oracle_fn = maskc.compile_mask if kind == "groups" else maskc.compile_mask_qheads
            try:
                oracle_fn(sh, sc, tg, budget, lo, hi)
            except ValueError:  # budget below the forced minimum: the library refuses it too
                args = (sc, tg, budget, lo, hi)
                with pytest.raises(lib.TaspError) as e:
                    if kind == "groups":
                        lib.mask_select(sh, lib.greedy_mask(*args))
                    else:
                        lib.mask_select_qheads(sh, lib.greedy_qhead_mask(*args))
                assert e.value.code == lib.EINVAL and "budget" in str(e.value)
                continue
            if kind == "groups":
                want = maskc.compile_mask(sh, sc, tg, budget, lo, hi)
                groups, units, fl = lib.mask_select(sh, lib.greedy_mask(sc, tg, budget, lo, hi))
                assert (groups, units) == (want.keep_groups, want.keep_units), (sh, budget, lo, hi)
            else:
                want = maskc.compile_mask_qheads(sh, sc, tg, budget, lo, hi)
                qh, groups, units, fl = lib.mask_select_qheads(sh, lib.greedy_qhead_mask(sc, tg, budget, lo, hi))
                assert (qh, groups, units) == (want.keep_qheads, want.keep_groups, want.keep_units), \
                    (sh, budget, lo, hi)
            assert fl[:sh.L].tolist() == want.info["layer_flops"]
            assert fl[sh.L + 1] == want.info["budget_flops"]
        cases += 1


def test_explicit_masks_fuzzed_against_the_ledger(lib):
    rng = np.random.default_rng(99)
    for _ in range(40):
        Hkv, g = int(rng.choice([1, 2, 4])), int(rng.choice([1, 2, 4, 8]))
        cu = int(rng.choice([16, 32]))
        sh = synth.ModelShape(L=int(rng.integers(1, 5)), d=16 * int(rng.integers(2, 10)), Hq=Hkv * g, Hkv=Hkv,
                              dh=32, df=cu * int(rng.integers(1, 7)), vocab=0, chan_unit=cu)
        units = [sorted(rng.choice(sh.n_chan_units, int(rng.integers(0, sh.n_chan_units + 1)), replace=False).tolist())
                 for _ in range(sh.L)]
        heads = [sorted(rng.choice(sh.Hq, int(rng.integers(0, sh.Hq + 1)), replace=False).tolist())
                 for _ in range(sh.L)]
        groups = [sorted({h // g for h in hs}) for hs in heads]
        want = maskc.explicit_qheads(sh, heads, units)
        qh, kg, ku, fl = lib.mask_select_qheads(sh, lib.explicit_qhead_mask(heads, units))
        assert (qh, kg, ku) == (heads, want.keep_groups, units)
        assert fl[sh.L] == ledger.mask_flops(sh, want.keep_groups, want.keep_chans, want.keep_qheads)
        kg2, ku2, fl2 = lib.mask_select(sh, lib.explicit_mask(groups, units))
        wg = maskc.explicit(sh, groups, units)
        assert (kg2, ku2) == (groups, units)
        assert fl2[sh.L] == ledger.mask_flops(sh, wg.keep_groups, wg.keep_chans)


def test_dispatch_matches_the_oracle(lib):
    from oracle import dispatch
    rng = np.random.default_rng(8)
    cases = [[0.9, 0.05, 0.05, 0.0, 0.0], [0.5, 0.3, 0.1, 0.05, 0.05], [0.2] * 5, [0.5, 0.5]]
    cases += [rng.dirichlet(np.full(5, 0.3)).astype(np.float32).tolist() for _ in range(300)]
    for p in cases:
        for tau in (0.85, 0.5, 0.0, 1.0):
            assert lib.dispatch(p, tau) == dispatch.choose_plan(np.float32(p), np.float32(tau))
    for bad, tau in (([], 0.85), ([0.5, -0.1], 0.85), ([0.5, float("inf")], 0.85), ([0.5], 1.5)):
        with pytest.raises(lib.TaspError) as e:
            lib.dispatch(bad, tau)
        assert e.value.code == lib.EINVAL


def test_header_is_a_plain_c_interface():
    # the boundary is C: the header compiles as C99 on its own (the exports are checked above)
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if not cc:
        pytest.skip("no C compiler")
    src = "#include <tasp.h>\nint main(void) { tasp_status s = TASP_OK; tasp_model_desc m = {0};\n" \
          "  (void)m; return (int)s + (tasp_last_error() == 0); }\n"
    r = subprocess.run([cc, "-x", "c", "-std=c99", "-Wall", "-Werror", "-fsyntax-only",
                        "-I", os.path.join(ROOT, "include"), "-"], input=src, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
def _store_row(shape, proj, row):
    # the store's qkv rows are group-major: per KV group its g head blocks, then K, then V
    g, dh = shape.g, shape.dh
    if proj == "q":
        h, i = divmod(row, dh)
        j, hh = divmod(h, g)
    else:
        j, i = divmod(row, dh)
        hh = g if proj == "k" else g + 1
    return (j * (g + 2) + hh) * dh + i


@pytest.mark.parametrize("shape,heads", [
    (synth.LAYER1, [[1, 2, 3, 4, 6]]),
    (dataclasses.replace(synth.LLAMA3_8B, L=2), [[0, 1, 2, 5, 9, 10, 11, 31], [3, 4, 7, 30]]),
    (dataclasses.replace(synth.LLAMA3_8B, L=1), [list(range(32))]),
])
def test_partial_group_tables_match_the_oracle_packing(lib, shape, heads):
    from oracle import pack
    units = [[0] for _ in range(shape.L)]
    m = maskc.explicit_qheads(shape, heads, units)
    g, dh = shape.g, shape.dh
    for layer in range(shape.L):
        t = lib.plan_layout(shape, lib.explicit_qhead_mask(heads, units), layer)
        kg, qh = m.keep_groups[layer], m.keep_qheads[layer]
        want = [_store_row(shape, p, r) for p, r in pack.qkv_rows(shape, kg, qh)]
        assert t["qkv_src"].tolist() == want
        assert t["o_src"].tolist() == [h * dh + i for h in qh for i in range(dh)]
        # role: block b of the panel holds (group slot, head or K / V); blk_of inverts it
        nblk = len(qh) + 2 * len(kg)
        assert len(t["role"]) == nblk and len(t["blk_of"]) == len(kg) * (g + 2)
        for b, code in enumerate(t["role"].tolist()):
            jl, hh = divmod(code, g + 2)
            assert t["blk_of"][code] == b
            assert t["qkv_src"][b * dh] == (kg[jl] * (g + 2) + hh) * dh
        assert sorted(int(x) for x in t["blk_of"] if x >= 0) == list(range(nblk))
        # slot: compact O position of each kept head, -1 for dropped ones
        for jl, j in enumerate(kg):
            for hh in range(g):
                h = j * g + hh
                assert t["slot"][jl * g + hh] == (qh.index(h) if h in qh else -1)


def _dense_of_store_row(shape, r):
    g, dh = shape.g, shape.dh
    blk, i = divmod(r, dh)
    j, hh = divmod(blk, g + 2)
    if hh < g:
        return ("q", (j * g + hh) * dh + i)
    return ("k" if hh == g else "v", j * dh + i)


@pytest.mark.parametrize("shape,heads", [
    (synth.LAYER1, [[1, 2, 3, 4, 6]]),
    (dataclasses.replace(synth.LLAMA3_8B, L=1), [[0, 1, 2, 5, 9, 10, 11, 31]]),
])
def test_kernel_index_math_with_partial_group_tables(lib, shape, heads):
    # the decode QKV epilogue, the attention output store and the prefill rotary kernel,
    # replayed on the host with the plan's tables: every query slot, K / V row and O column
    # receives exactly the dense row or column the oracle's mask-as-zero forward uses
    units = [[0]]
    m = maskc.explicit_qheads(shape, heads, units)
    kg, qh = m.keep_groups[0], m.keep_qheads[0]
    g, dh, half = shape.g, shape.dh, shape.dh // 2
    t = lib.plan_layout(shape, lib.explicit_qhead_mask(heads, units), 0)
    src, role, slot, blk_of = t["qkv_src"], t["role"], t["slot"], t["blk_of"]
    rows = len(src)
    # decode: work rows in pairs (w, w + 1) hold panel rows (hb dh + i, hb dh + i + d_h / 2)
    written = {}
    for wa in range(0, rows, 2):
        hb = wa // dh
        i = (wa - hb * dh) >> 1
        pr0, pr1 = hb * dh + i, hb * dh + i + half
        jl, hh = divmod(int(role[hb]), g + 2)
        dest = ("q", jl * g + hh) if hh < g else ("k" if hh == g else "v", jl)
        for off, pr in ((i, pr0), (i + half, pr1)):
            key = (dest, off)
            assert key not in written
            written[key] = _dense_of_store_row(shape, int(src[pr]))
    for jl, j in enumerate(kg):
        for hh in range(g):
            h = j * g + hh
            for i in range(dh):
                if h in qh:
                    assert written[(("q", jl * g + hh), i)] == ("q", h * dh + i)
                else:
                    assert (("q", jl * g + hh), i) not in written  # the slot stays zero
        for kv in ("k", "v"):
            for i in range(dh):
                assert written[((kv, jl), i)] == (kv, j * dh + i)
    # attention output: head (jl, hh) lands in compact O columns slot * d_h, which the O panel
    # maps back to the dense columns of head h
    for jl, j in enumerate(kg):
        for hh in range(g):
            s = int(slot[jl * g + hh])
            if s >= 0:
                assert t["o_src"][s * dh:(s + 1) * dh].tolist() == list(range((j * g + hh) * dh, (j * g + hh + 1) * dh))
    # prefill: the rotary kernel reads panel column block blk_of[jl (g + 2) + hh] (rows in panel order)
    for jl, j in enumerate(kg):
        for hh in range(g + 2):
            b = int(blk_of[jl * (g + 2) + hh])
            if hh < g and j * g + hh not in qh:
                assert b == -1
                continue
            want = ("q", (j * g + hh) * dh) if hh < g else ("k" if hh == g else "v", j * dh)
            assert _dense_of_store_row(shape, int(src[b * dh])) == want


def test_groupwise_shapes_are_validated_on_the_host(lib):
    import dataclasses
    sh = synth.LLAMA3_8B
    sc = synth.mask_scores_u32(1000, sh.L, sh.n_units)
    tg = synth.layer_target_u24(1000, sh.L)
    ok = lib.mask_select(dataclasses.replace(sh, quant_group=128), lib.greedy_mask(sc, tg))
    assert ok[0] == lib.mask_select(sh, lib.greedy_mask(sc, tg))[0]  # the mask does not depend on scales
    for bad in (48, 100, -16, 256 * 1024):
        with pytest.raises(lib.TaspError) as e:
            lib.mask_select(dataclasses.replace(sh, quant_group=bad), lib.greedy_mask(sc, tg))
        assert e.value.code == lib.EINVAL
