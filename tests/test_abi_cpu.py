"""C-ABI library: loads without a GPU, exports every declared symbol, and its
host-side validation answers without touching the device."""
import ctypes
import os
import re

import pytest

from paper_2609_32479_gb300 import trackfit as T, workloads as W

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "trackfit.h")


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(T.LIB_PATH):
        import __graft_entry__
        __graft_entry__.build()
    return T.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(trackfit_[a-z_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(T.EXPORTS)


@pytest.mark.parametrize("name", ["tiny", "small", "medium", "large", "sweep64"])
def test_weight_count_matches_layout(lib, name):
    m = W.workload(name).model
    assert T.weight_count(m) == W.weight_count(m)
    e = m.with_(pool=W.POOL_ENDPOINTS)
    assert T.weight_count(e) == W.weight_count(e)


@pytest.mark.parametrize("name", ["paper", "transformer"])
def test_weight_count_of_the_paper_models(lib, name):
    m = W.workload(name).model
    assert T.weight_count(m) == W.weight_count(m) > 0
    if m.topology == W.TOPOLOGY_ATTENTION:
        for kw in (dict(n_heads=2), dict(n_heads=16), dict(d_hidden=16), dict(n_layers=1)):
            assert T.weight_count(m.with_(**kw)) == W.weight_count(m.with_(**kw))
        assert T.weight_count(m.with_(n_heads=1)) == 0     # head width 128 > 64


@pytest.mark.parametrize("bad", [dict(d_model=24), dict(d_hidden=100), dict(max_hits=65), dict(max_hits=0),
                                 dict(n_layers=0), dict(n_layers=17), dict(head_hidden=64), dict(n_quantiles=6),
                                 dict(precision=3), dict(pool=3), dict(n_fourier=8), dict(rms_eps=0.0), dict(topology=3),
                                 dict(d_model=272, d_hidden=408), dict(topology=2, pool=1),
                                 dict(topology=2, n_heads=3), dict(topology=2, n_heads=8),
                                 dict(topology=2, n_heads=0), dict(topology=2, d_hidden=40),
                                 dict(topology=2, d_hidden=1040)])
def test_unsupported_configs_rejected_on_host(lib, bad):
    m = W.workload("tiny").model.with_(**bad)
    c = T.make_config(m)
    assert lib.trackfit_weight_count(ctypes.byref(c)) == 0
    h = ctypes.c_void_p()
    st = lib.trackfit_create(ctypes.byref(c), ctypes.c_void_p(16), 10, ctypes.byref(h))
    assert st == T.ERR_UNSUPPORTED and not h.value


def test_null_and_count_errors_on_host(lib):
    m = W.workload("tiny").model
    c = T.make_config(m)
    h = ctypes.c_void_p()
    assert lib.trackfit_create(None, ctypes.c_void_p(16), 1, ctypes.byref(h)) == T.ERR_INVALID_ARG
    assert lib.trackfit_create(ctypes.byref(c), None, 1, ctypes.byref(h)) == T.ERR_INVALID_ARG
    n = W.weight_count(m)
    assert lib.trackfit_create(ctypes.byref(c), ctypes.c_void_p(16), n + 1, ctypes.byref(h)) == T.ERR_INVALID_ARG
    for v in (T.ABI_VERSION - 1, T.ABI_VERSION + 1):   # another layout of the config struct
        c.abi_version = v
        assert lib.trackfit_create(ctypes.byref(c), ctypes.c_void_p(16), n, ctypes.byref(h)) == T.ERR_UNSUPPORTED
    assert lib.trackfit_forward(None, ctypes.c_void_p(16), ctypes.c_void_p(16), 4, ctypes.c_void_p(16),
                                None) == T.ERR_INVALID_ARG
    lib.trackfit_destroy(None)
    for s in range(7):
        assert T.strerror(s) and T.strerror(s) != "unknown status"
    assert lib.trackfit_path_name(None) == b"none"


def _epilogue_handovers(m):
    """Per-tile hand-overs of the fused kernel's epilogue warps, restated from
    their loop: the tile's Fourier operand, the embedding's SiLU, then x_hat one
    128-channel tile at a time; per layer one release of the z/n columns per scan
    chunk, the output gate and the MLP's SiLU per channel tile, and x_hat per
    channel tile except after the last layer (mean pooling instead).  The waits:
    the embedding's two products (the second per channel tile), per layer the
    z/n products of every chunk, the last merge, MLP1 and MLP2 per channel tile."""
    MT, NDC, L = m.d_model // 128, m.d_hidden // 64, m.n_layers
    signals = 2 + MT + sum(NDC + 2 * MT + (MT if l + 1 < L else 0) for l in range(L))
    waits = 1 + MT + L * (NDC + 3 * MT)
    return signals, waits


@pytest.mark.parametrize("D,H,L,prec", [(128, 192, 6, W.PRECISION_BF16), (256, 384, 8, W.PRECISION_BF16),
                                        (128, 192, 1, W.PRECISION_FP16), (256, 384, 1, W.PRECISION_FP16),
                                        (256, 384, 2, W.PRECISION_BF16), (128, 192, 16, W.PRECISION_BF16)])
def test_schedule_handovers_match_the_epilogue(lib, D, H, L, prec):
    """The issuer's hand-over waits and commits pair one to one with the epilogue's
    arrivals and waits (a mismatch would stall a wait until its time limit, or let
    one side run ahead), and the MMAs cover exactly the per-hit work of the model."""
    m = W.ModelConfig(max_hits=24, d_model=D, d_hidden=H, n_layers=L, precision=prec)
    c = T.schedule_counts(m)
    assert c is not None
    signals, waits = _epilogue_handovers(m)
    NDC = H // 64
    assert c["w_e"] == signals
    assert c["c_acc"] == waits
    assert c["w_h"] == L * NDC
    assert c["c_hb"] == L * (NDC - 1)
    E = 2 * m.n_features * m.n_fourier
    flops_per_column = 2 * (D * E + D * D) + L * (2 * D * (4 * H + D) + 4 * H * D + 4 * D * D)
    assert c["mmas"] * 128 * 128 * 16 * 2 == 128 * flops_per_column
    assert c["blocks"] * 4 >= c["mmas"]


def test_schedule_hook_rejects_cuda_core_configs(lib):
    assert T.schedule_counts(W.workload("tiny").model) is None
    assert T.schedule_counts(W.workload("large").model.with_(precision=W.PRECISION_FP32)) is None


def _epilogue_events(m, tiles=2, states=False):
    """The epilogue warps' hand-over events in program order for `tiles` tiles:
    'S' = an operand hand-over (W_E arrival), 'W' = a wait for an accumulator
    commit (C_ACC), restated from the epilogue loop; with states, also 'B' = a
    wait for a state-buffer commit (C_HB) and 'H' = a state hand-over (W_H)."""
    MT, NDC, L = m.d_model // 128, m.d_hidden // 64, m.n_layers
    ev = ["S"]                                   # the first tile's Fourier operand
    for _ in range(tiles):
        ev += ["W", "S"]                         # embedding product 1 -> its SiLU
        ev += ["W"] * MT + ["S"] * MT            # embedding product 2 -> x_hat per channel tile
        for l in range(L):
            for dc in range(NDC):                # z/n of each chunk -> columns released
                ev += ["W", "S"]                 # (-> previous merge done -> states handed over)
                if states:
                    ev += (["B"] if dc > 0 else []) + ["H"]
            ev += ["W", "S"] * MT                # last merge tile -> output gate of that tile
            ev += ["W", "S"] * MT                # MLP1 tile -> its SiLU
            ev += ["W"] * MT                     # MLP2 tiles
            ev += ["S"] * MT if l + 1 < L else ["S"]   # x_hat per tile, or the next tile's operand
    return ev


@pytest.mark.parametrize("D,H,L", [(128, 192, 6), (256, 384, 8), (256, 384, 1), (128, 192, 1)])
def test_no_epilogue_warp_runs_two_hand_overs_ahead(lib, D, H, L):
    """The operand hand-overs alternate between two barriers, which is enough only
    if no warp can arrive for hand-over k + 2 before every warp has arrived for k:
    hand-over k + 2 must come after a wait for an accumulator commit that the
    issuer makes only after consuming hand-over k.  Checked on the issuer's block
    order against the epilogue's event order over two tiles."""
    m = W.ModelConfig(max_hits=24, d_model=D, d_hidden=H, n_layers=L, precision=W.PRECISION_BF16)
    codes = T.schedule_counts(m, with_codes=True)["codes"] * 3
    w_before_commit = []                       # W_E hand-overs the issuer consumed before commit c
    n_we = 0
    for code in codes:
        if code & 3 == 1:
            n_we += 1
        if (code >> 2) == 1:
            w_before_commit.append(n_we)
    ev = _epilogue_events(m)
    n_sig = sum(e == "S" for e in ev)
    assert sum(e == "W" for e in ev) <= len(w_before_commit)
    waits = 0
    s = 0
    for e in ev:
        if e == "W":
            waits += 1
            continue
        # a warp reaching hand-over s has seen commit waits - 1, which needs hand-overs
        # 0 .. w_before_commit[waits - 1] - 1 from every warp
        done_by_all = w_before_commit[waits - 1] if waits else 0
        assert s - done_by_all <= 1, f"hand-over {s} can run {s - done_by_all} ahead"
        s += 1
    assert s == n_sig


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    """No CPU fallback: without the built library the binding raises instead of
    computing anything."""
    monkeypatch.setattr(T, "_lib", None)
    monkeypatch.setattr(T, "LIB_PATH", str(tmp_path / "libtrackfit.so"))
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        T.load()
    with pytest.raises(RuntimeError):
        T.weight_count(W.workload("tiny").model)


@pytest.mark.parametrize("D,H,L", [(128, 192, 6), (256, 384, 8), (256, 384, 1), (128, 192, 1), (128, 192, 16)])
def test_no_epilogue_warp_falls_two_commits_behind(lib, D, H, L):
    """The accumulator commits alternate between two barriers, which is enough only
    if no warp can still be waiting for commit k when commit k + 2 (same barrier)
    lands: the issuer must make commit k + 2 only after some hand-over (operand or
    state) that every warp gives after its wait for commit k.  Checked on the
    issuer's block order against the epilogue's event order over three tiles."""
    m = W.ModelConfig(max_hits=24, d_model=D, d_hidden=H, n_layers=L, precision=W.PRECISION_BF16)
    tiles = 3
    codes = T.schedule_counts(m, with_codes=True)["codes"] * tiles
    ev = _epilogue_events(m, tiles=tiles, states=True)
    # accumulator waits completed by a warp before it gives its k-th W_E / W_H hand-over
    done_before = {"S": [], "H": []}
    waits = 0
    for e in ev:
        if e == "W":
            waits += 1
        elif e in done_before:
            done_before[e].append(waits)
    n_commits = sum(1 for c in codes if (c >> 2) == 1)
    assert n_commits >= waits                    # every epilogue wait has its commit
    # walk the issuer: gate[j] = the most accumulator waits that every warp has
    # certainly completed when commit j is issued
    n_s = n_h = 0
    gate = 0
    j = 0
    for c in codes:
        if c & 3 == 1:
            if n_s < len(done_before["S"]):
                gate = max(gate, done_before["S"][n_s])
            n_s += 1
        elif c & 3 == 2:
            if n_h < len(done_before["H"]):
                gate = max(gate, done_before["H"][n_h])
            n_h += 1
        if (c >> 2) == 1:
            if j >= 2 and j < waits:
                assert gate >= j - 1, f"commit {j} can land while a warp still waits for commit {j - 2}"
            j += 1
    assert n_s >= len(done_before["S"]) - 1 and n_h >= len(done_before["H"])
