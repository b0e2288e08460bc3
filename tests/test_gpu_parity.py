"""GPU (sm_103a) path against the CPU oracle, element by element, through the C ABI.

Integer work, so the bar is bit-exact: makespan, every decision word, nseg and
status for the DP; every int64 of the generated profiles; every makespan of the
timeline replay. Inputs are seeded and synthetic; every expected value comes
from the oracle.
"""
import os

import numpy as np
import pytest

import oracle
from paper_2101_07968_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

FWD, BWD = 0, 1
NTHREADS = os.cpu_count() or 1


@pytest.fixture(scope="module")
def dc():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_07968_gb300 import build, dynacomm
    build.build()
    dynacomm.lib()
    return dynacomm


def _dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _gpu_schedule(dc, direction, comp, xfer, dt):
    import torch
    B, L = comp.shape
    out = dc.schedule(direction, _dev(comp), _dev(xfer), _dev(dt))
    torch.cuda.synchronize()
    W = dc.words(L)
    res = {k: v.cpu().numpy() for k, v in out.items()}
    res["bits"] = res["bits"].view(np.uint32)[:, :W] if W else np.zeros((B, 0), np.uint32)
    return res


def _assert_same(got, exp, label=""):
    for key in ("status", "makespan", "nseg", "bits"):
        g, e = got[key], exp[key]
        if key == "bits":
            g = g.reshape(e.shape)
        bad = np.nonzero(g != e)[0] if g.ndim == 1 else np.nonzero((g != e).any(axis=1))[0]
        assert bad.size == 0, (f"{label} {key}: {bad.size} mismatches, first at {bad[0]}: "
                               f"gpu={g[bad[0]]} oracle={e[bad[0]]}")


def _check_direction(dc, direction, comp, xfer, dt, label=""):
    got = _gpu_schedule(dc, direction, comp, xfer, dt)
    exp = oracle.schedule_batch(direction, comp, xfer, dt, nthreads=NTHREADS)
    _assert_same(got, exp, label)
    return got


# ------------------------------------------------------------------ DP parity
SMALL_LS = list(range(1, 21)) + [31, 32, 33, 40, 41, 48, 54, 63, 64, 65, 96, 128, 129, 130, 256]


@pytest.mark.parametrize("L", SMALL_LS)
@pytest.mark.parametrize("kind", ["tie", "uni", "skew"])
def test_dp_random_parity(dc, L, kind):
    """Several tiles and a ragged tail for every kernel variant and width."""
    B = {True: 700, False: 150}[L <= 20] + 13
    gen = {"tie": wl.tie_heavy_instances, "uni": wl.random_instances,
           "skew": wl.skewed_instances}[kind]
    comp, xfer, dt = gen(1000 * L + len(kind), B, L)
    for d in (FWD, BWD):
        _check_direction(dc, d, comp, xfer, dt, f"L={L} {kind} dir={d}")


@pytest.mark.parametrize("L", [9, 11, 12, 13, 14, 15, 16])
def test_dp_many_tiles_per_warp(dc, L):
    """Batches that give every resident warp of the short-L pass several tiles and
    a ragged last one: the shared-area design (L < 12) and the split design with
    its ticket and the next tile staged while one is solved (12 <= L <= 16; odd L
    copies 8-byte words), against the oracle on every instance."""
    B = 480_007
    comp, xfer, dt = wl.random_instances(7000 + L, B, L)
    for d in (FWD, BWD):
        _check_direction(dc, d, comp, xfer, dt, f"L={L} B={B} dir={d}")


@pytest.mark.parametrize("L", [257, 258, 300, 333, 512, 600])
@pytest.mark.parametrize("kind", ["tie", "uni", "skew"])
def test_dp_deep_random_parity(dc, L, kind):
    """The warp-per-instance deep-chain kernel (L > 256) and its work list:
    several waves of instances, odd and even L (odd L stages rows with plain
    loads), tie-heavy inputs for the traceback's lowest-k rule."""
    B = 45
    gen = {"tie": wl.tie_heavy_instances, "uni": wl.random_instances,
           "skew": wl.skewed_instances}[kind]
    comp, xfer, dt = gen(3000 * L + len(kind), B, L)
    for d in (FWD, BWD):
        _check_direction(dc, d, comp, xfer, dt, f"L={L} {kind} dir={d}")


@pytest.mark.parametrize("B", [500, 1000, 2000])
def test_dp_deep_warps_per_instance(dc, B):
    """Batch sizes that give the deep-chain kernel 4, 2 and 1 warps per instance
    (the rows of a column dealt to the warps strip by strip), full batches
    bit-exact with the oracle; the xfer array starts 8 bytes past a 16-byte
    boundary in one direction, which stages the rows with plain loads."""
    import torch
    L = 300
    comp, xfer, dt = wl.skewed_instances(4000 + B, B, L)
    buf = torch.empty(xfer.size + 1, dtype=torch.int64, device="cuda")
    xs = buf[1:].view(xfer.shape)
    xs.copy_(torch.from_numpy(xfer))
    W = dc.words(L)
    for d in (FWD, BWD):
        if d == FWD:
            got = _gpu_schedule(dc, d, comp, xfer, dt)
        else:
            out = dc.schedule(d, _dev(comp), xs, _dev(dt))
            torch.cuda.synchronize()
            got = {k: v.cpu().numpy() for k, v in out.items()}
            got["bits"] = got["bits"].view(np.uint32)[:, :W]
        exp = oracle.schedule_batch(d, comp, xfer, dt, nthreads=NTHREADS)
        _assert_same(got, exp, f"B={B} dir={d}")


@pytest.mark.parametrize("L", [1, 2, 8, 16, 17, 54, 70, 100, 200])
def test_dp_wide_values_parity(dc, L):
    """Instances whose bound exceeds 2^32 need 64-bit arithmetic; mix them with
    32-bit ones so both paths (and the work list) run in one call."""
    B = 640 + 7
    comp, xfer, dt = wl.skewed_instances(77 + L, B, L)
    rng = np.random.default_rng(L)
    wide = rng.random(B) < 0.3
    scale = rng.integers(1 << 26, 1 << 36, size=(B, 1))
    comp[wide] = comp[wide] * 3 + (scale[wide] * rng.random((wide.sum(), L))).astype(np.int64)
    xfer[wide] = xfer[wide] + (scale[wide] * rng.random((wide.sum(), L))).astype(np.int64)
    dt[wide[:]] += rng.integers(0, 1 << 30, size=wide.sum())
    bound = L * dt + comp.sum(1) + xfer.sum(1)
    assert (bound[wide] > 2**32).any() and (bound < 2**52).all()
    for d in (FWD, BWD):
        _check_direction(dc, d, comp, xfer, dt, f"wide L={L} dir={d}")


@pytest.mark.parametrize("L", [17, 40, 64, 65, 100, 257])
def test_dp_wide_latency_small_compute_parity(dc, L):
    """Bound above 2^32 from the latency and the transfers while the total compute
    stays below 2^29: the shifted 32-bit solves of the per-instance kernel. Thirds
    of the batch: a huge latency (every 8-row block wider than 2^30 of transfer
    plus latency); log-uniform transfers with a latency near 2^32 / L (blocks on
    both sides of 2^30); plain 32-bit instances."""
    B = 3 * 97 + 5
    comp, xfer, dt = wl.skewed_instances(313 + L, B, L)
    rng = np.random.default_rng(1000 + L)
    part = np.arange(B) % 3
    comp = comp % (1 << 20)
    big_dt = part == 0
    dt[big_dt] = rng.integers(1 << 30, 1 << 40, size=big_dt.sum())
    big_x = part == 1
    nb = int(big_x.sum())
    comp[big_x] = rng.integers((1 << 27) // L, (1 << 29) // L, size=(nb, L))
    xfer[big_x] = np.exp2(rng.uniform(16, 31, size=(nb, L))).astype(np.int64)
    dt[big_x] = rng.integers((1 << 31) // L, (1 << 33) // L, size=nb)
    bound = L * dt + comp.sum(1) + xfer.sum(1)
    assert (bound[part < 2] > 2**32).all() and (comp.sum(1) < 2**29).all()
    for d in (FWD, BWD):
        _check_direction(dc, d, comp, xfer, dt, f"wide-latency L={L} dir={d}")


@pytest.mark.parametrize("L", [2, 6, 8, 13, 14, 16])
@pytest.mark.parametrize("which", ["both", "xfer"])
def test_dp_unaligned_cost_arrays(dc, L, which):
    """Cost arrays starting 8 bytes past a 16-byte boundary: the short-L pass then
    stages single costs instead of 16-byte pairs. Same outputs as the oracle."""
    import torch
    B = 1000 + 17
    comp, xfer, dt = wl.random_instances(900 + L, B, L, 0, 100_000, 0, 10_000)

    def shifted(a):
        buf = torch.empty(a.size + 1, dtype=torch.int64, device="cuda")
        v = buf[1:].view(a.shape)
        v.copy_(torch.from_numpy(np.ascontiguousarray(a)))
        assert v.data_ptr() % 16 == 8
        return v

    W = dc.words(L)
    for d in (FWD, BWD):
        c = shifted(comp) if which == "both" else _dev(comp)
        out = dc.schedule(d, c, shifted(xfer), _dev(dt))
        torch.cuda.synchronize()
        got = {k: v.cpu().numpy() for k, v in out.items()}
        got["bits"] = got["bits"].view(np.uint32)[:, :W] if W else np.zeros((B, 0), np.uint32)
        exp = oracle.schedule_batch(d, comp, xfer, dt, nthreads=NTHREADS)
        _assert_same(got, exp, f"unaligned {which} L={L} dir={d}")
        # the replay of those decisions from the same unaligned arrays
        rep = dc.eval_timeline(d, c, shifted(xfer), _dev(dt), out["bits"][:, :max(W, 1)].contiguous())
        assert np.array_equal(rep.cpu().numpy(), exp["makespan"]), f"replay unaligned {which} L={L}"


@pytest.mark.parametrize("L", [8, 16, 54, 100])
def test_dp_status_faults_per_instance(dc, L):
    B = 300
    comp, xfer, dt = wl.random_instances(5 + L, B, L, 0, 100_000, 0, 10_000)
    comp[3, L - 1] = -5
    xfer[10, 0] = -1
    dt[20] = -7
    xfer[30, L // 2] = 1 << 52                       # one value alone too big
    comp[40, :] = (1 << 52) // L                      # sum too big
    dt[50] = 1 << 51                                  # L * dt too big (L >= 2)
    for d in (FWD, BWD):
        got = _check_direction(dc, d, comp, xfer, dt, f"faults L={L} dir={d}")
        assert list(got["status"][[3, 10, 20, 30, 40, 50]]) == [3, 3, 3, 4, 4, 4]
        assert (got["status"][[0, 1, 2, 4, 299]] == 0).all()


def test_dp_batch_zero_and_single(dc):
    import torch
    ws = torch.empty(4096, dtype=torch.uint8, device="cuda")
    z = torch.empty(0, dtype=torch.int64, device="cuda")
    assert dc.dc_schedule_forward_batch(0, 8, z, z, z, z, z, None, None, ws, 4096) == dc.DC_OK
    comp, xfer, dt = wl.random_instances(3, 1, 1, 0, 50, 0, 50)
    for d in (FWD, BWD):
        _check_direction(dc, d, comp, xfer, dt, "batch=1 L=1")
    # one instance, and one partial tile, on every kernel family and warp count
    for L in (16, 40, 64, 100, 200, 300):
        for B in (1, 33):
            comp, xfer, dt = wl.skewed_instances(11 * L + B, B, L)
            for d in (FWD, BWD):
                _check_direction(dc, d, comp, xfer, dt, f"batch={B} L={L}")


def test_dp_maximum_L(dc):
    """L = 4096 (the largest the ABI takes): the backward optimum equals the 1-D
    recurrence, both decisions replay to their makespans, and neither is worse
    than layer-by-layer or sequential."""
    L, B = 4096, 2
    comp, xfer, dt = wl.random_instances(9, B, L, 0, 5_000, 0, 50_000)
    for d in (FWD, BWD):
        got = _gpu_schedule(dc, d, comp, xfer, dt)
        assert (got["status"] == 0).all()
        rep = oracle.replay_batch(d, comp, xfer, dt, got["bits"], nthreads=2)
        assert np.array_equal(rep, got["makespan"])
        seq = np.zeros((B, dc.words(L)), np.uint32)
        lbl = oracle.replay_batch(d, comp, xfer, dt, np.full_like(seq, 0xFFFFFFFF) & _mask(L))
        assert (got["makespan"] <= oracle.replay_batch(d, comp, xfer, dt, seq)).all()
        assert (got["makespan"] <= lbl).all()
        assert (got["nseg"] == 1 + np.unpackbits(got["bits"].view(np.uint8), axis=1).sum(1)).all()
        if d == BWD:
            for i in range(B):
                assert got["makespan"][i] == oracle.dp_backward_1d(comp[i], xfer[i], dt[i])


def _mask(L):
    W = (L - 1 + 31) // 32
    m = np.zeros(W, np.uint32)
    for l in range(L - 1):
        m[l // 32] |= np.uint32(1 << (l % 32))
    return m


# ------------------------------------------------------- generator parity
@pytest.mark.parametrize("name", wl.CONFIG_NAMES)
def test_profile_gen_bitwise(dc, name):
    """Full batch of every configuration, every int64 equal to the oracle's."""
    import torch
    cfg = wl.config(name)
    got = dc.profile_gen(cfg)
    torch.cuda.synchronize()
    exp = oracle.profile_gen(cfg)
    for k in ("fc", "pt", "bc", "gt", "dt"):
        g = got[k].cpu().numpy()
        bad = np.nonzero((g != exp[k]).reshape(len(g), -1).any(axis=1))[0]
        assert bad.size == 0, f"{name}.{k}: {bad.size} rows differ, first {bad[:3]}"


def test_profile_gen_offset_and_ragged(dc):
    import torch
    cfg = wl.with_batch(wl.config("deepchain"), 37, inst0=123_456)
    cfg["L"] = 77
    got = dc.profile_gen(cfg)
    torch.cuda.synchronize()
    exp = oracle.profile_gen(cfg)
    for k in ("fc", "pt", "bc", "gt", "dt"):
        assert np.array_equal(got[k].cpu().numpy(), exp[k])


# -------------------------------------------------------- timeline parity
@pytest.mark.parametrize("L", [1, 2, 7, 16, 32, 33, 48, 54, 64, 65, 1024])
def test_eval_timeline_random_decisions(dc, L):
    import torch
    B = 500 + 3
    comp, xfer, dt = wl.skewed_instances(31 * L, B, L)
    comp[5, 0] = -1
    dt[9] = 1 << 52
    bits = wl.random_decisions(L, B, L, density=0.3)
    for d in (FWD, BWD):
        got = dc.eval_timeline(d, _dev(comp), _dev(xfer), _dev(dt),
                               _dev(bits.view(np.int32)) if bits.size else None)
        torch.cuda.synchronize()
        exp = oracle.replay_batch(d, comp, xfer, dt, bits, nthreads=NTHREADS)
        assert np.array_equal(got.cpu().numpy(), exp)


# ---------------------------------------------- full-size configurations
def _config_parity(dc, name, sample=None):
    cfg = wl.config(name)
    prof = oracle.profile_gen(cfg)
    for d, (c, x) in ((FWD, ("fc", "pt")), (BWD, ("bc", "gt"))):
        got = _gpu_schedule(dc, d, prof[c], prof[x], prof["dt"])
        if sample is None:
            exp = oracle.schedule_batch(d, prof[c], prof[x], prof["dt"], nthreads=NTHREADS)
            _assert_same(got, exp, f"{name} dir={d}")
        else:
            idx = np.asarray(sample)
            exp = oracle.schedule_batch(d, prof[c][idx], prof[x][idx], prof["dt"][idx],
                                        nthreads=NTHREADS)
            sub = {k: v[idx] for k, v in got.items()}
            _assert_same(sub, exp, f"{name} dir={d} sample")
            # every instance: the decision replays to the makespan
            rep = oracle.replay_batch(d, prof[c], prof[x], prof["dt"], got["bits"],
                                      nthreads=NTHREADS)
            assert np.array_equal(rep, got["makespan"])
            if d == BWD:
                for i in idx[:64]:
                    assert got["makespan"][i] == oracle.dp_backward_1d(
                        prof[c][i], prof[x][i], prof["dt"][i])


@pytest.mark.parametrize("name", ["tiny", "alexnet", "vgg16", "resnet50"])
def test_config_full_batch_parity(dc, name):
    _config_parity(dc, name)


def _solve_class(direction, comp, xfer, dt):
    """Which arithmetic the per-instance solvers use for each instance (a
    property of the inputs: the capped bound and the total compute), to spread
    a sample over every path. 0: shifted signed 32 bits; 1: backward E form;
    2: forward E form; 3: 32-bit template; 4: 64-bit."""
    sc = comp.sum(1)
    cx = np.minimum(xfer, sc[:, None]).sum(1)
    bound = sc + cx + comp.shape[1] * dt
    cls = np.full(len(dt), 4)
    cls[bound <= 2**32 - 2] = 3
    if direction == BWD:
        cls[sc < 2**31 - 1] = 1
    else:
        cls[sc < 2**29] = 2
    cls[bound <= 2**31 - 1] = 0
    return cls


def _deepchain_sample(prof, size, seed):
    """`size` instances spread over the whole batch: half uniformly, half from the
    instances that need a wide form in either direction."""
    rng = np.random.default_rng(seed)
    B = len(prof["dt"])
    wide = np.nonzero((_solve_class(FWD, prof["fc"], prof["pt"], prof["dt"]) > 0) |
                      (_solve_class(BWD, prof["bc"], prof["gt"], prof["dt"]) > 0))[0]
    pick = np.concatenate([[0, 1, B - 1], rng.choice(B, size // 2, replace=False),
                           rng.choice(wide, size - size // 2 - 3, replace=False)])
    return np.unique(pick)


def test_config_deepchain_sampled_parity(dc):
    """512+ deep-chain instances (L = 1024) from all over the batch, half of them
    from the instances that take the wide forms, bit-exact with the oracle in both
    directions; every decision of the batch replays to its makespan."""
    prof = oracle.profile_gen(wl.config("deepchain"))
    sample = _deepchain_sample(prof, 520, 4)
    assert len(sample) >= 512
    for d, (c, x) in ((FWD, ("fc", "pt")), (BWD, ("bc", "gt"))):
        cls = _solve_class(d, prof[c][sample], prof[x][sample], prof["dt"][sample])
        assert (cls == 0).sum() >= 100 and (cls == (1 if d == BWD else 2)).sum() >= 100
    _config_parity(dc, "deepchain", sample=sample)


def _digests():
    from conftest import GOLDEN
    prof, chunks = {}, {}
    with open(os.path.join(GOLDEN, "deepchain_oracle_digest.txt")) as f:
        for line in f:
            w = line.split()
            if not w or w[0].startswith("#"):
                continue
            if w[0] == "profile":
                prof[w[1]] = w[2]
            elif w[0] == "chunk":
                chunks[(int(w[1]), int(w[2]), int(w[3]))] = w[4]
    return prof, chunks


def test_config_deepchain_full_batch_digest(dc):
    """Every instance of the deep-chain batch (16,384 x L = 1024), both directions,
    bit for bit: the library's profiles and outputs hashed in chunks of 256
    instances against tests/golden/deepchain_oracle_digest.txt, which
    tests/golden/make_deepchain_digest.py wrote from the oracle's outputs."""
    import hashlib

    import torch
    sys_path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
    import importlib.util
    spec = importlib.util.spec_from_file_location(
        "make_deepchain_digest", os.path.join(sys_path, "make_deepchain_digest.py"))
    mk = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mk)
    want_prof, want_chunks = _digests()
    assert len(want_chunks) == 2 * 64
    cfg = wl.config("deepchain")
    prof = dc.profile_gen(cfg)
    torch.cuda.synchronize()
    host = {k: v.cpu().numpy() for k, v in prof.items()}
    for k in ("fc", "pt", "bc", "gt", "dt"):
        assert mk.profile_digest(host[k]) == want_prof[k], f"generated profile {k} differs"
    for d, (c, x) in ((FWD, ("fc", "pt")), (BWD, ("bc", "gt"))):
        got = _gpu_schedule(dc, d, host[c], host[x], host["dt"])
        bad = [(lo, hi) for (dd, lo, hi), h in sorted(want_chunks.items())
               if dd == d and mk.chunk_digest(got, lo, hi) != h]
        assert not bad, f"direction {d}: {len(bad)} chunks of 256 differ, first {bad[:4]}"


def test_deepchain_split_launches_match_one_launch(dc):
    """The full deep-chain batch runs as several chained launches (programmatic
    dependent launch, per-launch tickets, claimed slots); its first 1,500
    instances solved alone run as one launch. The outputs are bit-identical."""
    import torch
    assert dc.dc_schedule_kernel_launches(16384, 1024) > 2
    assert dc.dc_schedule_kernel_launches(1500, 1024) == 2
    prof = dc.profile_gen(wl.config("deepchain"))
    for d, (c, x) in ((FWD, ("fc", "pt")), (BWD, ("bc", "gt"))):
        full = dc.schedule(d, prof[c], prof[x], prof["dt"])
        part = dc.schedule(d, prof[c][:1500].contiguous(), prof[x][:1500].contiguous(),
                           prof["dt"][:1500].contiguous())
        torch.cuda.synchronize()
        for k in ("makespan", "nseg", "status", "bits"):
            assert torch.equal(full[k][:1500], part[k]), (d, k)


@pytest.mark.parametrize("direction", [FWD, BWD])
def test_deepchain_every_arithmetic_path(dc, direction):
    """L = 1024 instances built to take each of the per-instance solver's five
    arithmetic paths (shifted 32-bit, the backward and forward E forms, the
    32-bit template, 64-bit), four of each, bit-exact with the oracle."""
    L = 1024
    cfg = wl.with_batch(wl.config("deepchain"), 4096)
    prof = oracle.profile_gen(cfg)
    c, x = ("fc", "pt") if direction == FWD else ("bc", "gt")
    cls = _solve_class(direction, prof[c], prof[x], prof["dt"])
    idx = [int(i) for k in (0, 1 if direction == BWD else 2) for i in np.nonzero(cls == k)[0][:4]]
    comp, xfer, dt = prof[c][idx].copy(), prof[x][idx].copy(), prof["dt"][idx].copy()
    rng = np.random.default_rng(50 + direction)
    for target in (3, 4):  # total compute past the E forms' limits
        for j in range(4):
            cc = rng.integers(1, 100, size=L)
            scale = (2**31 + 2**27) if target == 3 else 2**33
            cc = cc * (scale // int(cc.sum())) + 1
            xx = rng.integers(0, 1000, size=L) * (1 if target == 3 else 1 << 20)
            comp = np.vstack([comp, cc[None]])
            xfer = np.vstack([xfer, xx[None]])
            dt = np.append(dt, rng.integers(0, 100))
    got_cls = _solve_class(direction, comp, xfer, dt)
    want = [0] * 4 + [1 if direction == BWD else 2] * 4 + [3] * 4 + [4] * 4
    assert list(got_cls) == want, got_cls
    _check_direction(dc, direction, comp, xfer, dt, f"deep paths dir={direction}")


@pytest.mark.parametrize("L,sample", [(256, 64), (512, 16), (2048, 2)])
def test_lsweep_sampled_parity(dc, L, sample):
    """The depth sweep's inputs (deep-chain draws at depth L) over several CTAs'
    worth of instances: a sample bit-exact with the oracle, every decision replayed."""
    B = 304
    cfg = wl.lsweep_config(L, B)
    prof = oracle.profile_gen(cfg)
    for d, (c, x) in ((FWD, ("fc", "pt")), (BWD, ("bc", "gt"))):
        got = _gpu_schedule(dc, d, prof[c], prof[x], prof["dt"])
        exp = oracle.schedule_batch(d, prof[c][:sample], prof[x][:sample], prof["dt"][:sample],
                                    nthreads=NTHREADS)
        _assert_same({k: v[:sample] for k, v in got.items()}, exp, f"lsweep L={L} dir={d}")
        rep = oracle.replay_batch(d, prof[c], prof[x], prof["dt"], got["bits"], nthreads=NTHREADS)
        assert np.array_equal(rep, got["makespan"])


def test_roof_probe_runs(dc):
    import torch
    sink = torch.empty(152 * 256, dtype=torch.int32, device="cuda")
    for v in (0, 1):
        assert dc.dc_roof_int_probe(v, 152, 256, 64, sink) == dc.DC_OK
    torch.cuda.synchronize()
