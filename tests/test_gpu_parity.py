"""GPU read against the float64 oracle, element by element (needs a GB300).

Tolerances are the target's: bf16 inputs -> fp32 output within max abs 2e-2
and mean abs 2e-3 of the oracle evaluated on the same bf16-rounded inputs
upcast to double; fp32 inputs within 1e-4.  Small cases span several key
tiles with ragged tails; the five workloads run at full size and are
compared on sampled rows (the oracle's row entry point) that always include
the first rows of a head (the causal rows with the fewest keys, where the
exact fix-up applies) and the last tile.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_07160_gb300 import build, fem
from paper_2602_07160_gb300 import workloads as W

pytestmark = pytest.mark.gpu

BF16_MAX, BF16_MEAN = 2e-2, 2e-3
F32_MAX = 1e-4
LSE_MAX = 2e-3


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    return fem.load()


def _gpu_bf16(q, k, v, beta, causal):
    dev = torch.device("cuda", 0)
    qd, kd, vd, bd = (x.to(dev) for x in (q, k, v, beta))
    out = torch.full(q.shape, float("nan"), dtype=torch.float32, device=dev)  # poisoned: every element must be written
    out, lse = fem.fem_fwd(qd, kd, vd, bd, causal=causal, out=out)
    fem.check_device_error()
    return out.cpu().double().numpy(), lse.cpu().double().numpy()


def _assert_close(out, ref, max_tol=BF16_MAX, mean_tol=BF16_MEAN, what=""):
    assert np.isfinite(out).all(), f"{what}: non-finite output"
    err = np.abs(out - ref)
    mx, mn = float(err.max()), float(err.mean())
    where = np.unravel_index(int(err.argmax()), err.shape)
    assert mx <= max_tol and mn <= mean_tol, f"{what}: max {mx:.3e} at {where}, mean {mn:.3e}"
    return mx, mn


SMALL = [
    # B, H, T, d, causal
    (1, 2, 1, 64, True),
    (1, 2, 2, 128, True),
    (2, 2, 127, 64, True),
    (2, 3, 129, 128, True),
    (1, 2, 300, 128, True),
    (2, 2, 384, 64, True),
    (1, 2, 1, 128, False),
    (2, 2, 129, 64, False),
    (2, 3, 197, 64, False),
    (1, 2, 300, 128, False),
    # the last length of the one-launch pre-pass (four key tiles) and the first of the three launches
    (1, 2, 512, 64, True),
    (1, 2, 513, 128, False),
]


@pytest.mark.parametrize("B,H,T,d,causal", SMALL)
def test_small_cases_full_compare(B, H, T, d, causal):
    q, k, v, beta = W.make_custom(B, H, T, d, seed=T + d)
    out, lse = _gpu_bf16(q, k, v, beta, causal)
    ref, ref_lse = oracle.fem_read(q, k, v, beta, causal)
    _assert_close(out, ref, what=f"B{B} H{H} T{T} d{d} causal={causal}")
    assert np.abs(lse - ref_lse).max() <= LSE_MAX


BETA_SWEEP = [0.0, 1e-4, 1e-3, 1e-2, 0.1, 0.5, 1.0, 5.0, 20.0, 100.0, 1e3]


@pytest.mark.parametrize("d,causal", [(64, True), (128, True), (128, False)])
def test_beta_sweep(d, causal):
    B, H, T = 1, 2, 320
    q, k, v, _ = W.make_custom(B, H, T, d, seed=7)
    beta = W.beta_grid(H, d, BETA_SWEEP)
    out, _ = _gpu_bf16(q, k, v, beta, causal)
    ref, _ = oracle.fem_read(q, k, v, beta, causal)
    _assert_close(out, ref, what=f"beta sweep d{d} causal={causal}")


@pytest.mark.parametrize("d", [64, 128])
def test_student_t_values_wide_beta(d):
    q, k, v, beta = W.make_custom(1, 3, 520, d, beta_lo=1e-3, beta_hi=100.0, v_dist="student_t3",
                                  const_channels=4, seed=11)
    out, _ = _gpu_bf16(q, k, v, beta, True)
    ref, _ = oracle.fem_read(q, k, v, beta, True)
    _assert_close(out, ref, what="student-t")


@pytest.mark.parametrize("d", [64, 128])
def test_long_recomputations_over_key_tile_segments(d):
    """T = 16384 has 128 key tiles, so fix-up chunks that recompute rows from the first key
    tile over 16 or more tiles are split into segments of 8 tiles taken by different blocks
    and merged by the last one (heavy-tailed values and beta up to 100 list such rows, at
    every query tile).  Compared with the oracle: every row of the last two query tiles of
    each head, where the segments are most, and rows drawn at random."""
    B, H, T = 1, 2, 16384
    q, k, v, beta = W.make_custom(B, H, T, d, beta_lo=1e-3, beta_hi=100.0, v_dist="student_t3",
                                  const_channels=4, seed=21)
    out, lse = _gpu_bf16(q, k, v, beta, True)
    assert fem.last_fixup_rows() > 0
    late = np.concatenate([np.arange(hh * T + T - 256, hh * T + T) for hh in range(B * H)])
    rows = np.unique(np.concatenate([late, np.random.default_rng(5).choice(B * H * T, size=256, replace=False)]))
    ref, ref_lse = oracle.fem_read_rows(q, k, v, beta, True, rows)
    _assert_close(out.reshape(-1, d)[rows], ref, what="segments")
    assert np.abs(lse.reshape(-1)[rows] - ref_lse).max() <= LSE_MAX


@pytest.mark.parametrize("d", [64, 128])
def test_maximum_sequence_length(d):
    """T = 2^20, the longest sequence the tensor-core read takes (8192 key tiles; the fix-up
    splits at 512 tiles per segment there).  Sampled rows against the oracle: the first rows,
    rows around key-tile edges, the last rows and rows drawn at random."""
    T = 1 << 20
    q, k, v, beta = W.make_custom(1, 1, T, d, seed=31)
    dev = torch.device("cuda", 0)
    qd, kd, vd, bd = (x.to(dev) for x in (q, k, v, beta))
    out, lse = fem.fem_fwd(qd, kd, vd, bd, causal=True)
    fem.check_device_error()
    rows = np.unique(np.concatenate([np.arange(8), [127, 128, 129, 65535, 65536, 524288],
                                     np.arange(T - 8, T),
                                     np.random.default_rng(7).choice(T, size=8, replace=False)]))
    ref, ref_lse = oracle.fem_read_rows(q, k, v, beta, True, rows)
    got = out.reshape(-1, d)[torch.from_numpy(rows).to(dev)].double().cpu().numpy()
    _assert_close(got, ref, what="T = 2^20")
    got_lse = lse.reshape(-1)[torch.from_numpy(rows).to(dev)].double().cpu().numpy()
    assert np.abs(got_lse - ref_lse).max() <= LSE_MAX


def test_first_row_is_first_value_and_constant_channels():
    """P1 and P2 on the device: row 0 reads v_0; constant channels read the constant."""
    q, k, v, beta = W.make_custom(2, 2, 260, 128, beta_lo=1e-3, beta_hi=100.0, const_channels=4, seed=3)
    out, _ = _gpu_bf16(q, k, v, beta, True)
    vf = v.double().numpy()
    assert np.abs(out[:, :, 0, :] - vf[:, :, 0, :]).max() <= BF16_MAX
    assert np.abs(out[..., :4] - vf[:, :, :1, :4]).max() <= 1e-5


def test_beta_zero_is_softmax_attention():
    """beta = 0 gives the prior mean, i.e. softmax attention (checked against torch SDPA in fp32)."""
    q, k, v, _ = W.make_custom(2, 2, 300, 128, seed=5)
    beta = torch.zeros(2, 128)
    out, _ = _gpu_bf16(q, k, v, beta, True)
    ref = torch.nn.functional.scaled_dot_product_attention(q.double(), k.double(), v.double(), is_causal=True)
    _assert_close(out, ref.numpy(), what="beta=0 vs sdpa")


def test_deterministic():
    q, k, v, beta = W.make_custom(1, 2, 300, 128, seed=9)
    a, la = _gpu_bf16(q, k, v, beta, True)
    b, lb = _gpu_bf16(q, k, v, beta, True)
    assert np.array_equal(a, b) and np.array_equal(la, lb)


@pytest.mark.parametrize("d", [64, 128])
def test_timed_launch_matches_dependent_launch(d):
    """With events around the tensor-core kernel (how bench.py times it) the read and the
    fix-up are plain launches; without them they are programmatic dependent launches that
    start in the previous kernel's tail.  Both orders give the same bits, fix-up rows included."""
    q, k, v, beta = W.make_custom(2, 4, 1000, d, seed=12)
    dev = torch.device("cuda", 0)
    qd, kd, vd, bd = (x.to(dev) for x in (q, k, v, beta))
    o1, l1 = fem.fem_fwd(qd, kd, vd, bd, causal=True)
    rows1 = fem.last_fixup_rows()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()  # torch creates the CUDA events at their first record
    e1.record()
    fem.set_kernel_events(e0, e1)
    o2, l2 = fem.fem_fwd(qd, kd, vd, bd, causal=True)
    torch.cuda.synchronize()
    assert e0.elapsed_time(e1) > 0.0
    assert rows1 > 0 and fem.last_fixup_rows() == rows1
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
    fem.check_device_error()


def test_workspace_variant_matches():
    q, k, v, beta = W.make_custom(1, 2, 300, 64, seed=4)
    dev = torch.device("cuda", 0)
    qd, kd, vd, bd = (x.to(dev) for x in (q, k, v, beta))
    o1, l1 = fem.fem_fwd(qd, kd, vd, bd, causal=True)
    ws = torch.empty(fem.workspace_bytes(1, 2, 300, 64, True), dtype=torch.uint8, device=dev)
    o2, l2 = fem.fem_fwd_ws(qd, kd, vd, bd, ws, causal=True)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2) and torch.equal(l1, l2)


def test_host_entry_point_matches():
    q, k, v, beta = W.make_custom(1, 2, 300, 128, seed=6)
    dev = torch.device("cuda", 0)
    o1, l1 = fem.fem_fwd(*(x.to(dev) for x in (q, k, v, beta)), causal=True)
    o2, l2 = fem.fem_fwd_host(q.pin_memory(), k.pin_memory(), v.pin_memory(), beta.pin_memory(), causal=True)
    assert torch.equal(o1.cpu(), o2) and torch.equal(l1.cpu(), l2)


@pytest.mark.parametrize("causal", [True, False])
def test_host_entry_point_chunks(causal):
    """B = 3, H = 5: the host entry point copies and reads chunks of three and two heads per
    batch element (the very first and last chunks split into one head and the rest),
    overlapped; every chunk matches the device entry point."""
    q, k, v, beta = W.make_custom(3, 5, 200, 64, seed=9)
    dev = torch.device("cuda", 0)
    o1, l1 = fem.fem_fwd(*(x.to(dev) for x in (q, k, v, beta)), causal=causal)
    o2, l2 = fem.fem_fwd_host(q.pin_memory(), k.pin_memory(), v.pin_memory(), beta.pin_memory(), causal=causal)
    assert torch.equal(o1.cpu(), o2) and torch.equal(l1.cpu(), l2)


# ---------------------------------------------------------------------------
# fp32-input path
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("B,H,T,d,causal", [(1, 1, 64, 16, True), (1, 2, 300, 64, True), (2, 1, 130, 128, False),
                                            (1, 1, 5, 256, True), (1, 1, 33, 7, False)])
def test_f32_path(B, H, T, d, causal):
    q, k, v, beta = W.make_custom(B, H, T, d, dtype="f32", beta_lo=1e-3, beta_hi=100.0, seed=B + T)
    beta[0, 0] = 0.0
    dev = torch.device("cuda", 0)
    out, lse = fem.fem_fwd_f32(*(x.to(dev) for x in (q, k, v, beta)), causal=causal)
    ref, ref_lse = oracle.fem_read(q, k, v, beta, causal)
    _assert_close(out.cpu().double().numpy(), ref, max_tol=F32_MAX, mean_tol=F32_MAX, what="f32")
    assert np.abs(lse.cpu().double().numpy() - ref_lse).max() <= 1e-5


# ---------------------------------------------------------------------------
# The five workloads at full size
# ---------------------------------------------------------------------------
def test_workload_tiny_f32_full():
    w = W.WORKLOADS["tiny_f32_causal"]
    q, k, v, beta = W.make_inputs(w)
    dev = torch.device("cuda", 0)
    out, _ = fem.fem_fwd_f32(*(x.to(dev) for x in (q, k, v, beta)), causal=w.causal)
    ref, _ = oracle.fem_read(q, k, v, beta, w.causal)
    _assert_close(out.cpu().double().numpy(), ref, max_tol=F32_MAX, mean_tol=F32_MAX, what=w.name)


def test_workload_vit_full():
    w = W.WORKLOADS["vit_s_full_prior"]
    q, k, v, beta = W.make_inputs(w)
    out, _ = _gpu_bf16(q, k, v, beta, w.causal)
    ref, _ = oracle.fem_read(q, k, v, beta, w.causal)
    _assert_close(out, ref, what=w.name)


def _sample_rows(w, n_random, seed=0):
    rows_per_bh = w.T
    r = np.random.default_rng(seed)
    first = np.arange(min(384, w.T))                     # head (0, 0): the first three tiles
    last_bh = w.B * w.H - 1
    last = last_bh * rows_per_bh + np.arange(max(0, w.T - 128), w.T)  # last tile of the last head
    rand = r.choice(w.B * w.H * w.T, size=n_random, replace=False)
    return np.unique(np.concatenate([first, last, rand]))


@pytest.mark.parametrize("d", [64, 128])
def test_fixup_rows_of_late_diagonal_tiles(d):
    """Spikes in small-valued beta=20 channels move the bank shift in the middle
    of diagonal tiles 0, 20 and the ragged last one, so the rows before each
    spike underflow on the bank and are completed by the fix-up from the state
    the tensor-core kernel leaves before the diagonal tile (none for tile 0)."""
    B, H, T = 1, 2, 3000  # 23 full key tiles and a 56-row tail
    q, k, v, beta = W.make_custom(B, H, T, d, seed=7)
    beta[:, :8] = 20.0
    vf = v.float()
    vf[..., :8] *= 0.1
    spikes = [5, 20 * 128 + 64, 23 * 128 + 40]
    for p in spikes:
        vf[:, :, p, :8] = 3.0
    v = vf.to(torch.bfloat16).contiguous()
    out, lse = _gpu_bf16(q, k, v, beta, True)
    n_fix = fem.last_fixup_rows()
    assert n_fix >= 2 * (5 + 64 + 40), n_fix  # at least the rows before each spike, both heads
    tiles = [0, 20, 23]
    rows = np.concatenate([bh * T + np.arange(t * 128, min(T, t * 128 + 128)) for bh in range(B * H) for t in tiles])
    ref, ref_lse = oracle.fem_read_rows(q, k, v, beta, True, rows)
    got = out.reshape(-1, d)[rows]
    _assert_close(got, ref, what=f"fix-up rows d={d}")
    assert np.abs(lse.reshape(-1)[rows] - ref_lse).max() <= LSE_MAX


@pytest.mark.parametrize("name,n_random", [("lm_causal_d64", 3000), ("lm_causal_d128", 1500),
                                           ("long_causal_student_t", 600)])
def test_workload_full_size_sampled(name, n_random):
    w = W.WORKLOADS[name]
    q, k, v, beta = W.make_inputs(w)
    out, lse = _gpu_bf16(q, k, v, beta, w.causal)
    rows = _sample_rows(w, n_random)
    ref, ref_lse = oracle.fem_read_rows(q, k, v, beta, w.causal, rows)
    got = out.reshape(-1, w.d)[rows]
    _assert_close(got, ref, what=name)
    assert np.abs(lse.reshape(-1)[rows] - ref_lse).max() <= LSE_MAX
    if name == "long_causal_student_t":
        vf = v.double().numpy()
        assert np.abs(out[..., :4] - vf[:, :, :1, :4]).max() <= 1e-5
