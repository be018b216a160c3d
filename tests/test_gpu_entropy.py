"""GPU parity of the entropy test (kvr_entropy_*) against the fp64 oracle.

Per token and row the kernel's H_e must match the oracle's within
2e-5 * (1 + H): the logits are read exactly, and the kernel's fp32 sums of
up to 64 terms per thread, its base-2 exponentials (relative error about
2^-22) and the merges of about 15 partials bound the relative error of
sum 2^(y - m) and of its weighted twin by about 5e-6, which moves H by at
most 5e-6 * (1 + H).  The moving mean and the stop position are decided in
fp32 from those entropies; the mean is checked against the fp64 detector's
within 2e-5 * (1 + m) + 4e-6 * m, and the stop position against the fp64
detector's, except for rows whose fp64 mean came within that tolerance of
tau at a tested position (either decision is correct there).  The number of
such rows is bounded in every run.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import entropy as ent
from paper_2608_15797_gb300 import inputs

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from paper_2608_15797_gb300 import kvr


def _tol(h):
    return 2e-5 * (1.0 + np.abs(h))


def _to_dev(x, dtype, stride=None):
    t = torch.from_numpy(np.ascontiguousarray(x, np.float32))
    t = t.to(torch.bfloat16 if dtype == "bf16" else torch.float32)
    if stride is not None and stride != x.shape[1]:
        pad = torch.zeros(x.shape[0], stride, dtype=t.dtype)
        pad[:, :x.shape[1]] = t
        return pad.cuda()[:, :x.shape[1]]
    return t.cuda()


def _sigma_schedule(rows, e):
    """Per-row spreads at generated position e (0-based): confident rows,
    incoherent rows, rows drifting across the threshold, and rows near it."""
    s = np.empty(rows, np.float32)
    for r in range(rows):
        kind = r % 4
        if kind == 0:
            s[r] = 4.2
        elif kind == 1:
            s[r] = 2.0
        elif kind == 2:
            s[r] = 3.6 - 0.9 * min(1.0, e / (30.0 + 3 * r))
        else:
            s[r] = 3.05 + 0.02 * (r % 7)
    return s


def _mean_tol(m):
    # each entropy within _tol, and the kernel's fp32 window sum of at most
    # 64 of them adds about 64 * 2^-24 relative
    return 2e-5 * (1.0 + np.abs(m)) + 4e-6 * np.abs(m)


def run_lockstep(rows, vocab, steps, dtype="bf16", stride=None, window=12,
                 guard=24, tau=7.0, temperature=1.0, seed=0, offset=None,
                 resets=(), kernel=0):
    """Drive the kernel and the fp64 oracle through `steps` tokens; check
    every output.  Returns (exempt, stops): the number of rows whose fp64
    moving mean came within the mean tolerance of tau at a tested position
    (their stop position is exempt from the comparison from then on, since
    either decision is correct there), and the kernel's stop positions."""
    det = kvr.EntropyDetector(rows, vocab, window, guard, tau, temperature,
                              dtype)
    det.set_kernel(kernel)
    ref = ent.EntropyDetector(rows, window, guard, tau)
    hist32 = [[] for _ in range(rows)]  # the kernel's entropies, per row
    stop_k = np.zeros(rows, np.int64)
    tied = np.zeros(rows, bool)
    for e in range(steps):
        for (at, b, en) in resets:
            if at == e:
                det.reset(b, en)
                ref.reset(b, en)
                for r in range(b, en):
                    hist32[r] = []
                    stop_k[r] = 0
                    tied[r] = False
        x = inputs.candidate_logits(seed, e, rows, vocab,
                                    _sigma_schedule(rows, e), boost=0.0,
                                    dtype=dtype)
        if offset is not None:
            x = inputs.round_to(x + np.float32(offset), dtype)
        H_ref = ent.token_entropy(x, temperature)
        H, mean, stopped = det.step(_to_dev(x, dtype, stride))
        H = H.cpu().numpy()
        mean = mean.cpu().numpy()
        stopped = stopped.cpu().numpy()
        live_k = stop_k == 0           # rows the kernel ran this token
        live_ref = ref.stop == 0       # rows the fp64 detector runs
        # stopped rows report NaN and are not read
        assert np.all(np.isnan(H[~live_k])) and np.all(np.isnan(mean[~live_k]))
        err = np.abs(H[live_k].astype(np.float64) - H_ref[live_k])
        assert np.all(err <= _tol(H_ref[live_k])), (e, err.max())
        for r in np.nonzero(live_k)[0]:
            hist32[r].append(np.float32(H[r]))
        # the fp64 detector on the oracle's entropies (Sec. 3.2)
        m64, _ = ref.step(np.where(live_ref, H_ref, 0.0))
        for r in np.nonzero(live_k & live_ref & ~tied)[0]:
            assert abs(mean[r] - m64[r]) <= _mean_tol(m64[r]), \
                (e, r, mean[r], m64[r])
            if len(ref.hist[r]) > guard and \
                    abs(m64[r] - tau) <= _mean_tol(tau):
                tied[r] = True
        # the stop position is sticky, and set only at the current position
        assert np.array_equal(stopped[~live_k], stop_k[~live_k])
        for r in np.nonzero(live_k)[0]:
            assert stopped[r] in (0, len(hist32[r])), (e, r, stopped[r])
        stop_k = stopped.astype(np.int64)
        for r in np.nonzero(~tied)[0]:
            assert ref.stop[r] == stop_k[r], (e, r, ref.stop[r], stop_k[r])
    det.sync_status()
    exported = det.export()
    assert np.array_equal(exported[2], stop_k)
    for r in range(rows):
        n = min(len(hist32[r]), window)
        assert exported[1][r] == len(hist32[r])
        assert np.array_equal(exported[0][r, :n],
                              np.array(hist32[r][-n:] if n else [], np.float32))
    # Exemptions are rare: at most the quarter of rows the schedule keeps
    # near tau, plus two.
    exempt = int(tied.sum())
    assert exempt <= rows // 4 + 2, exempt
    return exempt, stop_k


KERNELS = {"stream": 1, "pieces": 2}


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("vocab", [7, 1000, 16385, 40000])
def test_entropy_lockstep_shapes(dtype, vocab, kernel):
    exempt, stops = run_lockstep(12, vocab, 40, dtype, kernel=KERNELS[kernel])
    assert exempt <= 6


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("rows", [1, 3, 200])
def test_entropy_row_counts(rows, kernel):
    """One row spread over many CTAs' segments, and many rows."""
    run_lockstep(rows, 33333, 27, "bf16", kernel=KERNELS[kernel])


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_entropy_qwen_vocab(dtype, kernel):
    exempt, stops = run_lockstep(16, inputs.VOCAB, 40, dtype,
                               kernel=KERNELS[kernel])
    assert exempt <= 8
    # the schedule's incoherent rows stop at the first tested position
    assert all(stops[r] == 25 for r in range(1, 16, 4))
    assert all(stops[r] == 0 for r in range(0, 16, 4))


@pytest.mark.parametrize("dtype,stride", [("bf16", 1001), ("bf16", 1003),
                                          ("bf16", 1016), ("f32", 1001),
                                          ("f32", 1008)])
def test_entropy_padded_and_unaligned_rows(dtype, stride):
    run_lockstep(8, 1000, 30, dtype, stride=stride)


def test_entropy_temperature_window_guard_variants():
    run_lockstep(8, 5000, 30, "bf16", window=1, guard=0, tau=6.5)
    run_lockstep(8, 5000, 30, "f32", window=64, guard=3, tau=7.5,
                 temperature=0.8)
    run_lockstep(8, 5000, 30, "bf16", temperature=1.7)


def test_entropy_large_logit_offset():
    # logits around +-900: the max shift keeps every term finite
    run_lockstep(8, 3000, 26, "f32", offset=900.0)
    run_lockstep(8, 3000, 26, "f32", offset=-900.0)


@pytest.mark.parametrize("kernel", KERNELS)
def test_entropy_reset_rows(kernel):
    run_lockstep(8, 2000, 60, "bf16", resets=((30, 1, 3), (45, 0, 8)),
                 kernel=KERNELS[kernel])


@pytest.mark.parametrize("kernel", KERNELS)
def test_entropy_full_size_sampled(kernel):
    """The bench's launch: 512 rows of 152,064 bf16 logits (64 problems x 8
    candidates), every row checked against the oracle for 3 tokens."""
    rows, V = 512, inputs.VOCAB
    det = kvr.EntropyDetector(rows, V)
    det.set_kernel(KERNELS[kernel])
    gen = torch.Generator(device="cuda")
    gen.manual_seed(5)
    sig = torch.linspace(1.5, 5.0, rows, device="cuda").unsqueeze(1)
    for e in range(3):
        x = (torch.randn(rows, V, generator=gen, device="cuda") * sig).to(
            torch.bfloat16)
        H, mean, stopped = det.step(x)
        H_ref = ent.token_entropy(x.float().cpu().numpy())
        err = np.abs(H.cpu().numpy().astype(np.float64) - H_ref)
        assert np.all(err <= _tol(H_ref)), err.max()
    assert det.launch_count() == 3
    det.sync_status()


def test_entropy_golden_on_gpu(golden_dir):
    with open(os.path.join(golden_dir, "entropy_detector_worked.json")) as f:
        g = json.load(f)
    rows = g["rows"]
    ks = []
    for r in rows:
        k = []
        for count, kk in r["segments"]:
            k += [kk] * count
        ks.append(k)
    V = g["vocab"]
    det = kvr.EntropyDetector(len(rows), V, g["window"], g["guard"], g["tau"],
                              1.0, "f32")
    for e in range(max(len(k) for k in ks)):
        x = torch.full((len(rows), V), float("-inf"))
        for r, k in enumerate(ks):
            x[r, :k[min(e, len(k) - 1)]] = 0.0
        H, _, stopped = det.step(x.cuda())
        H = H.cpu().numpy()
        for r, k in enumerate(ks):
            if not np.isnan(H[r]):
                want = math.log(k[min(e, len(k) - 1)])
                assert abs(H[r] - want) <= _tol(want)
    assert list(stopped.cpu().numpy()) == [r["stop"] for r in rows]
    det.sync_status()


def test_entropy_nonfinite_rows_and_determinism():
    rows, V = 6, 20000
    det = kvr.EntropyDetector(rows, V, logits_dtype="f32")
    x = torch.randn(rows, V) * 3
    x[1, 777] = float("nan")
    x[2, 5] = float("inf")
    x[3, :] = float("-inf")
    x[4, 100:] = float("-inf")  # masked tokens are fine
    xd = x.cuda()
    H1, _, _ = det.step(xd)
    H1 = H1.cpu().numpy()
    assert np.isnan(H1[1]) and np.isnan(H1[2]) and np.isnan(H1[3])
    ref = ent.token_entropy(x[[0, 4, 5]].numpy())
    assert np.all(np.abs(H1[[0, 4, 5]] - ref) <= _tol(ref))
    with pytest.raises(kvr.KvrError) as ei:
        det.sync_status()
    assert ei.value.status == kvr.KVR_EDEVICE
    det.sync_status()  # the word was cleared
    # bitwise reproducible
    det2 = kvr.EntropyDetector(rows, V, logits_dtype="f32")
    x[1:4] = 0.0
    H2, _, _ = det2.step(x.cuda())
    H3, _, _ = det2.step(x.cuda())
    assert torch.equal(H2, H3)


def test_entropy_stopped_rows_are_not_read():
    rows, V = 4, 4096
    det = kvr.EntropyDetector(rows, V, window=2, guard=1, tau=5.0,
                              logits_dtype="f32")
    flat = torch.zeros(rows, V)  # H = ln 4096 = 8.3 > 5
    flat[2:] = torch.randn(2, V) * 6  # low entropy
    for _ in range(2):
        _, _, stopped = det.step(flat.cuda())
    assert list(stopped.cpu().numpy()) == [2, 2, 0, 0]
    poison = flat.clone()
    poison[:2] = float("nan")  # a stopped row's logits are never read
    H, mean, stopped = det.step(poison.cuda())
    assert torch.isnan(H[:2]).all() and torch.isnan(mean[:2]).all()
    assert list(stopped.cpu().numpy()) == [2, 2, 0, 0]
    det.sync_status()
    det.reset(0, 1)
    _, _, stopped = det.step(flat.cuda())
    assert list(stopped.cpu().numpy()) == [0, 2, 0, 0]
    hist, count, st = det.export()
    assert list(count) == [1, 2, 4, 4] and list(st) == [0, 2, 0, 0]


def test_entropy_argument_errors():
    d = kvr.kvr_entropy_desc(4, 100, 12, 24, 7.0, 1.0, kvr.KVR_BF16)
    for bad in [kvr.kvr_entropy_desc(0, 100, 12, 24, 7.0, 1.0, 0),
                kvr.kvr_entropy_desc(4, 0, 12, 24, 7.0, 1.0, 0),
                kvr.kvr_entropy_desc(4, 100, 0, 24, 7.0, 1.0, 0),
                kvr.kvr_entropy_desc(4, 100, 65, 24, 7.0, 1.0, 0),
                kvr.kvr_entropy_desc(4, 100, 12, -1, 7.0, 1.0, 0),
                kvr.kvr_entropy_desc(4, 100, 12, 24, 7.0, -1.0, 0),
                kvr.kvr_entropy_desc(4, 100, 12, 24, 7.0, 1.0, 7)]:
        assert kvr.kvr_entropy_required_bytes(bad) == 0
    need = kvr.kvr_entropy_required_bytes(d)
    buf = torch.empty(need, dtype=torch.uint8, device="cuda")
    with pytest.raises(kvr.KvrError) as ei:
        kvr.kvr_entropy_create(d, buf, need - 1)
    assert ei.value.status == kvr.KVR_ENOMEM
    h = kvr.kvr_entropy_create(d, buf, need)
    x = torch.zeros(4, 128, dtype=torch.bfloat16, device="cuda")
    for args in [(None, 128), (x, 99)]:
        with pytest.raises(kvr.KvrError) as ei:
            kvr.kvr_entropy_step(h, *args)
        assert ei.value.status == kvr.KVR_EINVAL
    with pytest.raises(kvr.KvrError) as ei:  # odd address for bf16
        kvr.kvr_entropy_step(h, x.data_ptr() + 1, 128)
    assert ei.value.status == kvr.KVR_EINVAL
    for b, e in [(-1, 2), (0, 5), (3, 2)]:
        with pytest.raises(kvr.KvrError):
            kvr.kvr_entropy_reset(h, b, e)
    kvr.kvr_entropy_reset(h, 1, 1)
    kvr.kvr_entropy_sync_status(h)
    kvr.kvr_entropy_destroy(h)
