"""ORIGAMI audit allocation on the GPU (kvgov_origami, fp32) against the
oracle (fp64 closed form).  Marked gpu.

Tolerance, from the arithmetic: the kernel's water level is (m - K) / S with
S a fp32 sum of m reciprocals (each correctly rounded), so its relative error
is at most about (m + 3) u, u = 2^-24; p_i = 1 - lambda / v_i adds one more
rounding, and lambda / v_i <= 1 for every audited tenant.  The tests allow
8 (n + 4) u: twice that bound with room for the order of the sum."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_09225_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"
U = 2.0 ** -24


def tol(n):
    return 8.0 * (n + 4) * U


def gpu(kv, b: W.AuditBatch):
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    v = torch.from_numpy(np.ascontiguousarray(b.values)).to(DEV)
    p, lam, u = kv.origami(v, torch.from_numpy(b.off).to(DEV), torch.from_numpy(b.budget).to(DEV), status=st)
    torch.cuda.synchronize()
    return p.cpu().numpy().astype(np.float64), lam.cpu().numpy().astype(np.float64), \
        u.cpu().numpy().astype(np.float64), int(st.item())


def check(b, p, lam, u, p_ref, lam_ref, u_ref):
    for q in range(b.n):
        s, e = int(b.off[q]), int(b.off[q + 1])
        t = tol(e - s)
        assert np.abs(p[s:e] - p_ref[s:e]).max(initial=0.0) <= t, q
        assert abs(lam[q] - lam_ref[q]) <= t * max(lam_ref[q], 1e-30), q
        assert abs(u[q] - u_ref[q]) <= t * max(abs(u_ref[q]), 1e-30), q


@pytest.mark.parametrize("seed,n_prob", [(1, 1), (2, 64), (3, 3000)])
def test_origami_ragged_matches_oracle(kv, seed, n_prob):
    b = W.audit_ragged(seed, n_prob)
    p, lam, u, st = gpu(kv, b)
    p_ref, lam_ref, u_ref, flag = oracle.origami(b.values, b.off, b.budget)
    assert st == 0 and not flag
    check(b, p, lam, u, p_ref, lam_ref, u_ref)


@pytest.mark.parametrize("seed", [11, 12])
def test_origami_thread_tiers_match_oracle(kv, seed):
    """Problems of 0 to 64 tenants, so that every CTA takes the thread-per-
    problem path and every register size (16, 32, 50, 64 slots) is used, with
    all-equal and Pareto values and budgets above n."""
    b = W.audit_ragged(seed, 4096, max_tenants=64)
    sizes = np.diff(b.off)
    assert sizes.max() <= 64 and ((sizes > 50) & (sizes <= 64)).any() and ((sizes > 32) & (sizes <= 50)).any()
    p, lam, u, st = gpu(kv, b)
    p_ref, lam_ref, u_ref, flag = oracle.origami(b.values, b.off, b.budget)
    assert st == 0 and not flag
    check(b, p, lam, u, p_ref, lam_ref, u_ref)


def test_origami_pareto_batch(kv):
    """131,072 problems of the section 5.5 setting (50 tenants, Pareto 1.29,
    K = 10): every probability within tolerance, and each problem's budget
    spent to within the rounding of its sum."""
    b = W.audit(seed=5, n_prob=131072)
    p, lam, u, st = gpu(kv, b)
    p_ref, lam_ref, u_ref, _ = oracle.origami(b.values, b.off, b.budget)
    assert st == 0
    assert np.abs(p - p_ref).max() <= tol(50)
    assert (np.abs(lam - lam_ref) <= tol(50) * lam_ref).all()
    sums = np.add.reduceat(p, b.off[:-1])
    assert np.abs(sums - 10.0).max() <= 50 * tol(50)


def test_origami_edge_cases_and_flags(kv):
    """Empty problems, K above n, K = 0, values <= 0, and flagged inputs: a NaN
    value, an infinite value, a negative budget."""
    vals = [np.zeros(0, np.float32), np.array([2, 4, 8], np.float32), np.array([5, 1], np.float32),
            np.array([-1, 0, 7], np.float32), np.array([3.0] * 10, np.float32)]
    off = np.concatenate([[0], np.cumsum([len(x) for x in vals])]).astype(np.int64)
    b = W.AuditBatch(values=np.concatenate(vals), off=off, budget=np.array([1, 3.5, 0, 1, 5], np.float32))
    p, lam, u, st = gpu(kv, b)
    p_ref, lam_ref, u_ref, flag = oracle.origami(b.values, b.off, b.budget)
    assert st == 0 and not flag
    check(b, p, lam, u, p_ref, lam_ref, u_ref)
    assert list(p[0:3]) == [1.0, 1.0, 1.0] and lam[1] == 0.0 and lam[2] == 5.0 and list(p[5:8]) == [0, 0, 1]
    for bad_vals, bad_budget in ((np.array([1, np.nan, 2], np.float32), 1.0),
                                 (np.array([1, np.inf, 2], np.float32), 1.0),
                                 (np.array([1, 3, 2], np.float32), -1.0)):
        b = W.AuditBatch(values=bad_vals, off=np.array([0, 3], np.int64), budget=np.array([bad_budget], np.float32))
        p, lam, u, st = gpu(kv, b)
        p_ref, lam_ref, _, flag = oracle.origami(b.values, b.off, b.budget)
        assert st == kv.F_BADINDEX and flag
        assert np.abs(p - p_ref).max() <= tol(3) and abs(lam[0] - lam_ref[0]) <= tol(3) * max(lam_ref[0], 1)
        assert math.isfinite(lam[0])


def test_origami_unusable_value_takes_its_cta_to_the_warp_path(kv):
    """3000 problems of 50 tenants with a NaN in problem 1000 and a zero in
    problem 2000: the batch is flagged, the two CTAs holding them solve every
    problem warp by warp, and every problem -- those two included (a NaN or a
    zero tenant gets p = 0) -- matches the oracle."""
    b = W.audit(seed=9, n_prob=3000)
    b.values[50 * 1000 + 7] = np.nan
    b.values[50 * 2000 + 3] = 0.0
    p, lam, u, st = gpu(kv, b)
    p_ref, lam_ref, u_ref, flag = oracle.origami(b.values, b.off, b.budget)
    assert st == kv.F_BADINDEX and flag
    good = np.ones(b.n, bool)
    good[1000] = False
    check_rows = np.nonzero(good)[0]
    for q in check_rows:
        s, e = int(b.off[q]), int(b.off[q + 1])
        assert np.abs(p[s:e] - p_ref[s:e]).max() <= tol(50), q
        assert abs(lam[q] - lam_ref[q]) <= tol(50) * lam_ref[q], q
    assert p[50 * 1000 + 7] == 0.0 and p[50 * 2000 + 3] == 0.0


@pytest.mark.parametrize("shift", [1, 2, 3])
def test_origami_unaligned_buffers(kv, shift):
    """Values and probabilities that do not start on a 16-byte boundary (views
    `shift` floats into larger buffers): the element-by-element staging path,
    same results as the oracle."""
    b = W.audit_ragged(13 + shift, 2000, max_tenants=64)
    n = len(b.values)
    vbuf = torch.zeros(n + 4, dtype=torch.float32, device=DEV)
    vbuf[shift:shift + n] = torch.from_numpy(b.values).to(DEV)
    pbuf = torch.full((n + 4,), -1.0, dtype=torch.float32, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    _, lam, u = kv.origami(vbuf[shift:shift + n], torch.from_numpy(b.off).to(DEV),
                           torch.from_numpy(b.budget).to(DEV), pbuf[shift:shift + n], status=st)
    torch.cuda.synchronize()
    p = pbuf.cpu().numpy().astype(np.float64)
    assert (p[:shift] == -1.0).all() and (p[shift + n:] == -1.0).all()
    p_ref, lam_ref, u_ref, flag = oracle.origami(b.values, b.off, b.budget)
    assert int(st.item()) == 0 and not flag
    check(b, p[shift:shift + n], lam.cpu().numpy().astype(np.float64), u.cpu().numpy().astype(np.float64),
          p_ref, lam_ref, u_ref)


def test_origami_large_problems_inside_small_tiles(kv):
    """Tiles of 32 problems whose values fit a warp's buffer but one of which
    has more than 64 tenants (the warp solves it in place), and problems with
    a value above 2^126 (its reciprocal is not a normal number: the warp
    solver takes it too); every problem against the oracle."""
    rng = np.random.default_rng(31)
    n_prob = 32 * 200
    sizes = np.full(n_prob, 20, np.int64)
    sizes[7::32] = rng.integers(65, 400, n_prob // 32)
    vals = (1.0 + rng.pareto(1.29, int(sizes.sum()))).astype(np.float32)
    off = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int64)
    for q in range(3, n_prob, 97):
        vals[off[q] + 1] = np.float32(2.0 ** 127)
    b = W.AuditBatch(values=vals, off=off, budget=np.full(n_prob, 5.0, np.float32))
    p, lam, u, st = gpu(kv, b)
    p_ref, lam_ref, u_ref, flag = oracle.origami(b.values, b.off, b.budget)
    assert st == 0 and not flag
    check(b, p, lam, u, p_ref, lam_ref, u_ref)


def test_origami_full_size_batch(kv):
    """The bench's batch: 2^20 problems of the section 5.5 setting (50
    tenants, Pareto 1.29, K = 10), every probability and level against the
    oracle."""
    b = W.audit(seed=2030, n_prob=1 << 20)
    p, lam, u, st = gpu(kv, b)
    p_ref, lam_ref, u_ref, _ = oracle.origami(b.values, b.off, b.budget)
    assert st == 0
    assert np.abs(p - p_ref).max() <= tol(50)
    assert (np.abs(lam - lam_ref) <= tol(50) * lam_ref).all()
    assert (np.abs(u - u_ref) <= tol(50) * np.abs(u_ref)).all()
