"""Pins of the oracle's schedule (Eq. 1) and lift/summary (Eq. 2, the 256-dim
summary of section "Kernelized Nonlinear Observation") against closed forms,
invariants and independent library routines."""
import json
import os

import numpy as np
import pytest
from scipy.spatial import distance

from oracle import schedule as sch
from oracle import summary as sm

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- schedule (Eq. 1)
def test_sigmas_endpoints_and_spacing():
    s = sch.sigmas(10)
    assert s[0] == 1.0 and s[-1] == 0.0
    assert np.allclose(np.diff(s), -0.1, atol=1e-15)


def test_shift_closed_form():
    # s = 3 maps sigma = 0.5 to 3*0.5 / (1 + 2*0.5) = 0.75; endpoints fixed
    s = sch.sigmas(2, shift=3.0)
    assert s[0] == 1.0 and s[2] == 0.0
    assert abs(s[1] - 0.75) < 1e-15


def test_constant_velocity_closed_form():
    # sum of the Euler steps is sigma_T - sigma_0 = -1, so z_T = z_0 - v
    g = np.random.default_rng(0)
    z = g.standard_normal(100)
    v = g.standard_normal(100)
    s = sch.sigmas(7, shift=2.5)
    x = z.copy()
    for k in range(7):
        x = sch.psi(x, v, s[k], s[k + 1])
    assert np.allclose(x, z - v, rtol=0, atol=1e-13)


def test_linear_field_euler_product():
    # v = a z  =>  z_T = prod_k (1 + a (sigma_{k+1} - sigma_k)) z_0 = (1 - a/T)^T z_0
    a, T = 0.7, 12
    z0 = np.array([1.0, -2.0, 3.5])
    s = sch.sigmas(T)
    x = z0.copy()
    for k in range(T):
        x = sch.psi(x, a * x, s[k], s[k + 1])
    assert np.allclose(x, (1 - a / T) ** T * z0, rtol=1e-13)


def test_phase_is_normalised_timestep():
    s = sch.sigmas(5)
    assert np.array_equal(sch.phase(s), s)
    assert np.allclose(sch.model_timestep(s), 1000 * s)


# ---------------------------------------------------------------- sign hash
def test_lowbias32_fixed_point_and_bijectivity():
    assert int(sm.lowbias32(np.array([0], dtype=np.uint32))[0]) == 0
    x = np.arange(1 << 18, dtype=np.uint32) * np.uint32(2654435761)
    h = sm.lowbias32(x)
    assert np.unique(h).size == x.size          # a bijection on uint32: no collisions


def test_sign_balance():
    s = sm.sketch_signs(1 << 20, seed=0x2545F491)
    assert set(np.unique(s)) == {-1.0, 1.0}
    assert abs(np.mean(s)) < 0.01


# ---------------------------------------------------------------- sketch S
def test_sketch_is_linear():
    g = np.random.default_rng(1)
    n = 128 * 250 + 77                          # ragged tail
    x, y = g.standard_normal(n), g.standard_normal(n)
    a, b = 1.7, -0.3
    lhs = sm.sketch(a * x + b * y, 5)
    rhs = a * sm.sketch(x, 5) + b * sm.sketch(y, 5)
    assert np.allclose(lhs, rhs, rtol=0, atol=1e-11)


def test_sketch_one_hot_and_run_structure():
    n = 128 * 300
    for i in [0, 127, 128, 128 * 119 + 5, 128 * 120 + 3, n - 1]:
        x = np.zeros(n)
        x[i] = 1.0
        S = sm.sketch(x, 9)
        nz = np.flatnonzero(S)
        assert nz.tolist() == [(i // 128) % 120]
        assert abs(abs(S[nz[0]]) - np.sqrt(120.0 / n)) < 1e-15
    # runs 120 apart fall into the same bucket, with their own signs
    x = np.zeros(n)
    x[5] = 1.0
    x[5 + 128 * 120] = 1.0
    S = sm.sketch(x, 9)
    sg = sm.sketch_signs(n, 9)
    assert abs(S[0] - np.sqrt(120.0 / n) * (sg[5] + sg[5 + 128 * 120])) < 1e-15


def test_sketch_preserves_norm_in_expectation():
    # E ||S(x)||^2 = ||x||^2 * 120/N  (unit-variance buckets for nu(x))
    n = 128 * 120 * 20
    ratios = []
    for seed in range(40):
        x = np.random.default_rng(seed).standard_normal(n)
        ratios.append(np.sum(sm.sketch(x, seed + 11) ** 2) / (np.sum(x * x) * 120.0 / n))
    assert abs(np.mean(ratios) - 1.0) < 0.05


# ---------------------------------------------------------------- nu, cosine
def test_nu_normalises():
    x = np.random.default_rng(2).standard_normal(1000) * 3.0
    y = sm.nu(x, 1e-12)
    assert abs(sm.rms(y) - 1.0) < 1e-12
    assert np.allclose(sm.nu(5.0 * x, 1e-12), y, atol=1e-12)
    assert np.all(sm.nu(np.zeros(10), 1e-12) == 0.0)


def test_cosine_against_scipy():
    g = np.random.default_rng(3)
    for _ in range(5):
        a, b = g.standard_normal(256), g.standard_normal(256)
        assert abs(sm.cosine(a, b) - (1.0 - distance.cosine(a, b))) < 1e-12
    a = g.standard_normal(256)
    assert abs(sm.cosine(a, a) - 1.0) < 1e-15 and abs(sm.cosine(a, -a) + 1.0) < 1e-15
    assert sm.cosine(np.zeros(256), a) == 0.0


# ---------------------------------------------------------------- summary layout
def test_summary_layout_and_dim():
    consts = json.load(open(os.path.join(GOLDEN, "structural_constants.json")))
    assert sm.SUMMARY_DIM == consts["summary_dim"]["value"]
    g = np.random.default_rng(4)
    n = 4096
    z = g.standard_normal(n)
    cam, depth = g.standard_normal(4), g.standard_normal(4)
    h = g.standard_normal(7)
    s = sm.summary_of_state(z, z, cam, depth, 0.37, h, 1e-12, 7)
    assert s.shape == (256,)
    assert np.all(s[sm.OFF_DZ:sm.OFF_DZ + 120] == 0.0)      # z = z_a: no displacement
    assert np.array_equal(s[sm.OFF_CAM:sm.OFF_CAM + 4], cam)
    assert np.array_equal(s[sm.OFF_DEPTH:sm.OFF_DEPTH + 4], depth)
    assert s[sm.OFF_Q] == 0.37
    assert np.array_equal(s[sm.OFF_H:], h)
    assert np.allclose(s[:120], sm.sketch(z / sm.rms(z), 7), atol=1e-12)


def test_summary_uses_linear_shortcut_consistently():
    # S(nu(z - z_a)) = (S(z) - S(z_a)) / rms(z - z_a): what the fused kernels use
    g = np.random.default_rng(5)
    n = 128 * 77 + 9
    z, za = g.standard_normal(n), g.standard_normal(n)
    s = sm.summary_of_state(z, za, np.zeros(4), np.zeros(4), 0.5, np.zeros(7), 1e-12, 3)
    want = (sm.sketch(z, 3) - sm.sketch(za, 3)) / (sm.rms(z - za) + 1e-12)
    assert np.allclose(s[sm.OFF_DZ:sm.OFF_DZ + 120], want, atol=1e-12)


def test_history_summary():
    class R:
        def __init__(self, r, qi, qo):
            self.r, self.q_in, self.q_out = r, qi, qo
    recs = [R(0.1, 0.9, 0.8), R(0.2, 0.7, 0.6)]      # newest first
    h = sm.history_summary(recs, T=10, capacity=4)
    assert np.allclose(h, [0.1, 0.2, 0.0, 1.0, 1.0, 0.0, 0.5], atol=1e-12)
    assert np.all(sm.history_summary([], 10, 4) == 0.0)
