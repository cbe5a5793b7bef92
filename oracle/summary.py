"""Lift Phi, RMS normalisation nu, the fixed 256-dimensional summary s(.) and
cosine similarity.

Test infrastructure only (see the package docstring).

Eq. 2 (section "Condition-Aware Lifted State") defines the lifted state

    phi_t = Phi(z_t, H_t) = [nu(z_t), nu(z_t - z_a), dz_cam, dz_depth, q_t, h(H_t)]

with nu the RMS normalisation, z_a the latest exact anchor, missing condition
descriptors set to zero and the normalised timestep standing in for the phase.
Section "Kernelized Nonlinear Observation" fixes a 256-dimensional summary
s(.) used for every similarity.  The paper defers normalisation details and the
history summary to supplementary material; the readings made here:

* nu(x) = x / (rms(x) + eps_nu)                       (so nu(0) = 0)
* s(phi) = [S(phi_1), S(phi_2), cam(4), depth(4), q(1), h(7)]   (120+120+16)
  where S is a signed blocked count sketch R^N -> R^120:
  element i belongs to run floor(i/128), its bucket is run mod 120 and its
  sign is +1 / -1 from bit 31 of lowbias32(i XOR seed) (C. Wellons' published
  32-bit integer hash); S_b(x) = sqrt(120/N) * sum_{bucket(i)=b} sign(i) x_i.
  S is linear and preserves inner products in expectation.
* h(H) = [r_1, r_2, r_3, T*dq_1, T*dq_2, T*dq_3, n_bank/K] over the three
  latest exact transitions (1 = newest): r_j = rms(z_out - z_in)/rms(z_in) and
  dq_j = q_in - q_out; absent entries are 0.
* sim = cosine similarity; a zero-norm argument gives similarity 0.

Parity unpinned: these readings fix the absolute summary values; linearity,
normalisation, and the sketch's statistics are pinned by tests.
"""
import numpy as np

SKETCH_BUCKETS = 120
SKETCH_RUN = 128
COND_DIM = 4
HIST_DIM = 7
SUMMARY_DIM = 2 * SKETCH_BUCKETS + 2 * COND_DIM + 1 + HIST_DIM  # = 256

# Offsets of the summary blocks.
OFF_Z = 0
OFF_DZ = SKETCH_BUCKETS
OFF_CAM = 2 * SKETCH_BUCKETS
OFF_DEPTH = OFF_CAM + COND_DIM
OFF_Q = OFF_DEPTH + COND_DIM
OFF_H = OFF_Q + 1


def lowbias32(x):
    """C. Wellons' 'lowbias32' integer hash on uint32 (vectorised, wraps mod 2^32)."""
    x = np.array(x, dtype=np.uint32, copy=True)
    x ^= x >> np.uint32(16)
    x *= np.uint32(0x7FEB352D)
    x ^= x >> np.uint32(15)
    x *= np.uint32(0x846CA68B)
    x ^= x >> np.uint32(16)
    return x


def sketch_signs(n, seed, start=0):
    """Signs (+1/-1, fp64) of flat indices start..start+n-1."""
    idx = (np.arange(start, start + n, dtype=np.uint64) & np.uint64(0xFFFFFFFF)).astype(np.uint32)
    h = lowbias32(idx ^ np.uint32(seed & 0xFFFFFFFF))
    return np.where((h >> np.uint32(31)) != 0, -1.0, 1.0)


def sketch_buckets(n, start=0):
    """Bucket of each flat index: floor(i / 128) mod 120."""
    return (np.arange(start, start + n, dtype=np.int64) // SKETCH_RUN) % SKETCH_BUCKETS


def sketch(x, seed, chunk=1 << 24):
    """Signed blocked count sketch S(x) in R^120 (fp64), scaled by sqrt(120/N)."""
    x = np.asarray(x).reshape(-1)
    n = x.size
    out = np.zeros(SKETCH_BUCKETS, dtype=np.float64)
    if n == 0:
        return out
    for s0 in range(0, n, chunk):
        xs = x[s0:s0 + chunk].astype(np.float64)
        m = xs.size
        out += np.bincount(sketch_buckets(m, s0), weights=sketch_signs(m, seed, s0) * xs,
                           minlength=SKETCH_BUCKETS)
    return out * np.sqrt(SKETCH_BUCKETS / n)


def rms(x):
    """Root mean square (fp64)."""
    x = np.asarray(x, dtype=np.float64).reshape(-1)
    if x.size == 0:
        return 0.0
    return float(np.sqrt(np.mean(x * x)))


def nu(x, eps_nu):
    """RMS normalisation nu(x) = x / (rms(x) + eps_nu) (section "Condition-Aware Lifted State")."""
    x = np.asarray(x, dtype=np.float64)
    return x / (rms(x) + eps_nu)


def cosine(a, b):
    """Cosine similarity; 0 when either argument has zero norm."""
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    na = float(np.sqrt(np.dot(a, a)))
    nb = float(np.sqrt(np.dot(b, b)))
    if na == 0.0 or nb == 0.0:
        return 0.0
    return float(np.dot(a, b) / (na * nb))


def history_summary(records_newest_first, T, capacity):
    """h(H_t) in R^7 from the three most recent exact transitions (reading above).

    ``records_newest_first`` is a sequence of objects with attributes r, q_in,
    q_out, newest first.
    """
    h = np.zeros(HIST_DIM, dtype=np.float64)
    for j, rec in enumerate(list(records_newest_first)[:3]):
        h[j] = rec.r
        h[3 + j] = T * (rec.q_in - rec.q_out)
    h[6] = len(records_newest_first) / float(capacity)
    return h


def lift_full(z, z_a, cam, depth, q, h, eps_nu):
    """The full lifted state phi = Phi(z, H) of Eq. 2 as one vector of length 2N+16."""
    z = np.asarray(z, dtype=np.float64).reshape(-1)
    z_a = np.asarray(z_a, dtype=np.float64).reshape(-1)
    return np.concatenate([nu(z, eps_nu), nu(z - z_a, eps_nu),
                           np.asarray(cam, dtype=np.float64).reshape(COND_DIM),
                           np.asarray(depth, dtype=np.float64).reshape(COND_DIM),
                           [float(q)], np.asarray(h, dtype=np.float64).reshape(HIST_DIM)])


def summarize_full(phi, n, seed):
    """The summary s(phi) of a full lifted vector (length 2n+16): a linear map."""
    phi = np.asarray(phi, dtype=np.float64)
    return np.concatenate([sketch(phi[:n], seed), sketch(phi[n:2 * n], seed), phi[2 * n:]])


def summary_of_state(z, z_a, cam, depth, q, h, eps_nu, seed):
    """s(Phi(z, H)): the summary of the lifted state, by its definition."""
    z = np.asarray(z).reshape(-1)
    return summarize_full(lift_full(z, z_a, cam, depth, q, h, eps_nu), z.size, seed)
