"""Configuration records for the oracle (test infrastructure only).

The paper prints the structure of every equation but defers its constants to
supplementary material that is not available.  The defaults below are the
readings this implementation adopts; the tests pass the same values explicitly
to both the oracle and the CUDA path, so the defaults here are never shared
code with the product.
"""
from dataclasses import dataclass, asdict

# Ablation variants of the method (Tables 3 and 4, section "Ablation Study"):
# bit flags of CacheParams.flags.  Their definitions are in oracle/ablation.py.
ABL_PERIODIC = 0x01       # controller: periodic placement at a fixed period
ABL_SECANT = 0x02         # surrogate: native latent secant
ABL_INSTANT_RISK = 0x04   # instantaneous risk (no accumulation, lambda = 0)
ABL_NO_IMPACT = 0x08      # w/o impact weighting (w = 1)
ABL_NO_CALIB = 0x10       # w/o counterfactual calibration (eta_d fixed)
ABL_NO_SUPPORT = 0x20     # w/o support constraint
ABL_LINEAR_OBS = 0x40     # linear observation instead of Eq. 5's kernel
ABL_NO_COND = 0x80        # lifted surrogate without condition descriptors
ABL_ALL = 0xFF
# Residual reading of Eq. 5 (a reading, not an ablation; see
# oracle/surrogate.observe_residual).
OBS_RESIDUAL = 0x100


@dataclass
class CacheParams:
    # Memory and retrieval (Eq. 3-5, section "Local Lifted Evolution").
    bank_capacity: int = 4        # FIFO capacity K of the exact-transition bank
    min_support: int = 1          # |N_t| that counts as enough retrieval support (Eq. 10 text)
    sim_min: float = 0.0          # compatibility: sim(s(phi_t), s(phi_in)) >= sim_min
    q_gap_max: float = 0.25       # compatibility: |q_t - q_in| <= q_gap_max
    gamma_q: float = 10.0         # phase penalty in the retrieval score (Eq. 3)
    tau_in: float = 0.1           # retrieval temperature (Eq. 3)
    tau_obs: float = 0.05         # observation temperature tau (Eq. 5)
    alpha_min: float = 0.5        # clip bounds of the scheduler scaling (Eq. 4)
    alpha_max: float = 2.0
    eps: float = 1e-8             # epsilon of Eq. 4, 7, 8
    eps_nu: float = 1e-12         # epsilon of the RMS normalisation nu(.)
    sketch_seed: int = 0x2545F491 # seed of the summary's sign hash
    # Defect proxy and calibration (Eq. 6-8).
    w_z: float = 1.0
    w_age: float = 0.05
    w_phase: float = 1.0
    w_cam: float = 0.5
    w_depth: float = 0.5
    eta_init: float = 1.0
    eta_min: float = 0.1
    eta_max: float = 10.0
    beta_d: float = 0.8
    # Risk accumulation and decision (Eq. 9-10).
    a_cam: float = 0.5
    a_depth: float = 0.5
    a_phase: float = 1.0
    lam: float = 0.9
    tau_risk: float = 0.5
    max_age: int = 6              # largest pre-decision anchor age that allows a candidate (Eq. 10 text)
    n_init_exact: int = 1         # mandatory-exact initialisation steps
    n_final_exact: int = 0        # mandatory-exact refinement steps at the end
    # Ablation variants (Tables 3 and 4).
    flags: int = 0                # ABL_* bits, OBS_RESIDUAL; 0 = the full method as printed
    period: int = 8               # ABL_PERIODIC: one exact step every `period` steps
    ridge: float = 1e-6           # ABL_LINEAR_OBS: ridge, relative to mean diag of the Gram matrix

    def has(self, flag):
        return bool(self.flags & flag)

    def as_dict(self):
        return asdict(self)


@dataclass
class DiTConfig:
    layers: int = 2
    hidden: int = 256
    heads: int = 4
    head_dim: int = 64
    mlp: int = 1024
    temb_dim: int = 256
    freq_dim: int = 256           # width of the sinusoidal timestep features
    in_ch: int = 16
    frames: int = 4
    height: int = 16
    width: int = 16
    patch: int = 2
    cond_tokens: int = 16
    cond_dim: int = 256
    dual_stream: int = 0

    @property
    def video_tokens(self):
        return self.frames * (self.height // self.patch) * (self.width // self.patch)

    @property
    def tokens(self):
        return self.cond_tokens + self.video_tokens

    @property
    def patch_dim(self):
        return self.in_ch * self.patch * self.patch

    @property
    def latent_numel(self):
        return self.in_ch * self.frames * self.height * self.width

    def as_dict(self):
        return asdict(self)
