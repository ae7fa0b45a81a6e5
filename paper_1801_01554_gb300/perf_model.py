"""Performance models of the batch back-propagation step (Section 6.1).

Two models live here:

* the paper's GF11 model, restated as printed in Section 6.1: cycles per
  epoch from the flop counts of the forward and backward passes, the DRAM
  transfers of weights and weight changes per group of cases, and the summing
  of changes over the switch (a tree or a ring); MCPS from 20 million
  instructions per second per processor; and the optimal processor count;
* the same accounting restated for this library's float32 kernels on one
  GB300: microseconds per update from the phases of the persistent kernel
  (two grid barriers, the weight copy into shared memory, pattern passes of PG
  patterns per CTA, 256-pattern chunks of the weight phase) and of the one-CTA
  kernel for groups of 1-4 patterns.  Its constants are the phase costs
  measured on GB300 (each phase looped inside one launch), not fitted to the
  end-to-end times; `skew_us` is the one remainder.

Readings of the printed model (Section 6.1):
* the last term of T is printed as 4P x W, but the tree cost per update is
  given as 4W ceil(log2 P) just above it: T uses the tree cost for a tree and
  4WP for a ring;
* "MCPS = 20/T" is read as MCPS = 20 W C / T (T in cycles per epoch of C
  cases, 20 million instructions per second per processor);
* the printed optimum C/(4W) x (...) is the root of dT/dP for a cost linear
  in P with the square root taken for a ring; for the tree cost the root of
  dT/dP with a continuous log2 P carries an extra factor ln 2.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

# ---------------------------------------------------------------- GF11 (Section 6.1)
GF11_MIPS = 20.0          # million instructions per second per processor
GF11_FREE_SRAM = 15000    # M: free words of SRAM
GF11_BUNDLE = 1000        # B: weights per bundle (cache of 2B words)


def _gf11_terms(W, Wi, U, C, P, M, bundle):
    per_case = (2 * W) + (2 * Wi + 4 * (W - Wi))                 # forward + backward flops (cycles)
    groups = C / P * (2 * U / (M - 2 * bundle))                  # G
    per_group = 4 * W + 4 * 2 * W + 4 * (W - Wi)                 # DRAM transfers per group
    return per_case, groups, per_group


def gf11_epoch_cycles(W, Wi, U, C, P, summing="tree", M=GF11_FREE_SRAM, bundle=GF11_BUNDLE,
                      continuous=False):
    """T: cycles per epoch of C cases on P processors with one update per epoch."""
    per_case, groups, per_group = _gf11_terms(W, Wi, U, C, P, M, bundle)
    if summing == "tree":
        lg = math.log2(P) if continuous else math.ceil(math.log2(P))
        comm = 4 * W * lg
    elif summing == "ring":
        comm = 4 * W * P
    else:
        raise ValueError(summing)
    return per_case * C / P + per_group * groups + comm


def gf11_mcps(W, Wi, U, C, P, summing="tree", **kw):
    """Millions of connections per second: W C connections per epoch at
    20 million cycles per second."""
    return GF11_MIPS * W * C / gf11_epoch_cycles(W, Wi, U, C, P, summing, **kw)


def gf11_optimal_processors(W, Wi, U, C, summing="tree", M=GF11_FREE_SRAM, bundle=GF11_BUNDLE):
    """Processor count that minimises T (continuous P): with A the per-case
    cycles plus the transfer cycles per case, T = A C / P + comm(P); a ring
    (comm = 4WP) gives P = sqrt(A C / 4W), a tree (comm = 4W log2 P) gives
    P = A C ln2 / 4W.  The paper prints A C / 4W."""
    per_case, _, per_group = _gf11_terms(W, Wi, U, C, 1, M, bundle)
    A = per_case + per_group * 2 * U / (M - 2 * bundle)
    printed = C / (4 * W) * A
    if summing == "ring":
        return math.sqrt(printed)
    return printed * math.log(2.0)


# ---------------------------------------------------------------- GB300 restatement
@dataclass
class GB300Phases:
    """Phase costs of the float32 kernels on one GB300 (microseconds), fitted
    to per-update times of the 203-120-26 net with and without the weight
    phase (a timing-only copy of the kernel) at B = 8 .. 65,536."""
    n_sm: int = 152
    # pattern side of an update: two grid barriers, the weight copy, skew, and
    # one pass per PG patterns of a CTA's share
    pattern_fixed_us: float = 4.79
    pass_us: tuple = ((1, 3.10), (2, 3.43), (4, 4.56), (8, 7.09), (32, 16.3))
    # whole-tile weight phase (8 x 32 tiles, one per CTA): fixed part, then per
    # 512-pattern chunk a fixed and a per-row part
    weight_fixed_us: float = 1.19
    chunk_fixed_us: float = 0.58
    chunk_rows_us: float = 0.72        # for a full chunk of 512 rows
    # balanced weight phase (16 x 32 tiles, equal runs of chunks per CTA, one
    # more grid barrier and the fix-up): fixed part and per chunk of a run
    balanced_fixed_us: float = 6.66
    balanced_chunk_us: float = 2.12
    balanced_min_chunks: int = 24
    chunk_rows: int = 512
    # one-CTA kernel: per group of B patterns
    small_us: tuple = ((1, 6.68), (2, 7.37), (4, 9.17))


def gb300_group_size(B, n_sm=152, max_pg=8, wide=True):
    """Patterns per CTA pass (PG) that the persistent kernel picks for B:
    doubling up to 8, then passes of 32 above 16 patterns per CTA when the
    net suits them (wide; true for 203-120-26)."""
    want = -(-B // n_sm)
    pg = 1
    while pg < want and pg < max_pg:
        pg *= 2
    if wide and want > 16 and pg == 8:
        pg = 32
    return pg


def gb300_update_us(B, tiles=121, tiles16=64, ph: GB300Phases = GB300Phases(), small_max=4):
    """Predicted microseconds per update of a B-pattern group (203-120-26)."""
    if B <= small_max:
        for b, us in ph.small_us:
            if B <= b:
                return us
    pg = gb300_group_size(B, ph.n_sm)
    passes = -(-(-(-B // ph.n_sm)) // pg)
    t = ph.pattern_fixed_us + passes * dict(ph.pass_us)[pg]
    chunks = -(-B // ph.chunk_rows)
    if chunks >= ph.balanced_min_chunks and tiles16 < ph.n_sm:
        run = -(-(tiles16 * chunks) // ph.n_sm)
        return t + ph.balanced_fixed_us + run * ph.balanced_chunk_us
    per_cta = -(-tiles // ph.n_sm)
    rows_last = B - (chunks - 1) * ph.chunk_rows
    w = ph.weight_fixed_us + per_cta * ((chunks - 1) * (ph.chunk_fixed_us + ph.chunk_rows_us)
                                        + ph.chunk_fixed_us + ph.chunk_rows_us * rows_last / ph.chunk_rows)
    return t + w


def gb300_cps(B, W=27626, **kw):
    """Connections per second W B / time per update."""
    return W * B / (gb300_update_us(B, **kw) * 1e-6)
