"""Plain oracle of the ADT-Tree depth / width controller (Sec. 4.1, 4.2).

TEST INFRASTRUCTURE: only tests, smoke() and bench's CPU-baseline leg use it.

Per image, for the draft tree that will emit grid position pos = (i, j):
  1. initialise (d~, k~) from a neighbour (Sec. 4.1):
       horizontal repeat - the tree that emitted (i, j-1), i.e. the raster
                           predecessor pos-1 (also across a row end);
       vertical repeat   - the tree that emitted (i-1, j); horizontal when
                           i = 0 or that position is not generated yet;
       random            - d~ ~ U{d_lo..d_hi}, k~ ~ U{k_lo..k_hi};
       TokenFlock        - (the alternative of Table 3) the set Omega of
                           generated positions t_j before pos within
                           Euclidean distance delta, x the column and y the
                           row; d~ = sum d_j w_j / sum w_j with
                           w_j = (delta - (y_i - y_j) + 1) / delta (norm()
                           read as dividing by the sum of the weights), k~
                           likewise, each rounded half up;
     the first tree of an image uses (d0, k0); fix_d / fix_k pin d~ / k~
     (the fixed-value ablations of Table 3).
  2. bisect with the acceptance rate alpha = a / d of the previous tree
     (Eq. 2): alpha >= beta -> (d~ + l_d, k~ - l_k), else (d~ - l_d, k~ + l_k);
     the first tree has no previous alpha and keeps (d~, k~).
  3. clamp (end of Sec. 4.2): depth to [d_lo, d_hi]; width to [k_lo, k_hi]
     when clamp_k_always or the bisected depth d~ +- l_d exceeds 1,
     otherwise only to [1, k_cap].
The paper's open bounds d in (0, 10), k in (3, 14) (Anole) are the closed
ranges [1, 9] and [4, 13] here.

Random initialisation draws from SplitMix64 (Steele, Lea and Flood, OOPSLA
2014) with counter 2*pos (depth) and 2*pos+1 (width) added to the seed.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from fractions import Fraction

INIT_HORIZONTAL = 0
INIT_VERTICAL = 1
INIT_RANDOM = 2
INIT_TOKENFLOCK = 3

_MASK = (1 << 64) - 1
_GAMMA = 0x9E3779B97F4A7C15


def splitmix64(state: int) -> int:
    """One SplitMix64 output for the given 64-bit state (after the gamma step)."""
    z = (state + _GAMMA) & _MASK
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK
    return z ^ (z >> 31)


def counter_draw(seed: int, counter: int) -> int:
    return splitmix64((seed + counter * _GAMMA) & _MASK)


@dataclass
class CtrlParams:
    beta: float = 1.0
    l_d: int = 1
    l_k: int = 3
    d_lo: int = 1
    d_hi: int = 9
    k_lo: int = 4
    k_hi: int = 13
    init_mode: int = INIT_HORIZONTAL
    d0: int = 5
    k0: int = 10
    clamp_k_always: bool = True
    k_cap: int = 64
    fix_d: int = 0
    fix_k: int = 0
    seed: int = 0
    flock_delta: int = 2


def anole_params(**kw) -> CtrlParams:
    """Sec. 5.1 (Anole): beta=1, l_d=1, l_k=3, d in (0,10), k in (3,14)."""
    return CtrlParams(beta=1.0, l_d=1, l_k=3, d_lo=1, d_hi=9, k_lo=4, k_hi=13, **kw)


def llamagen_params(**kw) -> CtrlParams:
    """Sec. 5.1 (LlamaGen): beta=1, l_d=1, l_k=10, d in (0,10), k in (3,40)."""
    return CtrlParams(beta=1.0, l_d=1, l_k=10, d_lo=1, d_hi=9, k_lo=4, k_hi=39, **kw)


def _clamp(x: int, lo: int, hi: int) -> int:
    return lo if x < lo else hi if x > hi else x


@dataclass
class Controller:
    params: CtrlParams
    grid_h: int
    grid_w: int
    d_grid: list = field(default_factory=list)
    k_grid: list = field(default_factory=list)
    alpha_prev: float | None = None
    cur: tuple | None = None

    def __post_init__(self):
        n = self.grid_h * self.grid_w
        self.d_grid = [0] * n
        self.k_grid = [0] * n

    def next(self, pos: int):
        P = self.params
        n = self.grid_h * self.grid_w
        if not (0 <= pos < n):
            raise ValueError("pos outside the grid")
        i = pos // self.grid_w
        flock = self._flock(pos) if P.init_mode == INIT_TOKENFLOCK else None
        if P.init_mode == INIT_TOKENFLOCK:
            d_t, k_t = flock if flock is not None else (P.d0, P.k0)
        elif P.init_mode == INIT_RANDOM:
            d_t = P.d_lo + counter_draw(P.seed, 2 * pos) % (P.d_hi - P.d_lo + 1)
            k_t = P.k_lo + counter_draw(P.seed, 2 * pos + 1) % (P.k_hi - P.k_lo + 1)
        elif P.init_mode == INIT_VERTICAL and i >= 1 and self.d_grid[pos - self.grid_w] > 0:
            d_t, k_t = self.d_grid[pos - self.grid_w], self.k_grid[pos - self.grid_w]
        elif pos >= 1 and self.d_grid[pos - 1] > 0:
            d_t, k_t = self.d_grid[pos - 1], self.k_grid[pos - 1]
        else:
            d_t, k_t = P.d0, P.k0
        if P.fix_d > 0:
            d_t = P.fix_d
        if P.fix_k > 0:
            k_t = P.fix_k
        if self.alpha_prev is None:
            d, k = d_t, k_t
        elif self.alpha_prev >= P.beta:
            d, k = d_t + P.l_d, k_t - P.l_k
        else:
            d, k = d_t - P.l_d, k_t + P.l_k
        restrict_k = P.clamp_k_always or d > 1
        d = _clamp(d, P.d_lo, P.d_hi)
        k = _clamp(k, P.k_lo, P.k_hi) if restrict_k else _clamp(k, 1, P.k_cap)
        self.cur = (d, k)
        return d, k

    def _flock(self, pos: int):
        """TokenFlock's weighted mean over Omega (exact fractions, rounded
        half up), or None when Omega is empty."""
        delta = self.params.flock_delta
        y_i, x_i = divmod(pos, self.grid_w)
        num_d, num_k, den = Fraction(0), Fraction(0), Fraction(0)
        for q in range(pos):  # j < i: the positions generated before
            y_j, x_j = divmod(q, self.grid_w)
            if (x_i - x_j) ** 2 + (y_i - y_j) ** 2 > delta ** 2 or self.d_grid[q] == 0:
                continue
            w = Fraction(delta - (y_i - y_j) + 1, delta)
            num_d += self.d_grid[q] * w
            num_k += self.k_grid[q] * w
            den += w
        if den == 0:
            return None
        half_up = lambda f: (f + Fraction(1, 2)).__floor__()
        return half_up(num_d / den), half_up(num_k / den)

    def update(self, pos: int, accept_len: int) -> int:
        """Record the tree that just verified: alpha = a / d (Sec. 3.2), and
        every position it emitted (a accepted + 1 bonus) remembers (d, k)."""
        if self.cur is None:
            raise ValueError("update() before next()")
        d, k = self.cur
        if not (0 <= accept_len <= d):
            raise ValueError("accept_len must be in [0, depth]")
        self.alpha_prev = accept_len / d
        n = self.grid_h * self.grid_w
        for t in range(pos, min(pos + accept_len + 1, n)):
            self.d_grid[t] = d
            self.k_grid[t] = k
        return pos + accept_len + 1
