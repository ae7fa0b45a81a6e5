"""CPU oracle for the batch back-propagation training step (float64).

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
execute this module: it is used by ``tests/``, by ``__graft_entry__.smoke()``
and by the ``cpu_baseline`` / ``--impl reference`` legs of ``bench.py``.  It
shares no code with the CUDA path.

What it computes is the plain definition of back-propagation with pooled
(batch) weight changes and a learning-rate/momentum update, as the paper states
it (Witbrock & Zagha, "An Implementation of Back-Propagation Learning on GF11",
CMU-CS-89-208):

* forward pass: each unit takes the weighted sum of the activations feeding it
  and applies the logistic function 1/(1+e^-x) (Section 3, footnote 4); the
  bias is a weight from the always-on "true" unit (Section 6.3);
* error measure: summed squared difference (Section 3, footnote 5; the "total
  squared error" of Section 8);
* backward pass: partial derivatives of the error with respect to each weight,
  from the output layer back (Section 3); no error is propagated into the
  input units, whose connections only take the gradient step (Section 6.1,
  "Cycles backward/case");
* pooled update: weight changes are summed over all patterns of a group and
  applied once (Sections 3 and 4.1);
* the update routine applies the learning rate and momentum to the summed
  change and zeroes the accumulator (Section 6.2.1);
* optionally, the table-lookup logistic of Section 4.3 (256 points over
  [-15, 15], linear interpolation, clamped outside) in place of 1/(1+e^-x);
* optionally, the fault guard of Section 8: a total weight change outside a
  reasonable range is set to zero and counted before the update.

Readings taken where the paper is silent:

* the update is the classic momentum rule of the paper's back-propagation
  reference: V <- lr*grad_scale*G + momentum*V, W <- W + V, G <- 0, with V
  starting at zero; G is the sum over the group of delta * activation, which is
  minus the gradient of E/2, so the "+" moves downhill;
* grad_scale = 1 (a sum, as the paper pools) is the default; 1/B gives a mean;
* SSE is reported as the plain sum of (t - o)^2 over patterns and outputs;
* minibatches are taken in index order without shuffling, and V persists across
  minibatches and epochs.

Every array is float64.  Matrix products use numpy's matmul as a library step.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np


# ---------------------------------------------------------------- counting
def connections(sizes) -> int:
    """Connections W, bias ("true unit") connections included (Section 7.1)."""
    return int(sum((sizes[l - 1] + 1) * sizes[l] for l in range(1, len(sizes))))


def input_connections(sizes) -> int:
    """W_i: weights leaving the input layer, the true unit's into layer 1 included
    (Section 6.1, variable table)."""
    return int((sizes[0] + 1) * sizes[1])


def flops_per_connection(sizes) -> float:
    """MFLOPS / MCPS = 4 + 2 (W - W_i) / W (Section 7.2)."""
    W = connections(sizes)
    Wi = input_connections(sizes)
    return 4.0 + 2.0 * (W - Wi) / W


def flops_per_pattern(sizes) -> int:
    """2W forward + 2W_i + 4(W - W_i) backward (Section 6.1 cycle counts)."""
    W = connections(sizes)
    Wi = input_connections(sizes)
    return 2 * W + 2 * Wi + 4 * (W - Wi)


# ---------------------------------------------------------------- parameters
def unpack(sizes, theta):
    """Flat vector -> (list of W_l [n_l, n_{l-1}], list of b_l [n_l]).

    Layout: for l = 1..L, W_l row-major then b_l.
    """
    theta = np.asarray(theta, dtype=np.float64)
    Ws, bs = [], []
    pos = 0
    for l in range(1, len(sizes)):
        n_out, n_in = sizes[l], sizes[l - 1]
        Ws.append(theta[pos:pos + n_out * n_in].reshape(n_out, n_in).copy())
        pos += n_out * n_in
        bs.append(theta[pos:pos + n_out].copy())
        pos += n_out
    if pos != theta.size:
        raise ValueError("parameter vector length does not match the layer sizes")
    return Ws, bs


def pack(Ws, bs) -> np.ndarray:
    parts = []
    for W, b in zip(Ws, bs):
        parts.append(np.asarray(W, dtype=np.float64).ravel())
        parts.append(np.asarray(b, dtype=np.float64).ravel())
    return np.concatenate(parts)


# ---------------------------------------------------------------- the step
def sigmoid(x):
    """Logistic squashing function 1 / (1 + e^-x) (Section 3, footnote 4)."""
    return 1.0 / (1.0 + np.exp(-x))


# Table-lookup logistic (Section 4.3, Figure 3): 256 precomputed values of the
# logistic at equally spaced points over [-15, 15].
SIGMOID_TABLE_LO = -15.0
SIGMOID_TABLE_HI = 15.0
SIGMOID_TABLE_POINTS = 256


def sigmoid_table(x):
    """The second GF11 method of Section 4.3, step by step:

    1. net inputs outside [-15, 15] are mapped to the extreme values of the
       table (the logistic at -15 and at 15);
    2. inputs inside are remapped by an addition and a multiplication to x1 in
       [0, 255];
    3. the integer part of x1 indexes a table of 1/(1+e^-x) at 256 equally
       spaced points, and the fractional part interpolates linearly between
       that entry and the next (at x1 = 255 the last entry is returned).
    """
    x = np.asarray(x, dtype=np.float64)
    n = SIGMOID_TABLE_POINTS
    nodes = SIGMOID_TABLE_LO + (SIGMOID_TABLE_HI - SIGMOID_TABLE_LO) * np.arange(n) / (n - 1)
    table = sigmoid(nodes)
    xc = np.clip(x, SIGMOID_TABLE_LO, SIGMOID_TABLE_HI)
    x1 = (xc - SIGMOID_TABLE_LO) * ((n - 1) / (SIGMOID_TABLE_HI - SIGMOID_TABLE_LO))
    i = np.minimum(np.floor(x1), n - 2).astype(np.int64)
    f = x1 - i
    return table[i] + f * (table[i + 1] - table[i])


SQUASH = {"logistic": sigmoid, "table": sigmoid_table}


def forward(Ws, bs, X, squash="logistic"):
    """Activations [A_0 = X, A_1, ..., A_L]; A_l = sigma(A_{l-1} W_l^T + b_l).

    Section 3: a unit's activation is the logistic of the weighted sum of the
    activations connected to it; the bias is the true unit's weight.  With
    squash="table" sigma is the table-lookup logistic of Section 4.3; the
    deltas still use a (1 - a) of the activations it produced.
    """
    fn = SQUASH[squash]
    As = [np.asarray(X, dtype=np.float64)]
    for W, b in zip(Ws, bs):
        net = As[-1] @ W.T + b[None, :]
        As.append(fn(net))
    return As


def sse(O, T) -> float:
    """Summed squared difference over patterns and outputs (Section 3, fn. 5)."""
    d = np.asarray(T, dtype=np.float64) - O
    return float(np.sum(d * d))


def output_delta(O, T):
    """delta_L = (t - o) o (1 - o): minus dE/dnet for E = sum (t - o)^2 / 2."""
    return (np.asarray(T, dtype=np.float64) - O) * O * (1.0 - O)


def hidden_delta(W_next, D_next, A):
    """delta_l = (delta_{l+1} W_{l+1}) * a (1 - a), for a hidden layer l.

    Section 3 works backwards from the output weights; Section 6.1 states that
    input units receive no back-propagated error, so callers never ask for l = 0.
    """
    return (D_next @ W_next) * A * (1.0 - A)


def deltas(Ws, As, T):
    """[delta_1, ..., delta_L] for one group of patterns."""
    L = len(Ws)
    Ds = [None] * L
    Ds[L - 1] = output_delta(As[L], T)
    for l in range(L - 1, 0, -1):
        Ds[l - 1] = hidden_delta(Ws[l], Ds[l], As[l])
    return Ds


def gradients(As, Ds):
    """Pooled weight changes summed over the group (Sections 3 and 4.1):
    G_l = delta_l^T A_{l-1},  g_l = sum over patterns of delta_l."""
    Gs = [D.T @ A for D, A in zip(Ds, As[:-1])]
    gs = [D.sum(axis=0) for D in Ds]
    return Gs, gs


def guard_changes(g, guard):
    """The fault guard of Section 8: every total weight change of the group is
    tested for a reasonable range; one outside it (|g| > guard, or not a
    number) is set to zero and counted.  guard <= 0 turns the test off.
    Returns (guarded changes, number zeroed)."""
    g = np.asarray(g, dtype=np.float64)
    if guard <= 0:
        return g, 0
    bad = ~(np.abs(g) <= guard)
    return np.where(bad, 0.0, g), int(np.count_nonzero(bad))


def momentum_update(w, v, g, lr, momentum, grad_scale=1.0):
    """Update routine of Section 6.2.1 (read as the classic momentum rule):
    v <- lr * grad_scale * g + momentum * v;  w <- w + v.  Returns (w, v)."""
    v_new = lr * grad_scale * g + momentum * v
    return w + v_new, v_new


# ---------------------------------------------------------------- training state
@dataclass
class State:
    sizes: tuple
    theta: np.ndarray            # flat weights + biases
    lr: float
    momentum: float
    grad_scale: float = 1.0
    V: np.ndarray = field(default=None)   # previous weight change
    G: np.ndarray = field(default=None)   # pooled change not yet applied
    squash: str = "logistic"              # or "table" (Section 4.3)
    guard: float = 0.0                    # weight-change range of the fault guard (0: off)
    faults: int = 0                       # changes the guard has zeroed

    def __post_init__(self):
        self.sizes = tuple(int(s) for s in self.sizes)
        self.theta = np.array(self.theta, dtype=np.float64)
        if self.V is None:
            self.V = np.zeros_like(self.theta)
        if self.G is None:
            self.G = np.zeros_like(self.theta)


def step_quantities(state: State, X, T):
    """Everything one group of patterns yields: activations, deltas, the pooled
    change (flat, same layout as theta) and the SSE.  Does not modify state."""
    Ws, bs = unpack(state.sizes, state.theta)
    As = forward(Ws, bs, X, state.squash)
    Ds = deltas(Ws, As, T)
    Gs, gs = gradients(As, Ds)
    return As, Ds, pack(Gs, gs), sse(As[-1], T)


def backward_accumulate(state: State, X, T) -> float:
    """Add one group's pooled change into state.G; return its SSE."""
    _, _, G, e = step_quantities(state, X, T)
    state.G = state.G + G
    return e


def apply_update(state: State) -> None:
    """Apply and zero the pooled change (Section 6.2.1), after the fault guard
    of Section 8 when one is set."""
    G, n_bad = guard_changes(state.G, state.guard)
    state.faults += n_bad
    state.theta, state.V = momentum_update(state.theta, state.V, G,
                                           state.lr, state.momentum, state.grad_scale)
    state.G = np.zeros_like(state.G)


def train_batch(state: State, X, T) -> float:
    """Forward, backward, pooled accumulation and one update over one group."""
    e = backward_accumulate(state, X, T)
    apply_update(state)
    return e


def train_epoch(state: State, X, T, minibatch: int):
    """One pass over the patterns in index order, one update per minibatch;
    a ragged last minibatch is a group of its own.  Returns the SSE per update."""
    n = len(X)
    out = []
    for p0 in range(0, n, minibatch):
        out.append(train_batch(state, X[p0:p0 + minibatch], T[p0:p0 + minibatch]))
    return out


def predict(state: State, X):
    Ws, bs = unpack(state.sizes, state.theta)
    return forward(Ws, bs, X, state.squash)[-1]
