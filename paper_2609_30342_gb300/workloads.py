"""Synthetic workloads: parameter-shape lists and seeded input generators.

This module holds no optimiser arithmetic.  It is the one place both the
CUDA path (tests, benchmark) and the CPU oracle (tests) take their inputs
from, so the two always see identical values.

Shapes follow PyTorch's ``nn.Linear`` storage, ``[out_features,
in_features]`` = ``(rows, cols)``.  A shape ``(L, 0)`` is a parameter that is
not a matrix (bias, LayerNorm scale or shift) with ``L`` elements; the
optimiser applies the element-wise rule to it.

Query, key and value projections are separate matrices: the paper counts 74
two-dimensional layers in GPT2-S (Section 4.4), i.e. 12 blocks x {q, k, v,
o, fc, proj} plus the token and position embeddings.  The token embedding is
tied to the output head and appears once.
"""
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np

try:  # torch is only needed for the bf16 rounding of gradients
    import torch
except ImportError:  # pragma: no cover
    torch = None


def gpt2_shapes(n_layer, n_embd, vocab, ctx, mlp_mult=4, fused_qkv=False):
    """Parameter shapes of a nanoGPT-style GPT-2 with biases, tied head.

    Returns a list of ``(name, (rows, cols))`` in module order.
    """
    d, f = n_embd, mlp_mult * n_embd
    out = [("wte", (vocab, d)), ("wpe", (ctx, d))]
    for b in range(n_layer):
        p = "h%d." % b
        out += [(p + "ln_1.weight", (d, 0)), (p + "ln_1.bias", (d, 0))]
        if fused_qkv:
            out += [(p + "attn.c_attn.weight", (3 * d, d)), (p + "attn.c_attn.bias", (3 * d, 0))]
        else:
            for q in ("q", "k", "v"):
                out += [(p + "attn.%s.weight" % q, (d, d)), (p + "attn.%s.bias" % q, (d, 0))]
        out += [(p + "attn.c_proj.weight", (d, d)), (p + "attn.c_proj.bias", (d, 0))]
        out += [(p + "ln_2.weight", (d, 0)), (p + "ln_2.bias", (d, 0))]
        out += [(p + "mlp.c_fc.weight", (f, d)), (p + "mlp.c_fc.bias", (f, 0))]
        out += [(p + "mlp.c_proj.weight", (d, f)), (p + "mlp.c_proj.bias", (d, 0))]
    out += [("ln_f.weight", (d, 0)), ("ln_f.bias", (d, 0))]
    return out


def gpt2_small():
    """GPT2-S (124M): 12 layers, width 768, vocab 50257, context 1024."""
    return gpt2_shapes(12, 768, 50257, 1024)


def gpt2_nano():
    """GPT2-Nano-shaped list: 6 layers, width 384, vocab 50304, context 256."""
    return gpt2_shapes(6, 384, 50304, 256)


# Large single matrices of the aspect-ratio sweep (tall, wide, square).
SWEEP_SHAPES = [(4096, 4096), (4096, 14336), (14336, 4096), (50304, 4096)]


def numel(shape):
    rows, cols = shape
    return rows if cols == 0 else rows * cols


def array_shape(shape):
    rows, cols = shape
    return (rows,) if cols == 0 else (rows, cols)


def count(shapes):
    """(N, number of matrices, sum of m + n over matrices, 1-D elements)."""
    N = mats = mn = one_d = 0
    for m, n in shapes:
        if n == 0:
            one_d += m
            N += m
        else:
            mats += 1
            mn += m + n
            N += m * n
    return N, mats, mn, one_d


def bf16_round(a):
    """Round a float32 array to bf16 (nearest-even) and return the bf16 values as float32."""
    if torch is None:
        raise RuntimeError("torch is required for bf16 rounding")
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t.to(torch.bfloat16).to(torch.float32).numpy()


_BLOCK = 1 << 22          # elements drawn from one stream
_pool = None


def _block_pool():
    global _pool
    if _pool is None:
        _pool = ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 4))
    return _pool


def tensor_normal(shape, seed, std):
    """float32 array of ``shape`` (a (rows, cols) pair), i.i.d. N(0, std^2).
    Elements [b 2^22, (b + 1) 2^22) come from the stream [*seed, b], so the
    blocks of a large tensor are drawn in parallel threads."""
    n = numel(shape)
    out = np.empty(n, np.float32)
    base = [int(v) for v in np.atleast_1d(seed)]

    def fill(b):
        lo, hi = b * _BLOCK, min(n, (b + 1) * _BLOCK)
        np.random.default_rng(base + [b]).standard_normal(hi - lo, dtype=np.float32, out=out[lo:hi])
        out[lo:hi] *= np.float32(std)

    nb = -(-n // _BLOCK)
    if nb == 1:
        fill(0)
    elif nb > 1:
        list(_block_pool().map(fill, range(nb)))
    return out.reshape(array_shape(shape))


def normal_list(shapes, seed, std):
    """One float32 array per shape, i.i.d. N(0, std^2); tensor t draws from its
    own stream [*seed, t], so any tensor can be drawn without the others."""
    base = list(np.atleast_1d(seed))
    return [tensor_normal(s, base + [t], std) for t, s in enumerate(shapes)]


class ModelInputs:
    """Seeded synthetic state for a parameter list.

    ``X`` ~ N(0, x_std^2) float32, ``P`` = 0, and ``grads(step)`` yields
    float32 arrays ~ N(0, g_std^2), already rounded to bf16 when
    ``grad_bf16`` (the rounded values are what both sides consume).  Every
    tensor has its own streams ([seed, 0, t] for X, [seed, 1, step, t] for
    its gradients): ``x(t)`` and ``grad(step, t)`` draw one tensor alone.
    """

    def __init__(self, shapes, seed, x_std=0.02, g_std=1e-3, grad_bf16=True, draw_x=True):
        self.shapes = list(shapes)
        self.seed = int(seed)
        self.x_std = float(x_std)
        self.g_std = float(g_std)
        self.grad_bf16 = bool(grad_bf16)
        self.X = [self.x(t) for t in range(len(self.shapes))] if draw_x else None
        self.P = [np.zeros(array_shape(s), np.float32) for s in self.shapes] if draw_x else None

    def x(self, t):
        return tensor_normal(self.shapes[t], [self.seed, 0, t], self.x_std)

    def grad(self, step, t):
        g = tensor_normal(self.shapes[t], [self.seed, 1, int(step), t], self.g_std)
        return bf16_round(g) if self.grad_bf16 else g

    def grads(self, step):
        return [self.grad(step, t) for t in range(len(self.shapes))]


class QuadraticProblem:
    """f(X) = 1/2 sum A (.) (X - X*)^2 on an m x n matrix, gradient A (.) (X - X*).

    A ~ U[0.1, 10] and X* ~ N(0, 1), both float32, from ``seed``; X(0) = 0 and
    P(0) = 0.
    """

    def __init__(self, m, n, seed):
        rng = np.random.default_rng(seed)
        self.A = rng.uniform(0.1, 10.0, size=(m, n)).astype(np.float32)
        self.Xstar = rng.standard_normal((m, n), dtype=np.float32)
        self.X0 = np.zeros((m, n), np.float32)
        self.P0 = np.zeros((m, n), np.float32)


def single_matrix_inputs(m, n, seed, steps, x_std=0.02, g_std=0.01):
    """Single m x n fp32 matrix: X ~ N(0, x_std^2), P = 0, one fresh fp32
    gradient N(0, g_std^2) per step (all drawn from ``seed``)."""
    rng = np.random.default_rng(seed)
    X = (rng.standard_normal((m, n), dtype=np.float32) * np.float32(x_std))
    G = [(rng.standard_normal((m, n), dtype=np.float32) * np.float32(g_std)) for _ in range(steps)]
    return X, np.zeros((m, n), np.float32), G


def dense_quadratic_instance(m, n, seed):
    """Test problem of the gamma = 0 rate validation (Section 3.2, numerical
    set-up appendix): f(X) = 1/2 vec(X)^T A vec(X) with A = B B^T / d + 0.8 I,
    d = m n, B standard normal; X(0) ~ N(0, 0.4^2) and P(0) ~ N(0, 0.3^2)
    element-wise (R(0) = C(0) = 0 is the caller's).  float64, from ``seed``;
    A is made exactly symmetric."""
    rng = np.random.default_rng(seed)
    d = m * n
    B = rng.standard_normal((d, d))
    A = B @ B.T / d + 0.8 * np.eye(d)
    A = 0.5 * (A + A.T)
    X = 0.4 * rng.standard_normal((m, n))
    P = 0.3 * rng.standard_normal((m, n))
    return A, X, P


def dense_quadratic_batch(m, n, seeds):
    """float32 (A, X, P) of shapes (b, d, d), (b, m, n), (b, m, n) for the
    instances of ``seeds`` (see dense_quadratic_instance)."""
    inst = [dense_quadratic_instance(m, n, s) for s in seeds]
    A = np.stack([a for a, _, _ in inst]).astype(np.float32)
    X = np.stack([x for _, x, _ in inst]).astype(np.float32)
    P = np.stack([p for _, _, p in inst]).astype(np.float32)
    return A, X, P


def log_records(T, h, per_decade=60, t_min=10.0):
    """Ascending step indices k with t = k h spread evenly in log t over
    [t_min, T], plus k = 0 and the last step."""
    n = int(round(T / h))
    decades = max(np.log10(T / t_min), 0.0)
    pts = np.logspace(np.log10(t_min), np.log10(T), max(2, int(round(per_decade * decades)) + 1))
    k = np.unique(np.concatenate([[0], np.round(pts / h).astype(np.int64), [n]]))
    return k[(k >= 0) & (k <= n)]
