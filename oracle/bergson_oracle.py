"""Plain fp64 CPU oracle for Bergson's projected-gradient attribution path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports this module:
only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline /
reference legs may call it.  It shares no code with the CUDA library.

What it computes (Bergson, Sec. 3.1 and Fig. 1; App. B, "Gradients"):
  1. the per-example gradient of an ``nn.Linear`` weight,
     W_b = sum_t m_{b,t} g_{b,t} a_{b,t}^T   (d_out x d_in), explicitly;
  2. optional Adafactor-style factored second-moment normalisation,
     W~_b[i, j] = W_b[i, j] / sqrt(r_i c_j)   (r over d_out, c over d_in);
  3. the double-sided per-module random projection
     G^_b = P_out^T W~_b P_in                (k_out x k_in, row-major, k_out major);
  4. concatenation over modules in call order and unit normalisation of the
     whole per-example row (grad-cosine), or, as an option, of each module's
     block on its own (the store is indexed by module, Sec. 3.1);
  5. an fp16 gradient store, cosine scores against unit-normalised queries and
     exact top-k, ordered by (score descending, index ascending), and the k
     least influential items (Sec. 3.1), ordered by (score ascending, index
     ascending);
  6. on-the-fly scores (Sec. 3.1, "bergson score"): training rows scored
     directly against query rows without a store, as cosines (grad-cosine) or
     plain inner products (grad-dot) -- Table 3's two identity-Hessian methods;
  7. per-token scores (Fig. 1: attribution scores per token or per sequence):
     the inner product of each token's own projected gradient with a query;
  8. query aggregation (Sec. 3.2): a query row formed as the mean or sum of
     several items' (optionally unit-normalised) projected gradients;
  9. TrackStar's empirical-Fisher preconditioner (Sec. 3.1; Fig. 2 "empirical
     Fisher information matrix fitting and mixing"): R = (1/n) sum_i x_i x_i^T
     over projected gradients, a mix of two such matrices plus damping, and
     its inverse square root (or inverse) applied to rows before unit norm;
 10. bias gradients (App. B, "linear (weight and bias) parameters"):
     sum_t m_t g_t, scaled by r^-1/2 and projected with P_out (k_out values).

Readings taken where the paper is silent:
  * the projection is Gaussian with entries N(0, 1/k) per side, drawn from a
    stateless counter-based generator (SplitMix64 finaliser of Steele, Lea and
    Flood 2014, then the Box-Muller transform of Box and Muller 1958), entry
    e = i*k + j of the row-major [d, k] matrix, rounded once to fp32; the
    Rademacher and uniform projections App. B names take one hash of the same
    counter per entry and are scaled to the same variance 1/k;
  * second moments divide by sqrt(r c^T) with no 1/sum(r) and no epsilon;
  * a masked token contributes nothing, whatever A and G hold there;
  * a row whose norm is zero stays zero.

Every function here is pinned by ``tests/test_oracle_pins.py`` against closed
forms, finite differences, published generator outputs and brute force.
"""
from __future__ import annotations

import numpy as np

# SplitMix64 constants (Steele, Lea, Flood: "Fast splittable pseudorandom
# number generators", OOPSLA 2014; finaliser variant "Mix13" by D. Stafford).
_GOLDEN_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_TWO_M53 = 2.0 ** -53

PROJ_GAUSSIAN = 0
PROJ_IDENTITY = 1
PROJ_RADEMACHER = 2
PROJ_UNIFORM = 3


def mix64(x):
    """SplitMix64 finaliser on a uint64 array (wrapping arithmetic)."""
    x = np.asarray(x, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (x ^ (x >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def splitmix64_sequence(seed: int, n: int) -> np.ndarray:
    """The first ``n`` outputs of the SplitMix64 generator started at ``seed``."""
    with np.errstate(over="ignore"):
        states = np.uint64(seed) + _GOLDEN_GAMMA * np.arange(1, n + 1, dtype=np.uint64)
    return mix64(states)


def gaussian_counter(seed: int, n: int) -> np.ndarray:
    """Standard normal draws z_0 .. z_{n-1} for counter e = 0 .. n-1 (fp64).

    Pair p = e >> 1 takes two 64-bit hashes h1 = mix(seed ^ mix(2p)) and
    h2 = mix(seed ^ mix(2p + 1)), turns them into u1 in (0, 1] and u2 in [0, 1)
    with 53-bit resolution, and applies Box-Muller: even e takes the cosine
    branch, odd e the sine branch.
    """
    e = np.arange(n, dtype=np.uint64)
    p = e >> np.uint64(1)
    s = np.uint64(seed)
    h1 = mix64(s ^ mix64(np.uint64(2) * p))
    h2 = mix64(s ^ mix64(np.uint64(2) * p + np.uint64(1)))
    u1 = ((h1 >> np.uint64(11)) + np.uint64(1)).astype(np.float64) * _TWO_M53
    u2 = (h2 >> np.uint64(11)).astype(np.float64) * _TWO_M53
    rho = np.sqrt(-2.0 * np.log(u1))
    theta = 2.0 * np.pi * u2
    return np.where((e & np.uint64(1)) == 0, rho * np.cos(theta), rho * np.sin(theta))


def counter_hash(seed: int, n: int) -> np.ndarray:
    """One 64-bit hash per counter: h_e = mix(seed ^ mix(e)), e = 0 .. n-1."""
    e = np.arange(n, dtype=np.uint64)
    return mix64(np.uint64(seed) ^ mix64(e))


def rademacher_counter(seed: int, n: int) -> np.ndarray:
    """Rademacher draws (App. B, "Gradients"): +1 where the top bit of h_e is
    set, -1 where it is clear (fp64)."""
    top = counter_hash(seed, n) >> np.uint64(63)
    return np.where(top == np.uint64(1), 1.0, -1.0)


def uniform_counter(seed: int, n: int) -> np.ndarray:
    """Uniform draws on (-1, 1) (App. B, "Gradients"): the top 24 bits v of h_e
    give x = (2v + 1 - 2^24) / 2^24, the midpoints of 2^24 equal cells, so the
    draws are symmetric about 0 and exactly representable in fp32."""
    v = (counter_hash(seed, n) >> np.uint64(40)).astype(np.float64)
    return (2.0 * v + 1.0 - 2.0 ** 24) / 2.0 ** 24


def projection_matrix(seed: int, d: int, k: int, kind: int = PROJ_GAUSSIAN) -> np.ndarray:
    """Dense projection P in R^{d x k}, stored as fp32 values held in fp64.

    Entry (i, j) takes counter e = i*k + j and has mean 0 and variance 1/k, so
    E||P^T x||^2 = ||x||^2 (Johnson-Lindenstrauss scaling):
      Gaussian:   P[i, j] = fl32(z_e / sqrt(k));
      Rademacher: P[i, j] = fl32(s_e / sqrt(k)), s_e = +-1;
      uniform:    P[i, j] = fl32(sqrt(3) x_e / sqrt(k)), x_e uniform on (-1, 1)
                  (variance 1/3, hence the sqrt(3));
      identity (tests only): k == d and P = I.
    """
    if kind == PROJ_IDENTITY:
        if k != d:
            raise ValueError("identity projection needs k == d")
        return np.eye(d, dtype=np.float64)
    if kind == PROJ_GAUSSIAN:
        z = gaussian_counter(seed, d * k)
    elif kind == PROJ_RADEMACHER:
        z = rademacher_counter(seed, d * k)
    elif kind == PROJ_UNIFORM:
        z = np.sqrt(3.0) * uniform_counter(seed, d * k)
    else:
        raise ValueError(f"unknown projection kind {kind}")
    return (z.reshape(d, k) / np.sqrt(k)).astype(np.float32).astype(np.float64)


def module_seeds(base_seed: int, module_index: int) -> tuple[int, int]:
    """Per-module seeds (s_in, s_out) derived from one base seed."""
    b = np.uint64(base_seed)
    m = np.uint64(module_index)
    s_in = int(mix64(b ^ (np.uint64(2) * m)))
    s_out = int(mix64(b ^ (np.uint64(2) * m + np.uint64(1))))
    return s_in, s_out


def per_example_gradient(a: np.ndarray, g: np.ndarray, m: np.ndarray | None) -> np.ndarray:
    """W = sum over valid tokens t of g_t a_t^T, shape [d_out, d_in], fp64.

    a: [T, d_in] layer inputs, g: [T, d_out] output gradients, m: [T] 0/1 mask
    (None = every token valid).  Only valid tokens enter the sum.
    """
    a = np.asarray(a, dtype=np.float64)
    g = np.asarray(g, dtype=np.float64)
    if m is not None:
        keep = np.asarray(m) != 0
        a = a[keep]
        g = g[keep]
    return g.T @ a


def adafactor_normalize(w: np.ndarray, r: np.ndarray | None, c: np.ndarray | None) -> np.ndarray:
    """W~[i, j] = W[i, j] / sqrt(r_i c_j); identity when r and c are absent."""
    if r is None and c is None:
        return w
    if r is None or c is None:
        raise ValueError("r and c come together")
    r = np.asarray(r, dtype=np.float64)
    c = np.asarray(c, dtype=np.float64)
    return w / np.sqrt(np.outer(r, c))


def double_sided_projection(w: np.ndarray, p_out: np.ndarray, p_in: np.ndarray) -> np.ndarray:
    """G^ = P_out^T W P_in, shape [k_out, k_in]."""
    return p_out.T @ w @ p_in


def bias_gradient(g: np.ndarray, m: np.ndarray | None) -> np.ndarray:
    """Per-example bias gradient sum over valid tokens t of g_t, shape [d_out], fp64."""
    g = np.asarray(g, dtype=np.float64)
    if m is not None:
        g = g[np.asarray(m) != 0]
    return g.sum(axis=0)


class Layer:
    """One nn.Linear's captured tensors and projection settings (host arrays).

    A: [B, T, d_in], G: [B, T, d_out] (any float dtype; bf16 values arrive as
    exact fp32), r: [d_out] or None, c: [d_in] or None.  bias_col_offset >= 0
    also places the projected bias gradient (k_out values) at that column.
    """

    def __init__(self, A, G, k_in, k_out, seed_in, seed_out, r=None, c=None,
                 col_offset=0, proj_kind=PROJ_GAUSSIAN, bias_col_offset=-1):
        self.A = np.asarray(A)
        self.G = np.asarray(G)
        self.k_in = int(k_in)
        self.k_out = int(k_out)
        self.seed_in = int(seed_in)
        self.seed_out = int(seed_out)
        self.r = None if r is None else np.asarray(r, dtype=np.float64)
        self.c = None if c is None else np.asarray(c, dtype=np.float64)
        self.col_offset = int(col_offset)
        self.proj_kind = int(proj_kind)
        self.bias_col_offset = int(bias_col_offset)

    @property
    def d_in(self):
        return self.A.shape[-1]

    @property
    def d_out(self):
        return self.G.shape[-1]


def project_module(layer: Layer, mask: np.ndarray | None, examples=None) -> np.ndarray:
    """Projected per-example gradients of one module, [len(examples), k_out*k_in].

    Steps 1-3 above for each example, flattened row-major (k_out major).
    """
    B = layer.A.shape[0]
    examples = range(B) if examples is None else examples
    p_in = projection_matrix(layer.seed_in, layer.d_in, layer.k_in, layer.proj_kind)
    p_out = projection_matrix(layer.seed_out, layer.d_out, layer.k_out, layer.proj_kind)
    rows = []
    for b in examples:
        m = None if mask is None else mask[b]
        w = per_example_gradient(layer.A[b], layer.G[b], m)
        w = adafactor_normalize(w, layer.r, layer.c)
        rows.append(double_sided_projection(w, p_out, p_in).reshape(-1))
    return np.stack(rows) if rows else np.zeros((0, layer.k_out * layer.k_in))


def project_grads(layers, mask, ld_out: int | None = None, examples=None) -> np.ndarray:
    """Unnormalised projected gradients of every module placed at its column offset.

    Returns [len(examples), ld_out] fp64; columns no module covers are zero.
    """
    B = layers[0].A.shape[0]
    examples = list(range(B)) if examples is None else list(examples)
    if ld_out is None:
        ld_out = max(max(l.col_offset + l.k_out * l.k_in, l.bias_col_offset + l.k_out)
                     for l in layers)
    out = np.zeros((len(examples), ld_out), dtype=np.float64)
    for layer in layers:
        blk = layer.k_out * layer.k_in
        out[:, layer.col_offset:layer.col_offset + blk] = project_module(layer, mask, examples)
        if layer.bias_col_offset >= 0:
            out[:, layer.bias_col_offset:layer.bias_col_offset + layer.k_out] = \
                project_bias(layer, mask, examples)
    return out


def project_bias(layer: Layer, mask: np.ndarray | None, examples=None) -> np.ndarray:
    """P_out^T (bias gradient / sqrt(r)) per example, [len(examples), k_out]."""
    B = layer.A.shape[0]
    examples = range(B) if examples is None else examples
    p_out = projection_matrix(layer.seed_out, layer.d_out, layer.k_out, layer.proj_kind)
    rows = []
    for b in examples:
        gb = bias_gradient(layer.G[b], None if mask is None else mask[b])
        if layer.r is not None:
            gb = gb / np.sqrt(layer.r)
        rows.append(p_out.T @ gb)
    return np.stack(rows) if rows else np.zeros((0, layer.k_out))


def unit_normalize(x: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """Rows divided by their l2 norm; zero rows stay zero.  Returns (rows, norms)."""
    x = np.asarray(x, dtype=np.float64)
    norms = np.sqrt(np.sum(x * x, axis=1))
    safe = np.where(norms > 0, norms, 1.0)
    return x / safe[:, None], norms


def build_store(proj: np.ndarray, unit: bool = True) -> tuple[np.ndarray, np.ndarray]:
    """fp16 store rows (round to nearest even from fp64) and the row norms."""
    rows, norms = unit_normalize(proj) if unit else (np.asarray(proj, np.float64), None)
    if norms is None:
        norms = np.sqrt(np.sum(rows * rows, axis=1))
    return rows.astype(np.float16), norms


def build_store_blocks(proj: np.ndarray, offsets) -> tuple[np.ndarray, np.ndarray]:
    """Per-module unit normalisation: each column block [o_j, o_{j+1}) of a row
    (one module's k_out x k_in block, the store being indexed by module,
    Sec. 3.1) divided by its own l2 norm, a zero block staying zero, then fp16
    (round to nearest even from fp64).  Returns (rows, norms [B, n_blocks])."""
    x = np.asarray(proj, dtype=np.float64)
    o = [int(v) for v in offsets]
    rows = np.zeros_like(x)
    norms = np.zeros((x.shape[0], len(o) - 1))
    for j in range(len(o) - 1):
        rows[:, o[j]:o[j + 1]], norms[:, j] = unit_normalize(x[:, o[j]:o[j + 1]])
    return rows.astype(np.float16), norms


def cosine_scores(store: np.ndarray, queries: np.ndarray, row_chunk: int = 1 << 18) -> np.ndarray:
    """S[q, n] = (q / ||q||) . s_n in fp64 for every query and store row.

    The store rows are used as stored (unit-norm up to fp16 rounding).  The
    product is formed in slices of ``row_chunk`` rows only to bound host memory.
    """
    q, _ = unit_normalize(queries)
    N = store.shape[0]
    S = np.empty((q.shape[0], N), dtype=np.float64)
    for n0 in range(0, N, row_chunk):
        n1 = min(N, n0 + row_chunk)
        S[:, n0:n1] = q @ np.asarray(store[n0:n1], dtype=np.float64).T
    return S


def topk_rows(S: np.ndarray, k: int) -> tuple[np.ndarray, np.ndarray]:
    """Exact top-k of each row of S by full sort on key (-score, index)."""
    Q, N = S.shape
    if k > N:
        raise ValueError("k > N")
    idx = np.empty((Q, k), dtype=np.int64)
    val = np.empty((Q, k), dtype=np.float64)
    cols = np.arange(N)
    for qi in range(Q):
        order = np.lexsort((cols, -S[qi]))[:k]
        idx[qi] = order
        val[qi] = S[qi, order]
    return val, idx


def bottomk_rows(S: np.ndarray, k: int) -> tuple[np.ndarray, np.ndarray]:
    """Exact bottom-k of each row of S (the k least influential items, Sec. 3.1)
    by full sort on key (score, index): lowest score first, ties by index."""
    Q, N = S.shape
    if k > N:
        raise ValueError("k > N")
    idx = np.empty((Q, k), dtype=np.int64)
    val = np.empty((Q, k), dtype=np.float64)
    cols = np.arange(N)
    for qi in range(Q):
        order = np.lexsort((cols, S[qi]))[:k]
        idx[qi] = order
        val[qi] = S[qi, order]
    return val, idx


def score_topk(store: np.ndarray, queries: np.ndarray, k: int):
    """Cosine scores of queries against the store and their exact top-k."""
    return topk_rows(cosine_scores(store, queries), k)


def score_bottomk(store: np.ndarray, queries: np.ndarray, k: int):
    """Cosine scores of queries against the store and their exact bottom-k."""
    return bottomk_rows(cosine_scores(store, queries), k)


def onthefly_scores(rows: np.ndarray, queries: np.ndarray, unit: bool = True) -> np.ndarray:
    """S[b, q] = <x_b, y_q>, with both sides unit-normalised when `unit` (fp64).

    Rows and queries are projected gradients straight from the projection
    step (no fp16 store in between); zero rows score 0 under normalisation.
    """
    x = np.asarray(rows, dtype=np.float64)
    y = np.asarray(queries, dtype=np.float64)
    if unit:
        x, _ = unit_normalize(x)
        y, _ = unit_normalize(y)
    return x @ y.T


def token_scores(layers, mask, queries: np.ndarray, examples=None) -> np.ndarray:
    """Per-token scores s[q, b, t] = sum over modules of <G^_{b,t}, Q~_q,m>_F (fp64).

    G^_{b,t} is the projected, normalised gradient of token t alone
    (P_out^T (g_t a_t^T / sqrt(r c^T)) P_in) and Q~_q,m is module m's
    k_out x k_in block of query row q (same column layout as project_grads).
    Masked tokens score 0.  Returns [Q, len(examples), T].
    """
    queries = np.asarray(queries, dtype=np.float64)
    B, T = layers[0].A.shape[0], layers[0].A.shape[1]
    examples = list(range(B)) if examples is None else list(examples)
    out = np.zeros((queries.shape[0], len(examples), T), dtype=np.float64)
    for layer in layers:
        p_in = projection_matrix(layer.seed_in, layer.d_in, layer.k_in, layer.proj_kind)
        p_out = projection_matrix(layer.seed_out, layer.d_out, layer.k_out, layer.proj_kind)
        blk = queries[:, layer.col_offset:layer.col_offset + layer.k_out * layer.k_in]
        qm = blk.reshape(-1, layer.k_out, layer.k_in)
        for bi, b in enumerate(examples):
            for t in range(T):
                if mask is not None and mask[b, t] == 0:
                    continue
                w = np.outer(np.asarray(layer.G[b, t], np.float64), np.asarray(layer.A[b, t], np.float64))
                w = adafactor_normalize(w, layer.r, layer.c)
                g_hat = double_sided_projection(w, p_out, p_in)
                out[:, bi, t] += np.einsum("qij,ij->q", qm, g_hat)
    return out


AGG_SUM = 0
AGG_MEAN = 1


def aggregate_rows(rows: np.ndarray, offsets, mode: int = AGG_MEAN,
                   normalize_each: bool = True) -> np.ndarray:
    """out[g] = sum or mean of rows[offsets[g]:offsets[g+1]] (each unit-normalised first
    when normalize_each).  An empty group gives a zero row.  fp64."""
    x = np.asarray(rows, dtype=np.float64)
    if normalize_each:
        x, _ = unit_normalize(x)
    G = len(offsets) - 1
    out = np.zeros((G, x.shape[1]), dtype=np.float64)
    for g in range(G):
        a, b = int(offsets[g]), int(offsets[g + 1])
        if b > a:
            acc = x[a:b].sum(axis=0)
            out[g] = acc / (b - a) if mode == AGG_MEAN else acc
    return out


def fisher_fit(rows: np.ndarray) -> np.ndarray:
    """Empirical Fisher (autocorrelation) R = (1/n) sum_i x_i x_i^T of n rows, fp64 [K, K]."""
    x = np.asarray(rows, dtype=np.float64)
    return x.T @ x / x.shape[0]


def fisher_mix(r1: np.ndarray, r2: np.ndarray | None, lam: float, damping: float) -> np.ndarray:
    """R = lam * R1 + (1 - lam) * R2 (R2 absent: R = R1), plus damping * (tr(R)/K) * I."""
    r = np.asarray(r1, dtype=np.float64)
    if r2 is not None:
        r = lam * r + (1.0 - lam) * np.asarray(r2, dtype=np.float64)
    K = r.shape[0]
    return r + damping * (np.trace(r) / K) * np.eye(K)


def fisher_power(r: np.ndarray, power: float) -> np.ndarray:
    """R^power for symmetric positive definite R (power -1/2 or -1) by eigendecomposition."""
    w, u = np.linalg.eigh(np.asarray(r, dtype=np.float64))
    return (u * w ** power) @ u.T


def precondition_rows(rows: np.ndarray, m: np.ndarray) -> np.ndarray:
    """x' = M x for every row x (M symmetric): rows @ M."""
    return np.asarray(rows, dtype=np.float64) @ np.asarray(m, dtype=np.float64)
