"""CPU oracle for the EOGP hot path (arxiv 2609.37842) -- TEST INFRASTRUCTURE.

This module is the slow, plain, float64 restatement of what the hot path
computes. It exists to check the CUDA library and is not part of the product:
only the tests, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline /
reference arm may import it. It shares no code with the CUDA path and imports
nothing from the package.

Conventions (the paper's notation):
  * a module with input activations a_t in R^{d_in} and output gradients
    s_t (delta in Sec. 2.2) in R^{d_out}, t = 1..T, has per-example gradient
    G = sum_t s_t a_t^T  (d_out x d_in); g = vec(G) in column-major order, so
    g = sum_t a_t (x) s_t, matching E[(a a^T) (x) (delta delta^T)] in
    Eq. kfac_factorization.
  * Q_A (d_in x d_in), Q_S (d_out x d_out): orthonormal eigenbases with
    eigenvectors as COLUMNS sorted by eigenvalue descending. The Kronecker
    eigenbasis Q_A (x) Q_S has its column i*d_out + j equal to
    Q_A[:, i] (x) Q_S[:, j], with eigenvalue Lam[j, i].
  * Lam is stored as a d_out x d_in array: Lam[j, i] is the (corrected)
    eigenvalue of Kronecker coordinate (j, i).

Function map:
  kfac_eigenvalues      Sec. 2.2 (eigenvalues of A (x) S)
  damping               App. C.2, Eq. app_module_damping
  select_retained       Sec. 3.2 (Eq. sigma_ekfac and the text after it), Alg. 1
  with_bias_channel     App. C.1 (biases as a constant-1 input channel)
  mask_tokens           App. C.1 (variable-length examples padded to T)
  per_example_gradient  Sec. 2.2 (K-FAC factors from a and delta)
  rotate                Sec. 2.2 (apply Q_A (x) Q_S through its two factors)
  ekfac_sumsq           Sec. 2.2 "EK-FAC approximation"; App. C.2 (corrected eigenvalues)
  first_stage           Sec. 3.2, Eq. first_stage
  fit_pca               App. B.2 "PCA fitting", Alg. 1
  fit_pca_from_moment   App. B.2 (covariance route from a summed second moment)
  project               Sec. 3.2, Eq. second_stage
  onebit                Sec. 3.3, Eq. onebit; App. A.3 Eq. app_onebit_scale
  pack_bits/unpack_bits App. E.1 (per-module byte packing, Eq. app_payload)
  score_codes           Sec. 3.3 Eq. onebit_influence with both sides one-bit
  onebit_dot_xor        the same +-1 inner product counted as k - 2 * (differing signs)
  score_paper           Sec. 3.3 Eq. onebit_influence; App. B.3 Eq. app_stored_influence
  score_fp              Sec. 3.1 (influence as an inner product of coordinates)
  srht                  Sec. 3.2 "A scalable alternative to PCA"; App. B.2 Eq. app_srht_definition
  top_k                 App. C (per-query ranking of stored examples, NDCG@20)
  payload_bytes         App. E.1, Eq. app_payload
  to_payload/from_payload  App. E.1 (per-module sign bytes + FP16 scale records)

Where the paper is silent, the function that needs a reading states it (ties
in the top-m selection, bit order, sign of zero, PCA sign convention, ranking
order, Hadamard ordering).
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

import numpy as np


# --------------------------------------------------------------------------
# Curvature, damping and the retained set
# --------------------------------------------------------------------------

def kfac_eigenvalues(lam_S: np.ndarray, lam_A: np.ndarray) -> np.ndarray:
    """Lam[j, i] = lam_S[j] * lam_A[i] in float64: the eigenvalue of A (x) S on the
    Kronecker eigenvector Q_A[:, i] (x) Q_S[:, j] (Sec. 2.2, Eq. kfac_factorization)."""
    return np.outer(np.asarray(lam_S, np.float64), np.asarray(lam_A, np.float64))


def damping(Lam: np.ndarray, rel: float) -> float:
    """lambda = rel * tr(Lam) / d over the module's full set of eigenvalues
    (App. C.2, Eq. app_module_damping; the paper uses rel = 0.1)."""
    Lam = np.asarray(Lam, np.float64)
    return float(rel * Lam.sum() / Lam.size)


def select_retained(Lam: np.ndarray, m: int) -> Tuple[np.ndarray, np.ndarray]:
    """The m eigen-coordinates with the largest eigenvalues (Sec. 3.2: the top-m
    eigenvectors of Sigma_proxy in Eq. sigma_ekfac are those with the largest
    corrected eigenvalues; Alg. 1 "Select Q_{u,m}, Lam_{u,m}").

    Returns (j, i) index arrays in canonical order: eigenvalue descending, ties
    broken by the Kronecker column position i*d_out + j ascending.
    """
    Lam = np.asarray(Lam, np.float64)
    d_out, d_in = Lam.shape
    if not (1 <= m <= d_out * d_in):
        raise ValueError("m out of range")
    vals = Lam.T.reshape(-1)              # position p = i*d_out + j
    pos = np.arange(vals.size)
    order = np.lexsort((pos, -vals))[:m]  # primary: -value, secondary: position
    j = order % d_out
    i = order // d_out
    return j.astype(np.int64), i.astype(np.int64)


# --------------------------------------------------------------------------
# First stage
# --------------------------------------------------------------------------

def with_bias_channel(a: np.ndarray) -> np.ndarray:
    """Activations with a constant-1 channel appended (App. C.1: GPT-2's biases
    are attributed; a bias is the weight of an input that is always 1, so the
    bias gradient sum_t s_t is the last column of G)."""
    a = np.asarray(a, np.float64)
    return np.concatenate([a, np.ones(a.shape[:-1] + (1,))], axis=-1)


def mask_tokens(s: np.ndarray, lengths) -> np.ndarray:
    """Output gradients with the padding positions t >= lengths[b] of each
    example zeroed, so only the example's own tokens enter G_b (App. C.1:
    examples are conversations of at most 2048 tokens)."""
    s = np.array(s, np.float64)
    for b, n in enumerate(lengths):
        s[b, int(n):] = 0.0
    return s


def per_example_gradient(a_b: np.ndarray, s_b: np.ndarray) -> np.ndarray:
    """G = sum_t s_t a_t^T, a d_out x d_in matrix, from one example's activations
    a_b [T, d_in] and output gradients s_b [T, d_out] (Sec. 2.2)."""
    a_b = np.asarray(a_b, np.float64)
    s_b = np.asarray(s_b, np.float64)
    return s_b.T @ a_b


def rotate(G: np.ndarray, Q_A: np.ndarray, Q_S: np.ndarray) -> np.ndarray:
    """Coordinates of vec(G) in the Kronecker eigenbasis Q_A (x) Q_S, applied through
    its two factors: Gt = Q_S^T G Q_A, so that Gt[j, i] is the coordinate on
    Q_A[:, i] (x) Q_S[:, j] (Sec. 2.2, last sentence of the K-FAC paragraph)."""
    Q_A = np.asarray(Q_A, np.float64)
    Q_S = np.asarray(Q_S, np.float64)
    return Q_S.T @ np.asarray(G, np.float64) @ Q_A


def ekfac_sumsq(a: np.ndarray, s: np.ndarray, Q_A: np.ndarray, Q_S: np.ndarray) -> np.ndarray:
    """Sum over examples of the squared eigenbasis coordinates,
    sum_b (Q_S^T G_b Q_A)[j, i]^2 with G_b = sum_t s_t a_t^T (d_out x d_in).
    Divided by the number of examples this is the EK-FAC corrected eigenvalue
    table (Sec. 2.2 "EK-FAC approximation": mean square of each coordinate of
    the gradients in the K-FAC eigenbasis; App. C.2: over examples, with
    sequence-level gradients)."""
    out = np.zeros((np.asarray(Q_S).shape[1], np.asarray(Q_A).shape[1]))
    for b in range(np.asarray(a).shape[0]):
        out += rotate(per_example_gradient(a[b], s[b]), Q_A, Q_S) ** 2
    return out


def first_stage(a: np.ndarray, s: np.ndarray, Q_A: np.ndarray, Q_S: np.ndarray,
                Lam: np.ndarray, lam: float, m: int) -> np.ndarray:
    """z_b = (Lam_m + lam I)^{-1/2} Q_m^T g_b for each example b (Sec. 3.2,
    Eq. first_stage), with a [B, T, d_in], s [B, T, d_out]. Returns z [B, m] in
    the canonical retained order of select_retained."""
    j, i = select_retained(Lam, m)
    c = 1.0 / np.sqrt(np.asarray(Lam, np.float64)[j, i] + lam)
    B = a.shape[0]
    z = np.empty((B, m), np.float64)
    for b in range(B):
        Gt = rotate(per_example_gradient(a[b], s[b]), Q_A, Q_S)
        z[b] = c * Gt[j, i]
    return z


# --------------------------------------------------------------------------
# Second stage: PCA directions and projection
# --------------------------------------------------------------------------

def canonical_signs(V: np.ndarray) -> np.ndarray:
    """Fix each column's sign so that its largest-magnitude entry is positive
    (ties: lowest row index). Eigenvectors are defined only up to sign."""
    V = np.array(V, np.float64, copy=True)
    for c in range(V.shape[1]):
        r = int(np.argmax(np.abs(V[:, c])))  # argmax returns the first maximum
        if V[r, c] < 0:
            V[:, c] = -V[:, c]
    return V


def fit_pca(Z: np.ndarray, k: int, route: str = "auto") -> Tuple[np.ndarray, np.ndarray]:
    """Uncentered PCA of the rows of Z [n, m] (App. B.2 "PCA fitting").

    P [m, k] holds the top-k eigenvectors of Z^T Z / n (columns, eigenvalue
    descending, canonical signs); mu [k] the matching eigenvalues. With n < m
    ("gram" route) the directions come from the n x n Gram matrix Z Z^T: for its
    eigenpair (w, u), Z^T u / sqrt(w) is a unit eigenvector of Z^T Z with
    eigenvalue w. A symmetric eigensolver (LAPACK via numpy.linalg.eigh) is the
    library step.
    """
    Z = np.asarray(Z, np.float64)
    n, m = Z.shape
    if not (1 <= k <= min(n, m)):
        raise ValueError("k must satisfy 1 <= k <= min(n, m)")
    if route == "auto":
        route = "gram" if n < m else "cov"
    if route == "cov":
        C = Z.T @ Z / n
        w, V = np.linalg.eigh(C)
        idx = np.argsort(-w, kind="stable")[:k]
        P = V[:, idx]
        mu = w[idx]
    elif route == "gram":
        K = Z @ Z.T
        w, U = np.linalg.eigh(K)
        idx = np.argsort(-w, kind="stable")[:k]
        w = w[idx]
        U = U[:, idx]
        if np.any(w <= 0):
            raise ValueError("rank of Z below k")
        P = (Z.T @ U) / np.sqrt(w)[None, :]
        mu = w / n
    else:
        raise ValueError(route)
    return canonical_signs(P), mu


def fit_pca_from_moment(C: np.ndarray, n: int, k: int) -> Tuple[np.ndarray, np.ndarray]:
    """fit_pca's covariance route (App. B.2) from a second moment already summed
    over all n rows, C = sum_r z_r z_r^T (e.g. added up over shards): the top-k
    eigenvectors of C / n with the canonical signs, and their eigenvalues."""
    w, V = np.linalg.eigh(np.asarray(C, np.float64) / n)
    idx = np.argsort(-w, kind="stable")[:k]
    return canonical_signs(V[:, idx]), w[idx]


def project(z: np.ndarray, P: np.ndarray) -> np.ndarray:
    """x = P^T z for each row z of z [B, m] (Sec. 3.2, Eq. second_stage)."""
    return np.asarray(z, np.float64) @ np.asarray(P, np.float64)


def srht_width(m: int) -> int:
    """Padded width p = 2^ceil(log2 m) of the SRHT (App. B.2, Eq. app_srht_definition)."""
    p = 1
    while p < m:
        p *= 2
    return p


def srht(z: np.ndarray, signs: np.ndarray, rows: np.ndarray) -> np.ndarray:
    """EOGP-R second stage x = sqrt(p/k) R H_p D J z for each row z of z [B, m]
    (Sec. 3.2 "A scalable alternative to PCA"; App. B.2 Eq. app_srht_definition).

    J zero-pads to width p = 2^ceil(log2 m); D = diag(signs) (the m signs that
    meet non-padded coordinates; the others multiply zeros); H_p is the
    orthonormal Walsh-Hadamard matrix in Sylvester (natural) order,
    H_p[r, c] = (-1)^popcount(r & c) / sqrt(p), the ordering the paper leaves
    unstated; R keeps rows `rows` (k distinct indices in [0, p)) in the given
    order. The random signs and rows are inputs: the same realisation serves
    stored examples and queries. H_p is formed explicitly (a library matrix)."""
    import scipy.linalg
    z = np.asarray(z, np.float64)
    B, m = z.shape
    p = srht_width(m)
    k = len(rows)
    zp = np.zeros((B, p))
    zp[:, :m] = z * np.asarray(signs, np.float64)[None, :m]
    H = scipy.linalg.hadamard(p).astype(np.float64) / np.sqrt(p)
    return np.sqrt(p / k) * (zp @ H.T)[:, np.asarray(rows, np.int64)]


# --------------------------------------------------------------------------
# One-bit quantization and packing
# --------------------------------------------------------------------------

def onebit(x: np.ndarray) -> Tuple[np.ndarray, np.ndarray]:
    """Sign bits and scale of each row of x [B, k] (Sec. 3.3, Eq. onebit):
    bit = 1 encodes +1 (taken for x >= 0, so both zeros map to +1, which App. A.3
    permits), bit = 0 encodes -1; scale = ||x||_1 / k, the minimiser of
    ||x - s b||^2 (Eq. app_onebit_scale)."""
    x = np.asarray(x, np.float64)
    k = x.shape[-1]
    bits = (x >= 0)
    scale = np.abs(x).sum(axis=-1) / k
    return bits, scale


def pack_bits(bits: np.ndarray) -> np.ndarray:
    """Pack a boolean array [..., k] into little-endian uint32 words [..., ceil(k/32)]:
    coordinate c is bit (c % 32) of word c // 32, i.e. bit (c % 8) of byte c // 8
    in the per-module byte packing of App. E.1. Pad bits are 0."""
    bits = np.asarray(bits, bool)
    k = bits.shape[-1]
    W = (k + 31) // 32
    out = np.zeros(bits.shape[:-1] + (W,), np.uint64)
    for c in range(k):
        out[..., c // 32] |= bits[..., c].astype(np.uint64) << np.uint64(c % 32)
    return out.astype(np.uint32)


def unpack_bits(words: np.ndarray, k: int) -> np.ndarray:
    """Inverse of pack_bits: words [..., ceil(k/32)] -> bool [..., k]."""
    words = np.asarray(words, np.uint32).astype(np.uint64)
    out = np.zeros(words.shape[:-1] + (k,), bool)
    for c in range(k):
        out[..., c] = ((words[..., c // 32] >> np.uint64(c % 32)) & np.uint64(1)) == 1
    return out


def module_word_offsets(ks: Sequence[int]) -> List[int]:
    """Word offset of each module's codes in a concatenated row (each module
    starts on a fresh 32-bit word; its pad bits are zero)."""
    off, o = [], 0
    for k in ks:
        off.append(o)
        o += (k + 31) // 32
    off.append(o)
    return off


def pack_concat(bits_per_module: Sequence[np.ndarray]) -> np.ndarray:
    """Concatenate per-module packed codes along the word axis (each module packed
    on its own, App. E.1)."""
    return np.concatenate([pack_bits(b) for b in bits_per_module], axis=-1)


def _signs(words: np.ndarray, k: int) -> np.ndarray:
    return np.where(unpack_bits(words, k), 1.0, -1.0)


# --------------------------------------------------------------------------
# Scores
# --------------------------------------------------------------------------

def score_codes(train_codes: np.ndarray, train_scales: np.ndarray, ks: Sequence[int],
                query_codes: np.ndarray, query_scales: np.ndarray) -> np.ndarray:
    """Score of query q against stored example i with both sides one-bit:
    sum_u s_iu s_qu <b_iu, b_qu>, each b a +-1 vector (Sec. 3.3, Eq. onebit_influence
    with the query coordinates replaced by their own one-bit code). float64,
    +-1 sums formed explicitly (no popcount). Returns [Q, N]."""
    off = module_word_offsets(ks)
    Q, N = query_codes.shape[0], train_codes.shape[0]
    out = np.zeros((Q, N), np.float64)
    for u, k in enumerate(ks):
        bt = _signs(train_codes[:, off[u]:off[u + 1]], k)      # [N, k]
        bq = _signs(query_codes[:, off[u]:off[u + 1]], k)      # [Q, k]
        dot = bq @ bt.T
        out += np.asarray(query_scales, np.float64)[:, u, None] * \
            np.asarray(train_scales, np.float64)[None, :, u] * dot
    return out


def score_codes_f32(train_codes: np.ndarray, train_scales: np.ndarray, ks: Sequence[int],
                    query_codes: np.ndarray, query_scales: np.ndarray) -> np.ndarray:
    """The same score evaluated in a fixed float32 order: per module the integer
    +-1 dot d_u, then acc = fl(acc + fl(fl(s_iu * s_qu) * d_u)) in module order,
    no fused multiply-add. Used to check the dequantization bit for bit."""
    off = module_word_offsets(ks)
    Q, N = query_codes.shape[0], train_codes.shape[0]
    acc = np.zeros((Q, N), np.float32)
    ts = np.asarray(train_scales, np.float32)
    qs = np.asarray(query_scales, np.float32)
    for u, k in enumerate(ks):
        bt = _signs(train_codes[:, off[u]:off[u + 1]], k)
        bq = _signs(query_codes[:, off[u]:off[u + 1]], k)
        d = (bq @ bt.T).astype(np.float32)                     # exact integers
        sp = (qs[:, u, None] * ts[None, :, u]).astype(np.float32)
        acc = (acc + (sp * d).astype(np.float32)).astype(np.float32)
    return acc


def onebit_dot_xor(train_words: np.ndarray, query_words: np.ndarray, k: int) -> np.ndarray:
    """<b_i, b_q> of +-1 vectors of one module, for every stored row i of
    train_words [N, ceil(k/32)] against one query row query_words [ceil(k/32)],
    through the identity <b, b'> = k - 2 * #{c : b_c != b'_c}: the differing
    signs are the set bits of the XOR of the packed codes (pad bits are 0 on
    both sides), counted per word. A closed form of the +-1 sum that
    score_codes forms explicitly, for checks over millions of stored rows.
    Returns int64 [N]."""
    t = np.asarray(train_words, np.uint32)
    q = np.asarray(query_words, np.uint32)
    x = np.bitwise_xor(t, q[None, :])
    if hasattr(np, "bitwise_count"):
        diff = np.bitwise_count(x).sum(axis=1, dtype=np.int64)
    else:
        table = np.array([bin(v).count("1") for v in range(256)], np.int64)
        diff = table[x.view(np.uint8)].sum(axis=1)
    return k - 2 * diff


def score_paper(train_codes: np.ndarray, train_scales: np.ndarray, ks: Sequence[int],
                y: np.ndarray) -> np.ndarray:
    """Paper's asymmetric score sum_u s_iu <y_u, b_iu> with unquantized query
    coordinates y [Q, sum_u k_u] (Sec. 3.3 Eq. onebit_influence; App. B.3
    Eq. app_stored_influence). Returns [Q, N]."""
    off = module_word_offsets(ks)
    y = np.asarray(y, np.float64)
    Q, N = y.shape[0], train_codes.shape[0]
    out = np.zeros((Q, N), np.float64)
    c0 = 0
    for u, k in enumerate(ks):
        bt = _signs(train_codes[:, off[u]:off[u + 1]], k)
        out += (y[:, c0:c0 + k] @ bt.T) * np.asarray(train_scales, np.float64)[None, :, u]
        c0 += k
    return out


def score_fp(x_train: np.ndarray, y: np.ndarray) -> np.ndarray:
    """Unquantized score <y, x_i> over all modules' coordinates (Sec. 3.1: with
    V = M, influence is the inner product of the stored and query coordinates).
    x_train [N, D], y [Q, D] -> [Q, N]."""
    return np.asarray(y, np.float64) @ np.asarray(x_train, np.float64).T


def top_k(scores: np.ndarray, K: int) -> Tuple[np.ndarray, np.ndarray]:
    """Per query (row of scores [Q, N]) the K highest-scoring stored examples,
    best first (App. C: stored examples ranked by score, descending; NDCG@20
    reads the first 20). Equal scores rank the lower stored index first; NaN
    scores never rank; places past the ranked examples hold (-inf, -1).
    Returns (values [Q, K] float64, indices [Q, K] int64)."""
    scores = np.asarray(scores, np.float64)
    Q = scores.shape[0]
    vals = np.full((Q, K), -np.inf)
    idx = np.full((Q, K), -1, np.int64)
    for q in range(Q):
        row = scores[q]
        cand = np.flatnonzero(~np.isnan(row))
        order = cand[np.lexsort((cand, -row[cand]))][:K]   # key 1: score desc; key 2: index asc
        vals[q, :len(order)] = row[order]
        idx[q, :len(order)] = order
    return vals, idx


# --------------------------------------------------------------------------
# Storage accounting
# --------------------------------------------------------------------------

def payload_bytes(ks: Sequence[int], scale_bytes: int = 2) -> int:
    """Per-example payload sum_u (ceil(k_u / 8) + 2) bytes (App. E.1, Eq. app_payload)."""
    return int(sum((k + 7) // 8 + scale_bytes for k in ks))


def to_payload(codes: np.ndarray, scales: np.ndarray, ks: Sequence[int]) -> np.ndarray:
    """Per-example store records (App. E.1, Eq. app_payload): for each module in
    order, its ceil(k_u / 8) bytes of signs packed byte by byte (coordinate c at
    bit c % 8 of byte c / 8) followed by its scale as an IEEE half (round to
    nearest even, little-endian). The order of signs and scale inside a module's
    record is not stated in the paper; signs first is the reading taken here.
    codes [N, W] uint32 (module u at its word offset), scales [N, U] ->
    uint8 [N, payload_bytes(ks)]."""
    off = module_word_offsets(ks)
    parts = []
    for u, k in enumerate(ks):
        bits = unpack_bits(np.asarray(codes)[:, off[u]:off[u + 1]], k)
        parts.append(np.packbits(bits.astype(np.uint8), axis=1, bitorder="little"))
        half = np.asarray(scales, np.float32)[:, u].astype(np.float16)
        parts.append(half.astype("<f2").view(np.uint8).reshape(-1, 2))
    return np.concatenate(parts, axis=1)


def from_payload(payload: np.ndarray, ks: Sequence[int]) -> Tuple[np.ndarray, np.ndarray]:
    """Inverse of to_payload: (codes [N, W] uint32 with zero pad bits, scales
    [N, U] float32 holding the stored halves exactly)."""
    payload = np.asarray(payload, np.uint8)
    mods, scl, o = [], [], 0
    for k in ks:
        nb = (k + 7) // 8
        bits = np.unpackbits(payload[:, o:o + nb], axis=1, bitorder="little")[:, :k].astype(bool)
        mods.append(bits)
        scl.append(payload[:, o + nb:o + nb + 2].copy().view("<f2").astype(np.float32)[:, 0])
        o += nb + 2
    return pack_concat(mods), np.stack(scl, axis=1)


def correction_bytes(m: int, k: int) -> int:
    """FP16 PCA correction matrix P_u in R^{m x k}: 2 m k bytes (Eq. app_correction_storage)."""
    return 2 * m * k


# --------------------------------------------------------------------------
# Whole layer, for convenience
# --------------------------------------------------------------------------

def compress_layer(a, s, Q_A, Q_S, Lam, lam, m, P):
    """Store step of Alg. 1 for one module: x = P^T L g, then sign bits and scale.
    Returns (z [B, m], x [B, k], codes [B, ceil(k/32)], scales [B])."""
    z = first_stage(a, s, Q_A, Q_S, Lam, lam, m)
    x = project(z, P)
    bits, sc = onebit(x)
    return z, x, pack_bits(bits), sc
