"""Shared helpers of the test suite (comparison metrics, row sampling)."""
import numpy as np

# Tolerance for bf16-in / fp32-accumulate attention against the float64 oracle
TOL_MAX_ABS = 2e-2
TOL_REL_RMS = 1e-2


def attn_errors(got: np.ndarray, ref: np.ndarray):
    """(max |got - ref|, ||got - ref||_2 / ||ref||_2) over all elements."""
    diff = got.astype(np.float64) - ref
    max_abs = float(np.max(np.abs(diff))) if diff.size else 0.0
    den = float(np.linalg.norm(ref))
    rel = float(np.linalg.norm(diff) / den) if den > 0 else float(np.linalg.norm(diff))
    return max_abs, rel


def assert_attn_close(got, ref, what=""):
    assert np.all(np.isfinite(got)), f"{what}: non-finite outputs"
    max_abs, rel = attn_errors(got, ref)
    assert max_abs <= TOL_MAX_ABS and rel <= TOL_REL_RMS, \
        f"{what}: max|err| {max_abs:.3g} (<= {TOL_MAX_ABS}), rel RMS {rel:.3g} (<= {TOL_REL_RMS})"
    return max_abs, rel


def sample_rows(w, n_random: int = 512, seed: int = 0) -> np.ndarray:
    """Rows (b, h, i): the first, middle and last new row of every request for
    every q head of every kv group's first and last head, plus random rows."""
    rng = np.random.default_rng(seed)
    rows = set()
    for b in range(w.B):
        n = int(w.new_lens[b])
        if n == 0:
            continue
        for i in {0, n // 2, n - 1}:
            for g in range(w.Hkv):
                for h in {g * w.G, g * w.G + w.G - 1}:
                    rows.add((b, h, i))
    nonempty = [b for b in range(w.B) if w.new_lens[b] > 0]
    for _ in range(n_random):
        b = int(rng.choice(nonempty))
        rows.add((b, int(rng.integers(w.Hq)), int(rng.integers(int(w.new_lens[b])))))
    return np.array(sorted(rows), dtype=np.int32)


def gather_rows(out: np.ndarray, w, rows: np.ndarray) -> np.ndarray:
    cu = w.cu_new_lens
    return np.stack([out[cu[b] + i, h] for b, h, i in rows])
