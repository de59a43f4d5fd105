"""CPU transcriptions of the tile sets the inverse Cholesky's kernels walk (csrc/trail_tc.cu,
csrc/chol.cu), and of its blocked schedule, checked for coverage and for the algebra.

The two-level inverse Cholesky (Algorithm 2's Inverse_Cholesky, computed by the
reverse-order route C = chol(J H J), Z = C^-1, L = J Z^T J) splits its work into tile sets
that different launches cover. These tests restate each set's index arithmetic in Python
and check that the launches of one super-panel write every block exactly once. They then
run the whole blocked schedule in float64 on small blocks and compare L with the Cholesky
factor of the inverse (Proposition 1: H^-1 = L L^T).
"""
import numpy as np
import pytest


# ---------------------------------------------------------------- pair kernel, mode 1
def pair_mode1_blocks(nbk, a_j0, a_j1, a_r0, a_r1, b_i0, b_i1, b_j1):
    """Blocks (region, i, j) written by the two-CTA kernel's Cholesky tile set
    (pair_tile_at, mode 1, with the host's tile counts from chol_update_tc)."""
    n_a = sum(max(0, (a_r1 - max(jp, a_r0) + 1) // 2) for jp in range(a_j0, a_j1, 2))
    n_b = ((b_i1 - b_i0 + 1) // 2) * ((b_j1 + 1) // 2) if (b_i1 > b_i0 and b_j1 > 0) else 0
    out = []
    for t0 in range(n_a + n_b):
        for rank in (0, 1):
            t = t0
            if t < n_a:
                jp = a_j0
                while t >= (a_r1 - max(jp, a_r0) + 1) // 2:
                    t -= (a_r1 - max(jp, a_r0) + 1) // 2
                    jp += 2
                i = max(jp, a_r0) + 2 * t + rank
                if i < a_r1:
                    out.append(("A", i, jp))
                if i < a_r1 and jp + 1 < a_j1 and jp + 1 <= i:
                    out.append(("A", i, jp + 1))
            else:
                t -= n_a
                ncp = (b_j1 + 1) // 2
                i = b_i0 + 2 * (t // ncp) + rank
                j0 = 2 * (t % ncp)
                if i < b_i1:
                    out.append(("Z", i, j0))
                if i < b_i1 and j0 + 1 < b_j1:
                    out.append(("Z", i, j0 + 1))
    return out


@pytest.mark.parametrize("nbk", [9, 10, 11, 12, 17, 32, 64, 224, 225])
def test_far_update_parts_cover_every_block_once(nbk):
    """The next diagonal block's part (caller's stream) and the rest (second stream) of a
    super-panel's update write the lower blocks of A right of the super-panel and the blocks
    of Z below it, left of its end, each exactly once; the first part stays in the next
    diagonal block."""
    for k0 in range(0, nbk, 8):
        k1 = min(nbk, k0 + 8)
        if k1 >= nbk:
            continue
        k2 = min(nbk, k1 + 8)
        head = pair_mode1_blocks(nbk, k1, k2, 0, k2, 0, 0, 0)
        rest = pair_mode1_blocks(nbk, k1, nbk, k2, nbk, k1, nbk, k1)
        got = head + rest
        assert len(got) == len(set(got))
        want = {("A", i, j) for j in range(k1, nbk) for i in range(j, nbk)}
        want |= {("Z", i, j) for i in range(k1, nbk) for j in range(k1)}
        assert set(got) == want
        assert all(k1 <= i < k2 and k1 <= j < k2 for _, i, j in head)


# ---------------------------------------------------------------- persistent walk
def round_tile(rd, pair, npairs):
    return rd * npairs + ((npairs - 1 - pair) if rd & 1 else pair)


@pytest.mark.parametrize("n_tiles,npairs", [(1, 76), (75, 76), (76, 76), (96, 76), (432, 76), (433, 68), (7, 3)])
def test_alternating_walk_visits_every_tile_once(n_tiles, npairs):
    seen = []
    for pair in range(npairs):
        rd = 0
        while rd * npairs < n_tiles:
            t = round_tile(rd, pair, npairs)
            if t < n_tiles:
                seen.append(t)
            rd += 1
    assert sorted(seen) == list(range(n_tiles))


def test_alternating_walk_balances_growing_k():
    """Column tiles with K bounds 1:2:3:4 (the C_DS product) on 76 clusters: the busiest
    cluster's K drops from the plain stride's to within one tile of the mean."""
    n_col, npairs = 4, 76
    for n_row in (24, 108):
        n_tiles = n_row * n_col
        cost = lambda t: t % n_col + 1
        plain = [sum(cost(t) for t in range(p, n_tiles, npairs)) for p in range(npairs)]
        alt = [sum(cost(round_tile(rd, p, npairs)) for rd in range(-(-n_tiles // npairs))
                   if round_tile(rd, p, npairs) < n_tiles) for p in range(npairs)]
        assert sum(plain) == sum(alt)
        assert max(alt) < max(plain)
        assert max(alt) <= sum(alt) / npairs + n_col


# ---------------------------------------------------------------- chain kernels
def rest_tiles(k, k0, k1):
    """chol_rest_kernel's tiles for step k inside blocks [k0, k1)."""
    m = k1 - k - 2
    out = []
    for t0 in range(m * (m + 1) // 2 + m * (k - k0 + 1)):
        t = t0
        if t < m * (m + 1) // 2:
            j = k + 2
            while t >= k1 - j:
                t -= k1 - j
                j += 1
            out.append((j + t, j))
        else:
            t -= m * (m + 1) // 2
            nzc = k - k0 + 1
            out.append((k + 2 + t // nzc, k0 + t % nzc))
    return out


def test_rest_kernel_tiles():
    for k0, k1 in [(0, 8), (8, 16), (0, 3), (16, 19)]:
        for k in range(k0, k1 - 2):
            got = rest_tiles(k, k0, k1)
            want = [(i, j) for j in range(k + 2, k1) for i in range(j, k1)]
            want += [(i, j) for i in range(k + 2, k1) for j in range(k0, k + 1)]
            assert sorted(got) == sorted(want) and len(set(got)) == len(got)


# ---------------------------------------------------------------- the blocked schedule
def blocked_inverse_cholesky(H, nb, spb):
    """The library's schedule on nb-blocks and super-panels of spb blocks, in float64:
    per step the diagonal block, the panel and the updates inside the super-panel only;
    then C_DS = A'_DS Z_SS^T and Z_SP = Z_SS B'_SP; then the update of every block beyond."""
    n = H.shape[0]
    npad = -(-n // nb) * nb
    nbk = npad // nb
    A = np.eye(npad)
    A[:n, :n] = H[::-1, ::-1]
    Z = np.zeros((npad, npad))
    b = lambda i: slice(i * nb, (i + 1) * nb)
    two = nbk > spb
    for k0 in range(0, nbk, spb if two else nbk):
        k1 = min(nbk, k0 + spb) if two else nbk
        for k in range(k0, k1):
            ci = np.linalg.inv(np.linalg.cholesky(A[b(k), b(k)]))
            Z[b(k), b(k)] = ci
            for q in range(k0, k1 - 1):                       # chol_panel_kernel, b0 = k0
                if q < k:
                    Z[b(k), b(q)] = ci @ Z[b(k), b(q)]
                else:
                    A[b(q + 1), b(k)] = A[b(q + 1), b(k)] @ ci.T
            if k + 1 >= k1:
                break

            def upd(i, j):                                    # update_quad
                if j > k:
                    A[b(i), b(j)] -= A[b(i), b(k)] @ A[b(j), b(k)].T
                else:
                    Z[b(i), b(j)] -= A[b(i), b(k)] @ Z[b(k), b(j)]
            for q in range(k0, k1):                           # chol_next_kernel, b0 = k0
                upd(k + 1, q) if q < k + 2 else upd(q, k + 1)
            for i, j in rest_tiles(k, k0, k1):
                upd(i, j)
        if not two:
            continue
        s0, s1 = k0 * nb, k1 * nb
        zss = Z[s0:s1, s0:s1].copy()
        A[s1:, s0:s1] = A[s1:, s0:s1] @ zss.T                 # C_DS
        Z[s0:s1, :s0] = zss @ Z[s0:s1, :s0]                   # Z_SP
        if k1 < nbk:
            cd = A[s1:, s0:s1]
            A[s1:, s1:] -= np.tril(cd @ cd.T)
            Z[s1:, :s1] -= cd @ Z[s0:s1, :s1]
    return Z[:n, :n].T[::-1, ::-1]                            # L[i][j] = Z[n-1-j][n-1-i]


@pytest.mark.parametrize("n,nb,spb", [(7, 4, 3), (24, 4, 3), (50, 4, 3), (100, 4, 8), (36, 4, 8), (37, 4, 2), (200, 8, 4)])
def test_blocked_schedule_gives_the_inverse_factor(n, nb, spb):
    rng = np.random.default_rng(n)
    X = rng.standard_normal((3 * n, n))
    H = X.T @ X + 0.01 * np.trace(X.T @ X) / n * np.eye(n)
    L = blocked_inverse_cholesky(H, nb, spb)
    ref = np.linalg.cholesky(np.linalg.inv(H))
    assert np.allclose(np.triu(L, 1), 0.0)
    assert np.linalg.norm(np.tril(L) - ref) <= 1e-12 * np.linalg.norm(ref)
