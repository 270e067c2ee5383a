"""CPU checks of the index and fragment arithmetic of two kernels, restated in
numpy (no GPU):

* the causal tile attention (attn_prefill_kernel): the 128-byte-swizzled K/V
  tile layout, the ldmatrix addressing, the m16n8k16 fragment layouts of the
  PTX ISA (A row g / g+8 in registers a0..a3, B column g, accumulator rows g
  and g+8), the bf16 hi / lo split of the queries in rows 0-7 / 8-15 and of
  the probabilities, the causal mask and the output recombination, against
  direct attention on one 16-entry group;
* the sampler's selection (sample_kernel): per-thread sorted top lists,
  k warp-merge rounds with owner hand-off, the warp-0 merge of the warp
  lists, against a sorted reference, with ties and small vocabularies;
* the decode attention's stage rings (attn_mma_kernel, 10 and 20 stages):
  per-warp stage ownership and the mbarrier phase parities.
"""
import numpy as np


# ---- tile attention ------------------------------------------------------

def _bf16(x):
    x = np.asarray(x, np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return r.astype(np.uint32).view(np.float32)


def _rest(x):
    return np.float32(x) - _bf16(np.float32(x))


HALF = 16 * 128  # one box: 16 rows x 64 dims bf16


def _tile_off(row, c):  # mma_tile_off: byte offset of 16-byte chunk c of row `row`
    return (c >> 3) * HALF + row * 128 + (((c & 7) ^ (row & 7)) << 4)


def _store_tile(M):
    buf = np.zeros(HALF, np.float32)  # 2 boxes of 2 KB as 2-byte slots
    for r in range(16):
        for c in range(16):
            off = _tile_off(r, c) // 2
            buf[off:off + 8] = M[r, c * 8:(c + 1) * 8]
    return buf


def _ldsm_x4(buf, addr, trans=False):
    mats = [np.array([buf[addr[m * 8 + i]: addr[m * 8 + i] + 8] for i in range(8)]) for m in range(4)]
    out = []
    for lane in range(32):
        g, t = lane // 4, lane % 4
        if trans:
            out.append([(mats[m][2 * t, g], mats[m][2 * t + 1, g]) for m in range(4)])
        else:
            out.append([(mats[m][g, 2 * t], mats[m][g, 2 * t + 1]) for m in range(4)])
    return out


def _mma16(d, a, b):
    A, Bm, Cm = np.zeros((16, 16)), np.zeros((16, 8)), np.zeros((16, 8))
    for lane in range(32):
        g, t = lane // 4, lane % 4
        for i in range(2):
            A[g, 2 * t + i], A[g + 8, 2 * t + i] = a[lane][0][i], a[lane][1][i]
            A[g, 2 * t + 8 + i], A[g + 8, 2 * t + 8 + i] = a[lane][2][i], a[lane][3][i]
            Bm[2 * t + i, g], Bm[2 * t + 8 + i, g] = b[lane][0][i], b[lane][1][i]
            Cm[g, 2 * t + i], Cm[g + 8, 2 * t + i] = d[lane][i], d[lane][2 + i]
    D = Cm + A @ Bm
    return [[D[l // 4, 2 * (l % 4)], D[l // 4, 2 * (l % 4) + 1], D[l // 4 + 8, 2 * (l % 4)],
             D[l // 4 + 8, 2 * (l % 4) + 1]] for l in range(32)]


def test_tile_attention_fragment_arithmetic():
    rng = np.random.default_rng(0)
    DH = 128
    K = _bf16(rng.standard_normal((16, DH)).astype(np.float32))
    V = _bf16(rng.standard_normal((16, DH)).astype(np.float32))
    Q = (rng.standard_normal((8, DH)) * 0.1).astype(np.float32)  # rotated, pre-scaled queries
    qpos = [3, 7, 15, 15, 0, 9, 12, 5]  # each query attends to entries 0 .. qpos
    kbuf, vbuf = _store_tile(K), _store_tile(V)
    qa = []
    for lane in range(32):
        g, t = lane // 4, lane % 4
        frags = []
        for kc in range(8):
            d0 = kc * 16 + 2 * t
            x0, x1, x8, x9 = Q[g, d0], Q[g, d0 + 1], Q[g, d0 + 8], Q[g, d0 + 9]
            frags.append([(_bf16(x0), _bf16(x1)), (_bf16(_rest(x0)), _bf16(_rest(x1))),
                          (_bf16(x8), _bf16(x9)), (_bf16(_rest(x8)), _bf16(_rest(x9)))])
        qa.append(frags)
    sacc = [[[0.0] * 4 for _ in range(32)] for _ in range(2)]
    for nt in range(2):
        for kc2 in range(4):
            addr = [_tile_off(nt * 8 + (l & 7), 4 * kc2 + 2 * ((l >> 3) >> 1) + ((l >> 3) & 1)) // 2 for l in range(32)]
            bk = _ldsm_x4(kbuf, addr)
            sacc[nt] = _mma16(sacc[nt], [qa[l][2 * kc2] for l in range(32)], [[bk[l][0], bk[l][1]] for l in range(32)])
            sacc[nt] = _mma16(sacc[nt], [qa[l][2 * kc2 + 1] for l in range(32)],
                              [[bk[l][2], bk[l][3]] for l in range(32)])
    sv = np.full((32, 2, 2), -np.inf)
    for lane in range(32):
        g, t = lane // 4, lane % 4
        for nt in range(2):
            for j in range(2):
                if nt * 8 + 2 * t + j <= qpos[g]:
                    sv[lane, nt, j] = sacc[nt][lane][j] + sacc[nt][lane][2 + j]
    m = [max(sv[4 * (l // 4) + i].max() for i in range(4)) for l in range(32)]
    P = [np.where(sv[l] == -np.inf, 0, np.exp(sv[l] - m[l])) for l in range(32)]
    lsum = [sum(P[4 * (l // 4) + i].sum() for i in range(4)) for l in range(32)]
    pa = []
    for lane in range(32):
        pv = P[lane].astype(np.float32)
        pa.append([(_bf16(pv[0, 0]), _bf16(pv[0, 1])), (_bf16(_rest(pv[0, 0])), _bf16(_rest(pv[0, 1]))),
                   (_bf16(pv[1, 0]), _bf16(pv[1, 1])), (_bf16(_rest(pv[1, 0])), _bf16(_rest(pv[1, 1])))])
    o = [[[0.0] * 4 for _ in range(32)] for _ in range(16)]
    for nd2 in range(8):
        addr = [_tile_off((l & 7) + ((l >> 3) & 1) * 8, nd2 * 2 + ((l >> 3) >> 1)) // 2 for l in range(32)]
        bv = _ldsm_x4(vbuf, addr, trans=True)
        o[nd2 * 2] = _mma16(o[nd2 * 2], pa, [[bv[l][0], bv[l][1]] for l in range(32)])
        o[nd2 * 2 + 1] = _mma16(o[nd2 * 2 + 1], pa, [[bv[l][2], bv[l][3]] for l in range(32)])
    out = np.zeros((8, DH))
    for lane in range(32):
        g, t = lane // 4, lane % 4
        for nd in range(16):
            out[g, nd * 8 + 2 * t] = (o[nd][lane][0] + o[nd][lane][2]) / lsum[lane]
            out[g, nd * 8 + 2 * t + 1] = (o[nd][lane][1] + o[nd][lane][3]) / lsum[lane]
    for i in range(8):
        s = K[: qpos[i] + 1].astype(np.float64) @ Q[i].astype(np.float64)
        p = np.exp(s - s.max())
        ref = (p / p.sum()) @ V[: qpos[i] + 1].astype(np.float64)
        assert np.abs(out[i] - ref).max() < 1e-4, i


# ---- sampler selection ---------------------------------------------------

KMAX, THREADS, WARPS = 32, 256, 8
SENT = (-np.inf, 0x7FFFFFFF)


def _before(a, b):
    return a[0] > b[0] or (a[0] == b[0] and a[1] < b[1])


def _select(vals, k):
    V = len(vals)
    k = min(k, V)
    lists = []
    for t in range(THREADS):
        L = [SENT] * KMAX
        for i in range(t, V, THREADS):
            c = (float(vals[i]), i)
            if not _before(c, L[-1]):
                continue
            L[-1] = c
            for j in range(KMAX - 1, 0, -1):
                if _before(L[j], L[j - 1]):
                    L[j], L[j - 1] = L[j - 1], L[j]
        lists.append(L)
    wl = []
    for w in range(WARPS):
        ls = lists[w * 32:(w + 1) * 32]
        out = []
        for _ in range(k):
            best = ls[0][0]
            for l in ls[1:]:
                if _before(l[0], best):
                    best = l[0]
            for l in ls:
                if l[0] == best:
                    l.pop(0)
                    l.append(SENT)
            out.append(best)
        wl.append(out)
    pos = [0] * 32
    fin = []
    for _ in range(k):
        offers = [wl[l][pos[l]] if (l < WARPS and pos[l] < k) else SENT for l in range(32)]
        best = offers[0]
        for c in offers[1:]:
            if _before(c, best):
                best = c
        for l in range(32):
            if l < WARPS and pos[l] < k and offers[l] == best:
                pos[l] += 1
        fin.append(best)
    return fin


def test_sampler_selection_is_the_sorted_top_k():
    rng = np.random.default_rng(0)
    for trial in range(40):
        V = int(rng.choice([5, 31, 33, 257, 600, 3001]))
        k = int(rng.integers(1, 33))
        vals = rng.standard_normal(V).astype(np.float32)
        if trial % 3 == 0:
            vals = np.round(vals * 2) / 2  # ties: the lower id first
        ref = sorted(((float(vals[i]), i) for i in range(V)), key=lambda x: (-x[0], x[1]))[:min(k, V)]
        assert _select(vals, k) == ref, (V, k)


def test_decode_attention_fragment_arithmetic_the_same_way():
    """The same restatement applied to the decode tensor-core attention
    (attn_mma_kernel, verified on the GPU against the oracle): rows 0..G-1 of
    A hold the bf16 part of the G heads' queries, rows G..2G-1 the remainder,
    rows 8..15 zero; a head's score is row h plus row h + G (the lane 4G
    apart).  Agreement here ties the layouts assumed above to a kernel whose
    results are known."""
    rng = np.random.default_rng(1)
    DH, G = 128, 4
    K = _bf16(rng.standard_normal((16, DH)).astype(np.float32))
    Q = (rng.standard_normal((G, DH)) * 0.1).astype(np.float32)
    kbuf = _store_tile(K)
    qa = []
    for lane in range(32):
        r, t = lane // 4, lane % 4
        frags = []
        for kc in range(8):
            pair = []
            for half in range(2):
                d0 = kc * 16 + half * 8 + 2 * t
                if r < G:
                    x0, x1 = Q[r, d0], Q[r, d0 + 1]
                elif r < 2 * G:
                    x0, x1 = _rest(Q[r - G, d0]), _rest(Q[r - G, d0 + 1])
                else:
                    x0 = x1 = 0.0
                pair.append((_bf16(x0), _bf16(x1)))
            frags.append([pair[0], (0.0, 0.0), pair[1], (0.0, 0.0)])  # a1 = a3 = 0: rows 8-15 zero
        qa.append(frags)
    sacc = [[[0.0] * 4 for _ in range(32)] for _ in range(2)]
    for nt in range(2):
        for kc2 in range(4):
            addr = [_tile_off(nt * 8 + (l & 7), 4 * kc2 + 2 * ((l >> 3) >> 1) + ((l >> 3) & 1)) // 2 for l in range(32)]
            bk = _ldsm_x4(kbuf, addr)
            sacc[nt] = _mma16(sacc[nt], [qa[l][2 * kc2] for l in range(32)], [[bk[l][0], bk[l][1]] for l in range(32)])
            sacc[nt] = _mma16(sacc[nt], [qa[l][2 * kc2 + 1] for l in range(32)],
                              [[bk[l][2], bk[l][3]] for l in range(32)])
    ref = K.astype(np.float64) @ Q.astype(np.float64).T  # [16 entries][G heads]
    for lane in range(32):
        r, t = lane // 4, lane % 4
        if r >= G:
            continue
        partner = lane ^ (4 * G)  # the lane holding row r + G
        for nt in range(2):
            for j in range(2):
                score = sacc[nt][lane][j] + sacc[nt][partner][j]
                assert abs(score - ref[nt * 8 + 2 * t + j, r]) < 1e-4


def _mma_stage(t, st, nw=5):
    """Stage of group t in attn_mma_kernel's ring of st stages (nw compute
    warps, st / nw stages each), restated."""
    spw = st // nw
    return (t % nw) * spw + (t // nw) % spw


def test_decode_attention_stage_ring_phases():
    """The tensor-core decode attention's stage rings (10 stages, and 20 for
    the deep ring): group t goes to compute warp t % 5 and only through that
    warp's own stages; the k-th group through a stage is its phase k, so the
    consumer's parity (t / ST) & 1 and the producer's wait for the stage's
    previous consumption (parity ((t / ST) & 1) ^ 1, from t >= ST) name the
    right phases; and the first ST groups (issued before any wait) use ST
    distinct stages."""
    for st in (10, 20):
        spw = st // 5
        uses = {}
        for t in range(12 * st):
            s = _mma_stage(t, st)
            assert 0 <= s < st and s // spw == t % 5  # the consuming warp's own stages
            k = len(uses.setdefault(s, []))
            assert (t // st) & 1 == k & 1  # consumer parity = phase k
            if t >= st:
                assert k >= 1 and ((t // st) & 1) ^ 1 == (k - 1) & 1  # previous consumption
            uses[s].append(t)
        assert sorted(_mma_stage(t, st) for t in range(st)) == list(range(st))
        # a warp's consecutive groups cycle through its stages in order
        for w in range(5):
            seq = [_mma_stage(t, st) for t in range(w, 6 * st, 5)]
            assert seq[:spw] == [w * spw + j for j in range(spw)] and seq[spw:2 * spw] == seq[:spw]
