"""CPU emulation of the Transformer tensor-core kernel's data movement (csrc/mca_tfm_tc.cu).

Test infrastructure: it is neither the kernel nor the oracle. It repeats the kernel's index arithmetic
step by step -- shared memory as a float array addressed in bytes, tensor memory as 128 lanes x 512
columns, each MMA executed from its decoded shared-memory descriptors under the canonical K-major
no-swizzle operand layout (core matrices of 8 rows x 16 bytes; LBO between core matrices adjacent in
K, SBO between 8-row groups) with tf32 operands, each bulk copy performed when it is issued (the
earliest it can complete, the worst case for overwriting live data), and each mbarrier wait checked
against the phases issued so far (the awaited phase complete and not lapped). Its losses are compared
with the oracle's, so a wrong offset, descriptor, chunk order, swizzle or rank-1 term in the kernel's
design shows up on the CPU. What it cannot show: the hardware's behaviour, races between threads,
and anything the kernel does differently from what is repeated here.
"""
import numpy as np

from oracle.mca_oracle import act_fn

f32 = np.float32
kThreads, kRows, kD, kT, kHc, kXLd = 512, 128, 128, 64, 64, 132
kStages, kStageBytes = 5, 16384
kXsBytes = kRows * kXLd * 4
kAloBytes = kRows * kD * 4
kSmem = kXsBytes + kAloBytes + kStages * kStageBytes
kALBO = (kRows // 8) * 128
kColQ, kColK, kColV, kColA = 0, 128, 256, 384
kColU, kColF, kColA2, kColA2lo = 0, 128, 256, 320
kQkvChunks, kWoChunk0, kFfnChunk0, kFfnPerPair, kHeadChunks = 24, 24, 32, 16, 8
kHp = 128           # hidden columns per W1 product (two 64-wide chunks)
kTcQ, kTcK, kTcV, kTcO, kTcW1, kTcW2, kTcHead, kNone = 0, 1, 2, 3, 4, 5, 6, -1
EVAL, COMMIT, FORWARD = 0, 1, 2


def idesc(M, N):
    return (1 << 4) | (2 << 7) | (2 << 10) | ((N >> 3) << 17) | ((M >> 4) << 24)


kIdN128 = idesc(128, 128)


def tf32_rna(x):
    x = np.asarray(x, dtype=np.float32)
    b = x.view(np.uint32).astype(np.uint64)
    b = (b + 0x1000) & 0xFFFFE000
    return b.astype(np.uint32).view(np.float32)


def tf32_trunc(x):
    x = np.asarray(x, dtype=np.float32)
    return (x.view(np.uint32) & np.uint32(0xFFFFE000)).view(np.float32)


def umma_desc(saddr, lbo, sbo):
    return ((saddr >> 4) & 0x3FFF) | (((lbo >> 4) & 0x3FFF) << 16) | (((sbo >> 4) & 0x3FFF) << 32) | (1 << 46)


# ---------------------------------------------------------------- layout (ports of the C++ header)

def tc_image_index(r, k, R, cols):
    return ((r // R) * (cols >> 4) + (k >> 4)) * R * 32 + ((k >> 2) & 3) * R * 4 + (r % R) * 4 + (k & 3)


def blk_floats(F):
    return 4 * 32768 + 512 * F


def image_offset(mat, b, r, k, F, nL):
    blk = blk_floats(F)
    if mat == kTcHead:
        return nL * blk + tc_image_index(r, k, 128, kD)
    base = b * blk
    if mat <= kTcO:
        return base + mat * 32768 + tc_image_index(r, k, 128, kD)
    if mat == kTcW1:
        return base + 131072 + tc_image_index(r, k, 128, kD)
    return base + 131072 + 256 * F + tc_image_index(r, k, 128, F)


def lo_off(mat):
    return 128 * 16


class Args:
    def __init__(self, spec, params, tokens):
        d, f, v, c = spec.d_model, spec.d_ff, spec.vocab, spec.ctx
        self.V, self.T, self.d, self.H, self.F, self.nL = v, c, d, spec.n_head, f, spec.n_layer
        self.B = tokens.shape[0]
        self.eps = f32(spec.ln_eps)
        self.act, self.g = spec.act, spec.act_param
        self.o_tok, self.o_pos = 0, v * d
        self.o_blk0 = self.o_pos + c * d
        sizes = [d, d, d * d, d, d * d, d, d * d, d, d * d, d, d, d, f * d, f, d * f, d]
        r, o = [], 0
        for s in sizes:
            r.append(o)
            o += s
        (self.r_ln1g, self.r_ln1b, self.r_wq, self.r_bq, self.r_wk, self.r_bk, self.r_wv, self.r_bv,
         self.r_wo, self.r_bo, self.r_ln2g, self.r_ln2b, self.r_w1, self.r_b1, self.r_w2,
         self.r_b2) = r
        self.blk_size = o
        self.o_lnf_g = self.o_blk0 + spec.n_layer * o
        self.o_lnf_b = self.o_lnf_g + d
        self.o_wh = self.o_lnf_b + d
        self.o_bh = self.o_wh + v * d
        self.P = self.o_bh + v
        self.params = np.array(params, dtype=np.float32)
        assert self.P == self.params.shape[0]
        self.tokens = np.asarray(tokens, dtype=np.int32)
        self.X = np.zeros((self.nL + 1, self.B, c, d), np.float32)
        self.Xmid = np.zeros((self.nL, self.B, c, d), np.float32)   # after each block's attention
        self.ell = np.zeros(self.B, np.float32)
        self.wimg = None

    def split(self):
        F, nL = self.F, self.nL
        wimg = np.zeros(nL * blk_floats(F) + 32768, np.float32)
        for slot in range(6 * nL + 1):
            rows = cols = kD
            if slot == 6 * nL:
                mat, b, src = kTcHead, 0, self.o_wh
            else:
                b, mat = divmod(slot, 6)
                base = self.o_blk0 + b * self.blk_size
                src = base + [self.r_wq, self.r_wk, self.r_wv, self.r_wo, self.r_w1, self.r_w2][mat]
                if mat == kTcW1:
                    rows = F
                if mat == kTcW2:
                    cols = F
            e = np.arange(rows * cols)
            r, kk = e // cols, e % cols
            valid = ~((mat == kTcHead) & (r >= self.V))
            w = np.zeros(rows * cols, np.float32)
            w[valid] = self.params[src + e[valid]]
            hi = tf32_rna(w)
            lo = tf32_rna(w - hi)
            o = image_offset(mat, b, r, kk, F, nL)
            wimg[o] = hi
            wimg[o + lo_off(mat)] = lo
        self.wimg = wimg


def tc_target(a, idx, stage):
    if 0 <= stage < a.nL:
        off = idx - a.o_blk0 - stage * a.blk_size
        dd, fd = a.d * a.d, a.F * a.d
        t = (kNone, 0, 0)
        for m, rq in enumerate([a.r_wq, a.r_wk, a.r_wv, a.r_wo]):
            if rq <= off < rq + dd:
                t = (m, (off - rq) // a.d, (off - rq) % a.d)
        if a.r_w1 <= off < a.r_w1 + fd:
            t = (kTcW1, (off - a.r_w1) // a.d, (off - a.r_w1) % a.d)
        if a.r_w2 <= off < a.r_w2 + fd:
            t = (kTcW2, (off - a.r_w2) // a.F, (off - a.r_w2) % a.F)
        return t
    if stage == a.nL and a.o_wh <= idx < a.o_wh + a.V * a.d:
        return (kTcHead, (idx - a.o_wh) // a.d, (idx - a.o_wh) % a.d)
    return (kNone, 0, 0)


def tfm_stage(a, idx):
    if idx < a.o_blk0:
        return -1
    if idx < a.o_lnf_g:
        return (idx - a.o_blk0) // a.blk_size
    return a.nL


RESTART_BLOCK, RESTART_FFN, RESTART_UNIT = 0, 1, 2


def restart(a, idx, stage):
    """Where a recomputation starts in block `stage`: its input, its mid stream (LN2 parameters) or
    one hidden unit of its feed-forward network (W1, b1, W2, b2: a rank-1 step, then stage + 1)."""
    if not 0 <= stage < a.nL:
        return RESTART_BLOCK
    off = idx - a.o_blk0 - stage * a.blk_size
    if off < a.r_ln2g:
        return RESTART_BLOCK
    return RESTART_FFN if off < a.r_w1 else RESTART_UNIT


def ffn_param(a, idx, stage):
    """A parameter of block `stage`'s feed-forward sub-block (LN2, W1, b1, W2, b2)."""
    return restart(a, idx, stage) != RESTART_BLOCK


def ffn_unit(a, cand, s0):
    """The kernel's rank-1 step for a hidden-unit candidate of block b: block b's new output
    stream for sequences s0, s0 + 1 ([128, d], rows as in the CTA), from the cached streams. The
    candidate's own entry enters at its old value (cand[5])."""
    idx, neww, delta, b, row, old = cand
    delta = f32(delta)
    base = a.o_blk0 + b * a.blk_size
    off = idx - base
    d, F = a.d, a.F
    P = a.params
    xn = a.X[b + 1, s0:s0 + 2].reshape(128, d).copy()
    if off >= a.r_b2:                                   # b2[i]
        xn[:, off - a.r_b2] += delta
        return xn
    x = a.Xmid[b, s0:s0 + 2].reshape(128, d)

    def part(v):        # the kernel's order: partial sums of four 32-column parts, left to right
        q = [v[:, 32 * g:32 * g + 32].astype(np.float32).sum(1, dtype=np.float32) for g in range(4)]
        return ((q[0] + q[1]) + q[2]) + q[3]

    mean = (part(x) / f32(d)).astype(np.float32)
    e = (x - mean[:, None]).astype(np.float32)
    var = (part(e * e) / f32(d)).astype(np.float32)
    rstd = (1.0 / np.sqrt(var.astype(np.float64) + float(a.eps))).astype(np.float32)
    ln = (e * rstd[:, None] * P[base + a.r_ln2g:base + a.r_ln2g + d] +
          P[base + a.r_ln2b:base + a.r_ln2b + d]).astype(np.float32)
    kcol = -1
    if off < a.r_b1:                                    # W1[j][kcol]
        j, kcol = divmod(off - a.r_w1, d)
    elif off < a.r_w2:                                  # b1[j]
        j = off - a.r_b1
    else:                                               # W2[i0][j]
        i0, j = divmod(off - a.r_w2, F)
    w1 = P[base + a.r_w1 + j * d:base + a.r_w1 + (j + 1) * d].copy()
    if kcol >= 0:
        w1[kcol] = old
    bj = f32(old) if a.r_b1 <= off < a.r_w2 else P[base + a.r_b1 + j]
    u = (part((ln * w1).astype(np.float32)) + bj).astype(np.float32)
    fu = act_fn(a.act, u.astype(np.float64), a.g).astype(np.float32)
    if off >= a.r_w2:
        xn[:, i0] += delta * fu
        return xn
    un = (u + delta * ln[:, kcol]) if kcol >= 0 else (u + delta)
    da = (act_fn(a.act, un.astype(np.float32).astype(np.float64), a.g).astype(np.float32) - fu)
    w2 = P[base + a.r_w2 + j:base + a.r_w2 + d * F:F]
    return (xn + w2[None, :] * da[:, None]).astype(np.float32)

# ---------------------------------------------------------------- the CTA

class Bar:
    def __init__(self):
        self.k = 0          # completed phases


class Slot:
    """A candidate's scratch slot: the residual streams and sequence losses its evaluation writes."""
    def __init__(self, a):
        self.X = np.full_like(a.X, np.nan)
        self.Xmid = np.full_like(a.Xmid, np.nan)
        self.ell = np.full_like(a.ell, np.nan)


def adopt(a, slot, cand):
    """The adopt kernel: the accepted candidate's recomputed streams (X[0..] and Xmid[0..] for an
    embedding; X[b+1..] and Xmid[b..] for block b, Xmid[b+1..] for its feed-forward sub-block; none
    for the head stage) and losses from its slot, sequences it skipped (a token embedding whose
    token they lack) left as they are."""
    idx, neww, delta, layer, row = cand[:5]
    if delta == 0.0:
        return
    first = 0 if layer < 0 else layer + 1
    first_mid = 0 if layer < 0 else (layer + 1 if ffn_param(a, idx, layer) else layer)
    for s in range(a.B):
        if row >= 0 and np.all(a.tokens[s, :kT] != row):
            continue
        a.ell[s] = slot.ell[s]
        for x in range(first, a.nL + 1):
            a.X[x, s] = slot.X[x, s]
        for x in range(first_mid, a.nL):
            a.Xmid[x, s] = slot.Xmid[x, s]


class CTA:
    def __init__(self, a, mode, cand, pair, slot=None):
        self.a, self.mode, self.pair = a, mode, pair
        self.slot = slot    # EVAL: the candidate's scratch slot, if it has one
        self.sm = np.zeros(kSmem // 4, np.float32)
        self.tm = np.zeros((128, 512), np.float32)
        self.full = [Bar() for _ in range(kStages)]
        self.empty = [Bar() for _ in range(kStages)]
        self.cand = cand    # (idx, neww, delta, layer, row, old) or None for forward

    # shared memory by byte address
    def smf(self, byte_addr):
        assert np.all(np.asarray(byte_addr) % 4 == 0)
        return np.asarray(byte_addr) // 4

    def wait(self, bar, x):
        e = x // kStages
        assert bar.k == e + 1, ("mbarrier wait", bar.k, e)

    # -------- ring
    def chunk_src(self, x):
        A = self.a
        if x < self.nbc:
            jb, q = divmod(x + self.q0, self.cpb)
            base = (self.b0s + jb) * blk_floats(A.F)
            if q < kFfnChunk0:
                return base + q * 4096, 16384
            f = q - kFfnChunk0
            p, u = divmod(f, kFfnPerPair)
            if u < 8:
                return base + 131072 + (p * 8 + u) * 4096, 16384
            return base + 131072 + 256 * A.F + (p * 8 + u - 8) * 4096, 16384
        return A.nL * blk_floats(A.F) + (x - self.nbc) * 4096, 16384

    def topup(self, upto):
        end = min(upto, self.limit)
        while self.nload < end:
            x = self.nload
            st = x % kStages
            if x >= kStages:
                self.wait(self.empty[st], x - kStages)
            src, nbytes = self.chunk_src(x)
            dst = (kXsBytes + kAloBytes + st * kStageBytes) // 4
            # overwrite hazard: record which bytes a load covers at issue time
            self.sm[dst:dst + nbytes // 4] = self.a.wimg[src:src + nbytes // 4]
            self.loaded_regions.append((x, dst * 4, nbytes))
            self.full[st].k += 1
            self.nload += 1

    def gather(self, desc, rows):
        start = (desc & 0x3FFF) << 4
        lbo = ((desc >> 16) & 0x3FFF) << 4
        sbo = ((desc >> 32) & 0x3FFF) << 4
        n = np.arange(rows)[:, None]
        k = np.arange(8)[None, :]
        addr = start + (n // 8) * sbo + (k // 4) * lbo + (n % 8) * 16 + (k % 4) * 4
        return tf32_trunc(self.sm[self.smf(addr)])

    def mma(self, d, adesc, bdesc, idsc, acc, a_tmem):
        N = ((idsc >> 17) & 0x3F) << 3
        M = ((idsc >> 24) & 0x1F) << 4
        assert M == 128
        B = self.gather(bdesc, N).astype(np.float64)
        if a_tmem:
            col = adesc & 0xFFFF
            assert (adesc >> 16) == 0
            A = tf32_trunc(self.tm[:M, col:col + 8]).astype(np.float64)
        else:
            A = self.gather(adesc, M).astype(np.float64)
        dcol = d & 0xFFFF
        D = (A @ B.T).astype(np.float32)
        if acc:
            self.tm[:M, dcol:dcol + N] = (self.tm[:M, dcol:dcol + N].astype(np.float64) + D).astype(np.float32)
        else:
            self.tm[:M, dcol:dcol + N] = D

    def issue(self, x0, n):
        salo, sw = kXsBytes, kXsBytes + kAloBytes
        for x in range(x0, x0 + n):
            st = x % kStages
            self.wait(self.full[st], x)
            self.nwait = x + 1
            dcol, idsc, alo, acol, R = kColU, kIdN128, salo, kColA, 128
            lo_tm = False                       # A's lo part in tensor memory (A2)
            if x < self.nbc:
                q = (x + self.q0) % self.cpb
                if q < kWoChunk0:
                    dcol = kColQ + 128 * (q >> 3)
                    kc = q & 7
                    first = kc == 0
                elif q < kFfnChunk0:
                    kc = q - kWoChunk0
                    first = kc == 0
                else:
                    f = q - kFfnChunk0
                    p, u = divmod(f, kFfnPerPair)
                    if u < 8:
                        kc = u
                        first = kc == 0
                    else:
                        dcol, lo_tm, acol, kc = kColF, True, kColA2, (u - 8) & 3
                        first = p == 0 and u == 8
            else:
                kc = x - self.nbc
                first = kc == 0
            lbo = R * 16
            for ks in range(2):
                gk = kc * 2 + ks
                da = umma_desc(alo + gk * 2 * kALBO, kALBO, 128)
                wb = sw + st * kStageBytes + ks * 2 * lbo
                dwhi = umma_desc(wb, lbo, 128)
                dwlo = umma_desc(wb + 4 * lbo, lbo, 128)
                ta = acol + gk * 8
                if lo_tm:
                    self.mma(dcol, kColA2lo + gk * 8, dwhi, idsc, 0 if (first and ks == 0) else 1, True)
                else:
                    self.mma(dcol, da, dwhi, idsc, 0 if (first and ks == 0) else 1, False)
                self.mma(dcol, ta, dwlo, idsc, 1, True)
                self.mma(dcol, ta, dwhi, idsc, 1, True)
            self.empty[st].k += 1
            self.ncommit = x + 1
            self.topup(x + kStages)

    def group_done(self, last):
        self.wait(self.empty[last % kStages], last)

    # -------- per-thread helpers, vectorised over (g, r)
    def prm(self, idx):
        idx = np.asarray(idx, dtype=np.int64)
        v = self.a.params[idx]
        return np.where(idx == self.midx, f32(self.mval), v).astype(np.float32)

    def xr_addr(self, g):
        r = np.arange(128)
        return (r * kXLd + 32 * g)  # float index of element 0 of the thread's 32

    def store_a(self, v, col, lo_base_bytes, k0, g, N):
        # v: [128 rows, N]; col, k0: this part's tensor-memory column and first K index
        r = np.arange(128)
        for h in range(N // 16):
            seg = v[:, 16 * h:16 * h + 16].astype(np.float32)
            hi = tf32_rna(seg)
            lo = tf32_rna(seg - hi)
            self.tm[:, col + 16 * h: col + 16 * h + 16] = hi
            for q in range(4):
                k = k0 + 16 * h + 4 * q
                addr = lo_base_bytes + (k >> 2) * kALBO + r * 16
                fi = self.smf(addr)
                for e in range(4):
                    self.sm[fi + e] = lo[:, 4 * q + e]

    def store_a2(self, v, col, lo_col):
        # v: [128 rows, 16]: hi and lo tf32 parts into tensor-memory columns col.. and lo_col..
        seg = v.astype(np.float32)
        hi = tf32_rna(seg)
        self.tm[:, col:col + 16] = hi
        self.tm[:, lo_col:lo_col + 16] = tf32_rna(seg - hi)

    def ln_to_a(self, og, ob, stash):
        x = np.stack([self.sm[self.xr_addr(g)[:, None] + np.arange(32)[None, :]] for g in range(4)])  # [4,128,32]
        s = np.zeros((4, 128), np.float32)
        for i in range(32):
            s = (s + x[:, :, i]).astype(np.float32)
        mean = ((((s[0] + s[1]) + s[2]) + s[3]) / f32(kD)).astype(np.float32)
        v = np.zeros((4, 128), np.float32)
        for i in range(32):
            e = (x[:, :, i] - mean).astype(np.float32)
            v = (e * e + v).astype(np.float32)
        var = ((((v[0] + v[1]) + v[2]) + v[3]) / f32(kD)).astype(np.float32)
        rstd = (1.0 / np.sqrt(var.astype(np.float64) + float(self.a.eps))).astype(np.float32)
        out = np.zeros_like(x)
        for g in range(4):
            for i in range(32):
                col = 32 * g + i
                out[g, :, i] = ((x[g, :, i] - mean) * rstd * self.prm(og + col) + self.prm(ob + col)).astype(np.float32)
                if col == stash:
                    self.s_acol = out[g, :, i].copy()
        for g in range(4):
            self.store_a(out[g], kColA + 32 * g, kXsBytes, 32 * g, g, 32)

    def attention(self, q):
        # q: [4 (head), 128, 32]; K, V in shared memory (swizzled slots)
        a = self.a
        scale = f32(1.0 / np.sqrt(32.0))
        o = np.zeros((4, 128, 32), np.float32)
        r = np.arange(128)
        sl, t = r // kT, r % kT
        ks0, vs0 = kXsBytes // 4, kXsBytes // 4 + 128 * 128
        for g in range(4):
            m = np.full(128, -np.inf, np.float32)
            l = np.zeros(128, np.float32)
            acc = np.zeros((128, 32), np.float32)
            jend = (t | 31) + 1
            for j0 in range(0, 64, 8):
                live = j0 < jend
                sc = np.full((128, 8), -np.inf, np.float32)
                for jj in range(8):
                    j = j0 + jj
                    row = sl * kT + j
                    s = np.zeros(128, np.float32)
                    for i in range(8):
                        base = ks0 + row * kD + 32 * g + 4 * (i ^ jj)
                        for e in range(4):
                            s = (q[g, :, 4 * i + e] * self.sm[base + e] + s).astype(np.float32)
                    sc[:, jj] = np.where(j <= t, s * scale, -np.inf)
                bm = sc.max(axis=1)
                mn = np.maximum(m, bm)
                with np.errstate(invalid="ignore"):
                    corr = np.exp((m - mn).astype(np.float64)).astype(np.float32)
                corr = np.where(np.isnan(corr), 0, corr)
                newl = l * corr
                newacc = acc * corr[:, None]
                for jj in range(8):
                    j = j0 + jj
                    row = sl * kT + j
                    p = np.exp((sc[:, jj] - mn).astype(np.float64)).astype(np.float32)
                    newl = newl + p
                    for i in range(8):
                        base = vs0 + row * kD + 32 * g + 4 * (i ^ jj)
                        for e in range(4):
                            newacc[:, 4 * i + e] = (p * self.sm[base + e] + newacc[:, 4 * i + e]).astype(np.float32)
                l = np.where(live, newl, l)
                acc = np.where(live[:, None], newacc, acc)
                m = np.where(live, mn, m)
            o[g] = acc * (f32(1.0) / l)[:, None]
        return o

    def run(self):
        a, mode = self.a, self.mode
        pair = self.pair
        s0 = 2 * pair
        toks = a.tokens[s0:s0 + 2]
        r = np.arange(128)
        sl, t = r // kT, r % kT
        if mode == FORWARD:
            idx, neww, delta, layer, row = 0xFFFFFFFF, 0.0, 1.0, -1, -1
        else:
            idx, neww, delta, layer, row = self.cand[:5]
        skip = [0, 0]
        if mode != FORWARD and row >= 0:
            skip = [int(all(toks[q, :kT] != row)) for q in range(2)]
        if skip[0] and skip[1]:
            return np.zeros(2, np.float32) if mode == EVAL else None
        self.midx = -1 if mode == FORWARD else idx
        self.mval = f32(neww)
        dlt = f32(0.0) if mode == FORWARD else f32(delta)
        cstage = -1 if mode == FORWARD else layer
        tg = (kNone, 0, 0) if mode == FORWARD else tc_target(a, idx, layer)
        b0 = -1 if (mode == FORWARD or layer < 0) else layer
        rs = RESTART_BLOCK if mode == FORWARD else restart(a, idx, layer)
        self.unit0 = rs == RESTART_UNIT
        self.b0s = 0 if b0 < 0 else b0 + (1 if self.unit0 else 0)
        self.nb = a.nL - self.b0s
        self.cpb = kFfnChunk0 + kFfnPerPair * (a.F // kHp)
        self.ffn0 = rs == RESTART_FFN
        self.q0 = kFfnChunk0 if self.ffn0 else 0
        self.nbc = self.nb * self.cpb - self.q0
        self.total = self.nbc + kHeadChunks
        self.nload = self.nwait = self.ncommit = 0
        if self.nb == 0:
            self.limit = kHeadChunks
        elif not self.ffn0:
            self.limit = kWoChunk0
        else:
            self.limit = self.cpb - self.q0 + kWoChunk0 if self.nb > 1 else self.total
        self.loaded_regions = []
        self.topup(kStages)
        self.s_acol = np.zeros(128, np.float32)
        # residual
        xout = a.X if mode != EVAL else (self.slot.X if self.slot is not None else None)
        xmout = a.Xmid if mode != EVAL else (self.slot.Xmid if self.slot is not None else None)
        lout = a.ell if mode != EVAL else (self.slot.ell if self.slot is not None else None)
        xs = np.zeros((128, kD), np.float32)
        if b0 < 0:
            tok = toks[sl, t]
            for col in range(kD):
                xs[:, col] = self.prm(a.o_tok + tok * kD + col) + self.prm(a.o_pos + t * kD + col)
            if xout is not None:
                for q in range(2):
                    if not skip[q]:
                        xout[0, s0 + q] = xs[q * kT:(q + 1) * kT]
        elif self.unit0:
            xs[:] = ffn_unit(a, self.cand, s0)
            if xout is not None:
                for q in range(2):
                    xout[b0 + 1, s0 + q] = xs[q * kT:(q + 1) * kT]
        else:
            xs[:] = (a.Xmid if self.ffn0 else a.X)[b0, s0 + sl, t]
        for g in range(4):
            self.sm[self.xr_addr(g)[:, None] + np.arange(32)[None, :]] = xs[:, 32 * g:32 * g + 32]
        gc = 0
        nP = a.F // kHp
        for b in range(self.b0s, a.nL):
            here = b == cstage
            base = a.o_blk0 + b * a.blk_size
            if not (self.ffn0 and b == self.b0s):   # a feed-forward candidate starts at its mid stream
                self.ln_to_a(base + a.r_ln1g, base + a.r_ln1b, tg[2] if (here and kTcQ <= tg[0] <= kTcV) else -1)
                self.issue(gc, kQkvChunks)
                gc += kQkvChunks
                self.group_done(gc - 1)
                q = np.zeros((4, 128, 32), np.float32)
                for g in range(4):
                    for p in range(2):
                        v = self.tm[:, (kColV if p else kColK) + 32 * g:(kColV if p else kColK) + 32 * g + 32].copy()
                        bb = base + (a.r_bv if p else a.r_bk) + 32 * g
                        for i in range(32):
                            v[:, i] = v[:, i] + self.prm(bb + i)
                        if here and tg[0] == (kTcV if p else kTcK):
                            at = tg[1] - 32 * g
                            if 0 <= at < 32:
                                v[:, at] += dlt * self.s_acol
                        dst = kXsBytes // 4 + (0 if not p else 128 * 128) + r * kD + 32 * g
                        for i in range(8):
                            for e in range(4):
                                self.sm[dst + 4 * (i ^ (r & 7)) + e] = v[:, 4 * i + e]
                    qq = self.tm[:, kColQ + 32 * g:kColQ + 32 * g + 32].copy()
                    for i in range(32):
                        qq[:, i] = qq[:, i] + self.prm(base + a.r_bq + 32 * g + i)
                    if here and tg[0] == kTcQ:
                        at = tg[1] - 32 * g
                        if 0 <= at < 32:
                            qq[:, at] += dlt * self.s_acol
                    q[g] = qq
                # K and V overlay the first stages: every load issued so far has been consumed
                assert self.nload == gc == self.nwait, ("loads outstanding over K/V", self.nload, gc)
                # check: no load has overwritten K / V since they were written -- loads issued so far
                kv_lo, kv_hi = kXsBytes, kXsBytes + 2 * 128 * 128 * 4
                self.kv_guard = len(self.loaded_regions)
                o = self.attention(q)
                for (x, st_b, nbytes) in self.loaded_regions[self.kv_guard:]:
                    assert st_b + nbytes <= kv_lo or st_b >= kv_hi, ("load over K/V", x)
                if here and tg[0] == kTcO:
                    g = tg[2] // 32
                    self.s_acol = o[g, :, tg[2] - 32 * g].copy()
                for g in range(4):
                    self.store_a(o[g], kColA + 32 * g, kXsBytes, 32 * g, g, 32)
                jb = b - self.b0s
                self.limit = (jb + 1) * self.cpb - self.q0 + kWoChunk0 if jb + 1 < self.nb else self.total
                self.topup(gc + kStages)
                self.issue(gc, kFfnChunk0 - kWoChunk0)
                gc += kFfnChunk0 - kWoChunk0
                self.group_done(gc - 1)
                for g in range(4):
                    v = self.tm[:, kColU + 32 * g:kColU + 32 * g + 32].copy()
                    if here and tg[0] == kTcO:
                        at = tg[1] - 32 * g
                        if 0 <= at < 32:
                            v[:, at] += dlt * self.s_acol
                    xa = self.xr_addr(g)
                    for i in range(32):
                        self.sm[xa + i] = self.sm[xa + i] + (v[:, i] + self.prm(base + a.r_bo + 32 * g + i))
                if xmout is not None:                  # the mid stream
                    for q in range(2):
                        if not skip[q]:
                            for g in range(4):
                                xmout[b, s0 + q, :, 32 * g:32 * g + 32] = self.sm[self.xr_addr(g)[q * kT:(q + 1) * kT, None] + np.arange(32)[None, :]]
            self.ln_to_a(base + a.r_ln2g, base + a.r_ln2b, tg[2] if (here and tg[0] == kTcW1) else -1)
            self.issue(gc, 8)
            gc += 8
            for h in range(2 * nP):
                self.group_done(gc - 1)
                for g in range(4):
                    c0 = kColU + (h & 1) * kHc + 16 * g       # the pair's U, chunk h's columns
                    u = self.tm[:, c0:c0 + 16].copy()
                    f0 = h * kHc + 16 * g
                    if here and tg[0] == kTcW1:
                        at = tg[1] - f0
                        if 0 <= at < 16:
                            u[:, at] += dlt * self.s_acol
                    for i in range(16):
                        u[:, i] = act_fn(a.act, (u[:, i] + self.prm(base + a.r_b1 + f0 + i)).astype(np.float64), a.g).astype(np.float32)
                    if here and tg[0] == kTcW2 and f0 <= tg[2] < f0 + 16:
                        self.s_acol_w2 = u[:, tg[2] - f0].copy()
                    self.store_a2(u, kColA2 + 16 * g, kColA2lo + 16 * g)
                if here and tg[0] == kTcW2 and h * kHc <= tg[2] < h * kHc + kHc:
                    self.s_acol = self.s_acol_w2
                n = 12 if (h & 1) and h + 1 < 2 * nP else 4
                self.issue(gc, n)
                gc += n
            self.group_done(gc - 1)
            for g in range(4):
                v = self.tm[:, kColF + 32 * g:kColF + 32 * g + 32].copy()
                if here and tg[0] == kTcW2:
                    at = tg[1] - 32 * g
                    if 0 <= at < 32:
                        v[:, at] += dlt * self.s_acol
                xa = self.xr_addr(g)
                for i in range(32):
                    self.sm[xa + i] = self.sm[xa + i] + (v[:, i] + self.prm(base + a.r_b2 + 32 * g + i))
            if xout is not None:
                for q in range(2):
                    if not skip[q]:
                        for g in range(4):
                            xout[b + 1, s0 + q, :, 32 * g:32 * g + 32] = self.sm[self.xr_addr(g)[q * kT:(q + 1) * kT, None] + np.arange(32)[None, :]]
        # head
        here = cstage == a.nL
        self.ln_to_a(a.o_lnf_g, a.o_lnf_b, tg[2] if (here and tg[0] == kTcHead) else -1)
        self.issue(gc, kHeadChunks)
        gc += kHeadChunks
        self.group_done(gc - 1)
        assert gc == self.total and self.nload == self.total
        z = np.zeros((4, 128, 32), np.float32)
        for g in range(4):
            zz = self.tm[:, kColU + 32 * g:kColU + 32 * g + 32].copy()
            if here and tg[0] == kTcHead:
                at = tg[1] - 32 * g
                if 0 <= at < 32:
                    zz[:, at] += dlt * self.s_acol
            for i in range(32):
                col = 32 * g + i
                zz[:, i] = (zz[:, i] + self.prm(a.o_bh + col)) if col < a.V else -np.inf
            z[g] = zz
        m = z.max(axis=2).max(axis=0)
        se = np.zeros(128, np.float32)
        for g in range(4):
            for i in range(32):
                if 32 * g + i < a.V:
                    se = se + np.exp((z[g, :, i] - m).astype(np.float64)).astype(np.float32)
        y = toks[sl, t + 1]
        zy = np.array([z[yy // 32, rr, yy % 32] for rr, yy in enumerate(y)], np.float32)
        rowv = (np.log(se.astype(np.float64)).astype(np.float32) + m) - zy
        out = np.zeros(2, np.float32)
        for q in range(2):
            lsum = f32(0)
            for tt in range(kT):
                lsum = f32(lsum + rowv[q * kT + tt])
            if mode == EVAL:
                out[q] = 0.0 if skip[q] else lsum - a.ell[s0 + q]
            if lout is not None and not skip[q]:
                lout[s0 + q] = lsum
        return out


