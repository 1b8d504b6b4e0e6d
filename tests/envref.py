"""Brute-force restatement of the environment for tiny cases (test helper).

Independent of the oracle's incremental bookkeeping: it keeps the full
actuated history of every consumed sample and recomputes every window sum
and observation feature from scratch (Sec. 4.1 trace replay and actuator,
Eq. 1 windows, Eq. 2 violations, Eq. 3 excess, Eq. 6 / G1 rewards).
Only the Philox draw is shared with the oracle, and that is pinned by the
published known-answer vectors.
"""
import numpy as np

ACT_SET_LEVEL, ACT_INCDEC = 0, 1
W_SHORT, W_LONG = 20, 60


def _f32ratio(num, den):
    return np.float32(np.float32(num) / np.float32(den))


class BruteEnv:
    def __init__(self, spec, trace, phase, env_id, philox):
        self.s, self.e, self.philox = spec, env_id, philox
        # trace families (domain randomisation): family-major [f][n_channels][L_f] buffers;
        # one family: the [C][L] trace itself
        if getattr(spec, "n_families", 0) > 1:
            self.fams, to, po = [], 0, 0
            for L, c, B in zip(spec.fam_len, spec.fam_channels, spec.fam_budget_q):
                tr = np.asarray(trace[to:to + spec.n_channels * L], np.float32).reshape(spec.n_channels, L)[:c]
                self.fams.append((tr, phase[po:po + L], B))
                to += spec.n_channels * L
                po += L
        else:
            self.fams = [(trace, phase, spec.budget_q)]
        self.use_family(0)
        self.reset(0, 0, 2)

    def scale(self, level, c):
        s = self.s
        if s.actuator_kind == ACT_INCDEC:
            return np.float32(0.8 + 0.2 * level / s.g_max)
        return np.float32(s.level_scale[level][c])

    def q(self, c, pos, level):
        x = np.float32(self.trace[c, pos])
        sc = self.scale(level, c) if (self.s.scale_phase_mask >> int(self.phase[pos])) & 1 else np.float32(1.0)
        return int(np.rint(np.float32(np.float32(x * sc) * np.float32(64.0))))

    def use_family(self, f):
        self.fam = f
        self.trace, self.phase, self.B = self.fams[f]
        self.C, self.L = self.trace.shape

    def reset(self, t, it, purpose):
        s = self.s
        seed = s.seed
        w = self.philox([self.e, t, it, purpose], [seed & 0xFFFFFFFF, seed >> 32])
        u, v = int(w[0]), int(w[1])
        self.use_family((v * len(self.fams)) >> 32 if len(self.fams) > 1 else 0)
        span = self.L - s.episode_len * self.nmax() - W_LONG + 1
        self.reset_at(W_LONG + ((u * span) >> 32))

    def nsamp(self, level):
        ls = self.s.level_samples
        return ls[level] if ls and ls[level] > 0 else 1

    def nmax(self):
        ls = self.s.level_samples
        return max([1] + [v for v in (ls or [])])

    def reset_at(self, o):
        s = self.s
        self.pos, self.k = o, 0
        self.level = self.prev = s.level_init
        self.b, self.til = s.b_init, 0
        self.hist = {p: [self.q(c, p, s.level_init) for c in range(self.C)] for p in range(o - W_LONG, o)}
        self.offset = o

    def Qc(self, c, i):
        return self.hist[self.pos - 1 - i][c]

    def Q(self, i):
        return sum(self.hist[self.pos - 1 - i])

    def S(self, w, c=None):
        vals = [self.hist[self.pos - 1 - i] for i in range(w)]
        return sum(v[c] for v in vals) if c is not None else sum(sum(v) for v in vals)

    def obs(self):
        s, B, C = self.s, self.B, self.C
        S20, S60, Q0 = self.S(W_SHORT), self.S(W_LONG), self.Q(0)
        ph = np.float32(self.phase[self.pos - 1])
        if s.obs_kind == 0:
            f = [_f32ratio(self.Q(4 - i), B) for i in range(5)]
            f += [_f32ratio(B - Q0, B), ph, _f32ratio(self.level, s.n_levels - 1)]
        elif s.obs_kind == 1:
            f = [_f32ratio(self.Q(7 - i), B) for i in range(8)]
            f += [_f32ratio(S60, 60 * B), _f32ratio(60 * B - S60, 60 * B), ph,
                  _f32ratio(self.level - s.g_min, s.g_max - s.g_min),
                  _f32ratio(self.b - s.b_min, s.b_max - s.b_min), _f32ratio(S20, 20 * B),
                  _f32ratio(Q0 - self.Q(10), B), np.float32(0)]
        else:
            # d / 20 s: time since the last level change, or with a cadence table
            # the duration of the batch just completed
            d = _f32ratio(self.nsamp(self.level), 40) if self.s.level_samples else _f32ratio(self.til, 40)
            f = [_f32ratio(Q0, B), _f32ratio(S20, 20 * B), _f32ratio(S60, 60 * B),
                 _f32ratio(60 * B - S60, 60 * B), _f32ratio(Q0 - self.Q(10), B),
                 _f32ratio(self.level + 1, s.n_levels), _f32ratio(self.prev + 1, s.n_levels),
                 min(d, np.float32(1.0))]
            last = 4 if s.obs_kind == 2 else 12
            per = []
            for c in range(4):
                per += [(_f32ratio(C * self.Qc(c, last - 1 - i), B) if c < C else np.float32(0))
                        for i in range(last)]
            f += per
            if s.obs_kind == 2:
                f += [_f32ratio(C * self.S(60, c), 60 * B) if c < C else np.float32(0) for c in range(4)]
                f += [np.float32(0)] * 4
            else:
                f += [_f32ratio(C * self.S(20, c), 20 * B) if c < C else np.float32(0) for c in range(4)]
                f += [_f32ratio(C * self.S(60, c), 60 * B) if c < C else np.float32(0) for c in range(4)]
        return np.asarray(f, np.float32)

    def rate(self, level, b):
        s = self.s
        if s.actuator_kind == ACT_INCDEC:
            return s.level_tokens[level] * b / s.b_init
        return s.level_tokens[level]

    def rate_max(self):
        s = self.s
        if s.actuator_kind == ACT_INCDEC:
            return max(self.rate(l, s.b_max) for l in range(s.g_min, s.g_max + 1))
        return max(self.rate(l, s.b_init) for l in range(s.n_levels))

    def step(self, a, lam, t, it):
        s, B = self.s, self.B
        new = self.level
        if s.actuator_kind == ACT_INCDEC:
            if a == 1:
                new = max(new - 1, s.g_min)
            elif a == 2:
                new = min(new + 1, s.g_max)
            elif a == 3:
                self.b = max(self.b - 1, s.b_min)
            elif a == 4:
                self.b = min(self.b + 1, s.b_max)
        else:
            new = a
        self.til = 0 if new != self.level else self.til + 1
        self.prev, self.level = self.level, new
        # one step consumes nsamp(level) samples (one without a cadence table)
        v1 = v60 = qsum = 0
        tokens = excess = peak_w = fixed = 0.0
        for _ in range(self.nsamp(new)):
            p = self.pos
            self.hist[p] = [self.q(c, p, new) for c in range(self.C)]
            self.pos += 1
            Q = self.Q(0)
            S60 = self.S(W_LONG)
            a1, a60 = int(Q > B), int(S60 > 60 * B)
            exc_w = (S60 - 60 * B) / 3840.0 if a60 else 0.0
            tok = self.rate(new, self.b) if self.phase[p] == 0 else 0.0
            v1 += a1
            v60 += a60
            qsum += Q
            tokens += tok
            excess += exc_w * 0.5
            peak_w = max(peak_w, exc_w)
            viol = a1 if s.reward_window == 1 else a60
            fixed += (s.r_viol if viol else s.r_ok) + s.bonus_coef * self.rate(new, self.b) / self.rate_max()
        self.k += 1
        if s.reward_kind == 1:
            r = tokens / 1000.0 - lam * excess - 2.0 * lam * peak_w
        else:
            r = fixed
        done = self.k == s.episode_len
        out = dict(r=r, done=int(done), v1=v1, v60=v60, q=qsum, tokens=tokens, excess=excess,
                   samples=self.nsamp(new))
        if done:
            self.reset(t, it, 1)
        return out
