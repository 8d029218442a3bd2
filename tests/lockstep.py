"""Lock-step comparison of the CUDA step against the oracle (test helper).

Every iteration, the GPU runs draft_step / verify_step / accept_commit; the
oracle then recomputes the same iteration from the same committed history (it
follows the GPU's draft tokens and its committed n / final token, so a single
legitimate divergence cannot cascade) and the two are compared:

* draft and target logits: max |z_gpu - z_oracle| <= 0.03 * max |z_oracle| per row;
* every discrete decision (draft token, accepted length n, final token) must be
  identical.  A mismatch is allowed only as a *flag*, of one of two kinds:

  - tolerance flags, the cases the stated tolerance itself exempts:
      acceptance test: |u_i - p_i(x_i)/q_i(x_i)| < 1e-3 (oracle p, q);
      inverse-CDF sample (draft token, resampled or bonus token): u within 1e-3
        of the oracle's CDF boundary between the two candidates, in normalised
        units;
      greedy argmax: the oracle's gap between the two candidates is below
        0.03 * max |z| (the logit tolerance);
  - error-band flags: the oracle's own margin lies inside the band that the
    measured logit error d of that row allows (a probability moves by at most a
    factor exp(+-2 d / T)): argmax candidates within 2 d; a sample's u within
    exp(2 d / T) - 1 of the boundary (residual rows: 2 (rho_p + rho_q) / R); an
    acceptance margin |log u + log q - log p| <= 2 (d_p + d_q) / T.

  Any other mismatch fails.  Tests cap the error-band flags separately (zero on
  the tiny pair) and every test reports its counts through ``RECORDS``, which
  the conftest prints in the terminal summary.
"""
from __future__ import annotations

import dataclasses

import numpy as np

from oracle.philox import step_uniforms
from oracle.speculative import accept, argmax_first, draft_token, softmax_t

LOGIT_TOL = 0.03
U_TOL = 1e-3          # |u - p/q| and CDF-boundary distance that the tolerance exempts

# one summary line per lock-step test, printed by conftest.pytest_terminal_summary
RECORDS: list = []


@dataclasses.dataclass
class LockstepReport:
    steps: int = 0
    decisions: int = 0
    tol_flags: int = 0          # exempted by the stated tolerance
    band_flags: int = 0         # inside the measured-error band only
    max_logit_err_frac: float = 0.0
    tokens_committed: int = 0
    flag_notes: list = dataclasses.field(default_factory=list)

    @property
    def flags(self) -> int:
        return self.tol_flags + self.band_flags

    def record(self, name: str) -> str:
        line = (f"{name}: steps {self.steps} decisions {self.decisions} tokens "
                f"{self.tokens_committed} tolerance-flags {self.tol_flags} band-flags "
                f"{self.band_flags} max-logit-err {self.max_logit_err_frac:.2e}")
        if self.flag_notes:
            line += " notes " + ";".join(str(n) for n in self.flag_notes)
        RECORDS.append(line)
        return line


def _row_err(zg, zo):
    d = float(np.max(np.abs(zg.astype(np.float64) - zo)))
    return d, d / float(np.max(np.abs(zo)))


def _cdf_boundary(w, a, b):
    c = np.cumsum(w)
    return c[min(a, b)] / c[-1]


def _classify(tol_ok: bool, band_ok: bool, report: LockstepReport, note, msg: str):
    """Record a mismatch as a tolerance flag, else an error-band flag, else fail."""
    if tol_ok:
        report.tol_flags += 1
        report.flag_notes.append(("tol",) + note)
        return
    assert band_ok, msg
    report.band_flags += 1
    report.flag_notes.append(("band",) + note)


def _greedy(zo, a, b, d, report, note, msg):
    gap = abs(float(zo[a]) - float(zo[b]))
    _classify(gap < LOGIT_TOL * float(np.max(np.abs(zo))), gap <= 2 * d + 1e-9, report,
              note + (f"gap {gap:.3e}",), msg)


def _sampled(w, u, a, b, band, report, note, msg):
    dist = abs(u - _cdf_boundary(w, a, b))
    _classify(dist < U_TOL, dist <= band + 1e-6, report, note + (f"|u-F| {dist:.2e}",), msg)


def check_step(eng, sd, K, T, seed, step, report: LockstepReport, req: int = 0, batch: int = 1,
               bits=None):
    """Compare one GPU iteration (already enqueued by the caller) with the oracle.

    ``bits``: the device status word if the caller already synchronised (it is
    then not read again)."""
    if bits is None:
        bits = eng.sync()
    assert bits == 0, f"device status 0x{bits:x}"
    xg = [int(t) for t in eng.draft_tokens(batch)[req, :K]]
    zdg = eng.draft_logits(batch, K)[req]
    ztg = eng.target_logits(batch, K)[req]
    state = eng.seq_state()[req]
    L = sd.L
    u_d, u_a, u_f = step_uniforms(seed, req, step, K)
    # ---- draft: oracle follows the GPU's tokens
    zdo_rows = []
    feed = sd.tokens[sd.dc.length:L]
    for j in range(K):
        zo = sd.draft.forward(sd.dc, feed)[-1]
        zdo_rows.append(zo)
        d, frac = _row_err(zdg[j], zo)
        report.max_logit_err_frac = max(report.max_logit_err_frac, frac)
        assert frac <= LOGIT_TOL, f"step {step} draft row {j}: logit error {frac:.4f} of max"
        xo = draft_token(zo, T, u_d[j])
        report.decisions += 1
        if xo != xg[j]:
            msg = f"req {req} step {step} draft token {j}: gpu {xg[j]} oracle {xo} (unflagged)"
            note = ("draft", req, step, j)
            if T == 0.0:
                _greedy(zo, xo, xg[j], d, report, note, msg)
            else:
                _sampled(softmax_t(zo, T), u_d[j], xo, xg[j], np.expm1(2 * d / T), report,
                         note, msg)
        feed = [xg[j]]
    zdo = np.stack(zdo_rows)
    # ---- verify
    zto = sd.verify(xg)
    dt = []
    for i in range(K + 1):
        d, frac = _row_err(ztg[i], zto[i])
        dt.append(d)
        report.max_logit_err_frac = max(report.max_logit_err_frac, frac)
        assert frac <= LOGIT_TOL, f"step {step} target row {i}: logit error {frac:.4f} of max"
    dd = [_row_err(zdg[j], zdo[j])[0] for j in range(K)]
    # ---- acceptance
    ro = accept(zto, zdo, xg, T, u_a, u_f)
    Lg = int(state[0])
    n_g = Lg - L - 1
    toks = eng.committed_tokens(req)
    y_g = int(toks[-1])
    assert 0 <= n_g <= K, f"step {step}: GPU committed {Lg - L} tokens"
    assert list(toks[L:L + n_g]) == xg[:n_g], f"step {step}: committed drafts differ from x"
    report.decisions += 1
    if n_g != ro.n_accepted:
        i = min(n_g, ro.n_accepted)
        msg = f"req {req} step {step}: accepted n gpu {n_g} oracle {ro.n_accepted} (unflagged)"
        note = ("n", req, step, i)
        if T == 0.0:
            zo = zto[i]
            top = argmax_first(zo)
            srt = np.sort(zo)
            gap = min(float(zo[top] - zo[xg[i]]), float(srt[-1] - srt[-2]))
            _classify(gap < LOGIT_TOL * float(np.max(np.abs(zo))), gap <= 2 * dt[i] + 1e-9,
                      report, note + (f"gap {gap:.3e}",), msg)
        else:
            p = softmax_t(zto[i], T)[xg[i]]
            q = softmax_t(zdo[i], T)[xg[i]]
            margin = abs(np.log(u_a[i]) + np.log(q) - np.log(p))
            dist = abs(u_a[i] - p / q)
            _classify(dist < U_TOL, margin <= 2 * (dt[i] + dd[i]) / T + 1e-6, report,
                      note + (f"|u-p/q| {dist:.2e}",), msg)
    else:
        report.decisions += 1
        n = n_g
        if y_g != ro.token:
            msg = f"req {req} step {step}: final token gpu {y_g} oracle {ro.token} (unflagged)"
            note = ("y", req, step, n)
            if T == 0.0:
                _greedy(zto[n], ro.token, y_g, dt[n], report, note, msg)
            else:
                rho_p = np.expm1(2 * dt[n] / T)
                if n < K:
                    rho_q = np.expm1(2 * dd[n] / T)
                    r = np.maximum(softmax_t(zto[n], T) - softmax_t(zdo[n], T), 0.0)
                    R = r.sum()
                    band = 2 * (rho_p + rho_q) / max(R, 1e-12)
                    w = r if R > 0 else softmax_t(zto[n], T)
                else:
                    band = rho_p
                    w = softmax_t(zto[n], T)
                _sampled(w, u_f, ro.token, y_g, band, report, note, msg)
    # ---- follow the GPU's committed result and check the bookkeeping
    sd.commit(xg, n_g, y_g)
    assert int(state[0]) == sd.L
    assert int(state[1]) == sd.tc.length, (state, sd.tc.length)
    assert int(state[2]) == step + 1
    assert int(state[3]) == sd.dc.length, (state, sd.dc.length)
    report.steps += 1
    report.tokens_committed += n_g + 1
    return n_g, y_g
