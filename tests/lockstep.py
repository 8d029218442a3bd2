"""Lock-step comparison of the CUDA step against the oracle (test helper).

Every iteration, the GPU runs draft_step / verify_step / accept_commit; the
oracle then recomputes the same iteration from the same committed history (it
follows the GPU's draft tokens and its committed n / final token, so a single
legitimate divergence cannot cascade) and the two are compared:

* draft and target logits: max |z_gpu - z_oracle| <= 0.03 * max |z_oracle| per row;
* every discrete decision (draft token, accepted length n, final token) must be
  identical, except where the oracle's own margin for that decision lies
  inside the band that the measured logit error allows.  For a logit error of
  at most d on a row, a probability can move by a factor exp(+-2 d / T), so:
    - greedy argmax: flagged iff the two candidates' oracle logits are within 2 d;
    - inverse-CDF sample: flagged iff u is within rho = exp(2 d / T) - 1 of the
      oracle CDF boundary between the two candidates (residual rows: the band
      of the normalised residual, 2 (rho_p + rho_q) / R);
    - acceptance test u * q <= p: flagged iff |log u + log q - log p| (oracle)
      <= 2 (d_p + d_q) / T, or |u - p/q| < 1e-3.
  Flags are counted and reported; an unflagged mismatch fails.
"""
from __future__ import annotations

import dataclasses

import numpy as np

from oracle.philox import step_uniforms
from oracle.speculative import accept, argmax_first, draft_token, softmax_t

LOGIT_TOL = 0.03


@dataclasses.dataclass
class LockstepReport:
    steps: int = 0
    decisions: int = 0
    flags: int = 0
    max_logit_err_frac: float = 0.0
    tokens_committed: int = 0
    flag_notes: list = dataclasses.field(default_factory=list)


def _row_err(zg, zo):
    d = float(np.max(np.abs(zg.astype(np.float64) - zo)))
    return d, d / float(np.max(np.abs(zo)))


def _cdf_boundary(w, a, b):
    c = np.cumsum(w)
    return c[min(a, b)] / c[-1]


def _greedy_flag(zo, a, b, d):
    return abs(zo[a] - zo[b]) <= 2 * d + 1e-9


def check_step(eng, sd, K, T, seed, step, report: LockstepReport, req: int = 0, batch: int = 1):
    """Run one GPU iteration (already enqueued by the caller) and compare it."""
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
            if T == 0.0:
                ok = _greedy_flag(zo, xo, xg[j], d)
            else:
                q = softmax_t(zo, T)
                rho = np.expm1(2 * d / T)
                ok = abs(u_d[j] - _cdf_boundary(q, xo, xg[j])) <= rho + 1e-6
            assert ok, f"step {step} draft token {j}: gpu {xg[j]} oracle {xo} (unflagged)"
            report.flags += 1
            report.flag_notes.append(("draft", step, j))
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
        if T == 0.0:
            zo = zto[i]
            top = argmax_first(zo)
            srt = np.sort(zo)
            ok = (zo[top] - zo[xg[i]] <= 2 * dt[i] + 1e-9) or (srt[-1] - srt[-2] <= 2 * dt[i] + 1e-9)
        else:
            p = softmax_t(zto[i], T)[xg[i]]
            q = softmax_t(zdo[i], T)[xg[i]]
            margin = abs(np.log(u_a[i]) + np.log(q) - np.log(p))
            ok = margin <= 2 * (dt[i] + dd[i]) / T + 1e-6 or abs(u_a[i] - p / q) < 1e-3
        assert ok, f"step {step}: accepted n gpu {n_g} oracle {ro.n_accepted} (unflagged)"
        report.flags += 1
        report.flag_notes.append(("n", step, i))
    else:
        report.decisions += 1
        n = n_g
        if y_g != ro.token:
            if T == 0.0:
                ok = _greedy_flag(zto[n], ro.token, y_g, dt[n])
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
                ok = abs(u_f - _cdf_boundary(w, ro.token, y_g)) <= band + 1e-6
            assert ok, f"step {step}: final token gpu {y_g} oracle {ro.token} (unflagged)"
            report.flags += 1
            report.flag_notes.append(("y", step, n))
    # ---- follow the GPU's committed result and check the bookkeeping
    sd.commit(xg, n_g, y_g)
    assert int(state[0]) == sd.L
    assert int(state[1]) == sd.tc.length, (state, sd.tc.length)
    assert int(state[2]) == step + 1
    assert int(state[3]) == sd.dc.length, (state, sd.dc.length)
    report.steps += 1
    report.tokens_committed += n_g + 1
    return n_g, y_g
