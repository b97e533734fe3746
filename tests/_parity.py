"""Lockstep parity of the GPU path against the CPU oracle, shared by the full-size GPU tests.

A speculative round runs on the GPU; the oracle runs the same passes on the same rows (the
GPU's pending token and the GPU's drafts), so both sides stay on one token sequence even where
the GPU picks a different argmax inside a near-tie.  Every comparison is recorded, not only
asserted: per workload, pass and round the measured max |GPU logit - oracle logit|, the
disagreement of two valid oracles (fp32 and fp64 accumulation) on the same rows, the bound
applied, and the ids that differ from the oracle's argmax with their logit gap.  The records are
printed in pytest's terminal summary (and written to $PBD_PARITY_JSON when that is set).

The bound: 3e-2 (the stated logit tolerance) or, where two valid oracles already disagree by
more than half of that on the same rows, twice their measured disagreement, never above 0.1.
Ids must equal the oracle's argmax except where the oracle's own top two are within the bound
(a near-tie, counted); accepted lengths and cached lengths are exact.
"""
import numpy as np

import oracle

TOL = 3e-2
RECORDS = []  # dicts, see record()


def bound(drift):
    return min(0.1, max(TOL, 2.0 * drift))


def record(workload, pass_kind, rnd, seq, gpu_logits, ref_logits, ref64_logits, gpu_ids):
    """Compare one pass of one sequence; returns the bound.  Asserts logits within the bound
    and ids equal to the oracle's argmax up to counted near-ties inside it."""
    gpu_logits = np.asarray(gpu_logits, np.float32).reshape(ref_logits.shape)
    dmax = float(np.abs(gpu_logits - ref_logits).max())
    drift = float(np.abs(ref_logits - ref64_logits).max()) if ref64_logits is not None else 0.0
    tol = bound(drift)
    ids = np.asarray(gpu_ids).reshape(-1)
    ties = []
    for j, t in enumerate(ids):
        best = int(np.argmax(ref_logits[j]))
        if int(t) != best:
            ties.append((j, int(t), best, float(ref_logits[j][best] - ref_logits[j][int(t)])))
    RECORDS.append(dict(workload=workload, pass_kind=pass_kind, round=rnd, seq=seq, max_abs_diff=dmax,
                        oracle_drift=drift, bound=tol, rows=int(len(ids)), id_mismatches=len(ties),
                        max_tie_gap=max((t[3] for t in ties), default=0.0)))
    assert dmax <= tol, (workload, pass_kind, rnd, seq, dmax, tol)
    for j, t, best, gap in ties:
        assert gap <= tol, (workload, pass_kind, rnd, seq, "row", j, "gpu", t, "oracle", best, "gap", gap)
    return tol


def record_tokens(workload, seq, n_tokens, ties):
    """A teacher-forced comparison of a whole generation: ties = [(position, gap), ...]."""
    RECORDS.append(dict(workload=workload, pass_kind="greedy-generation", round=-1, seq=seq, max_abs_diff=None,
                        oracle_drift=None, bound=None, rows=int(n_tokens), id_mismatches=len(ties),
                        max_tie_gap=max((g for _, g in ties), default=0.0)))


class Seq:
    """One sequence on the oracle (fp32 accumulation; and fp64 accumulation when m64 is given, for
    the drift) after its prefill."""

    def __init__(self, m, m64, prompt, D, rounds):
        self.m, self.m64, self.D, self.L = m, m64, D, len(prompt)
        cap = len(prompt) + (rounds + 1) * (D + 1)
        self.cache, self.p, self.lg0 = m.prefill(prompt, cap, want_logits=True)
        self.cache64 = m64.prefill(prompt, cap)[0] if m64 is not None else None

    def _fwd(self, rows, adapter, mask, n_read):
        _, lg, _ = self.m.forward(self.cache, self.L, rows, adapter, mask, 0, n_read, want_logits=True)
        lg64 = None
        if self.cache64 is not None:
            _, lg64, _ = self.m64.forward(self.cache64, self.L, rows, adapter, mask, 0, n_read, want_logits=True)
        return lg, lg64

    def draft(self):
        return self._fwd([self.p] + [-1] * self.D, True, oracle.MASK_BLOCK_DRAFT, self.D)

    def verify(self, drafts):
        return self._fwd([self.p] + list(drafts), False, oracle.MASK_CAUSAL, self.D + 1)

    def advance(self, n, verify_ids):
        self.L += n + 1
        self.p = int(verify_ids[n])


def start(eng, prompts, seqs, max_new, workload):
    """Prefill on the GPU; the first token must be the oracle's argmax up to a near-tie (counted;
    both sides go on with the GPU's token)."""
    first = eng.pbd_prefill(prompts, max_new=max_new)
    for b, sq in seqs.items():
        g = int(first[b])
        best = int(np.argmax(sq.lg0))
        ties = [] if g == best else [(0, float(sq.lg0[best] - sq.lg0[g]))]
        record_tokens(workload + ":first-token", b, 1, ties)
        for _, gap in ties:
            assert gap <= 0.1, (workload, b, g, best, gap)
        sq.p = g


def rounds(eng, seqs, n_rounds, workload):
    """n_rounds speculative rounds of the engine's batch in lockstep with the oracle."""
    for rnd in range(n_rounds):
        d_ids, d_lg = eng.pbd_draft_block(want_logits=True)
        for b, sq in seqs.items():
            od, od64 = sq.draft()
            record(workload, "draft", rnd, b, d_lg[b].cpu().numpy(), od, od64, d_ids[b].cpu().numpy())
        v_ids, v_lg = eng.pbd_verify_block(want_logits=True)
        n_gpu = eng.pbd_accept_commit()
        Lg, pend, _ = eng.pbd_get_state()
        for b, sq in seqs.items():
            drafts = [int(t) for t in d_ids[b].cpu()]
            ov, ov64 = sq.verify(drafts)
            verify = [int(t) for t in v_ids[b].cpu()]
            record(workload, "verify", rnd, b, v_lg[b].cpu().numpy(), ov, ov64, verify)
            n = oracle.accept_length(drafts, verify)
            assert int(n_gpu[b]) == n, (workload, rnd, b)
            sq.advance(n, verify)
            assert int(Lg[b]) == sq.L and int(pend[b]) == sq.p, (workload, rnd, b)


def summary_lines():
    if not RECORDS:
        return []
    out = ["GPU vs oracle logits (max |diff|; oracle fp32-vs-fp64 drift; bound; ids differing from "
           "the oracle argmax, all near-ties inside the bound):"]
    by = {}
    for r in RECORDS:
        by.setdefault((r["workload"], r["pass_kind"]), []).append(r)
    for (w, k), rs in sorted(by.items()):
        if rs[0]["max_abs_diff"] is None:
            out.append("  %-44s %-18s tokens %5d  near-ties %d (max gap %.3g)" % (
                w, k, sum(r["rows"] for r in rs), sum(r["id_mismatches"] for r in rs),
                max(r["max_tie_gap"] for r in rs)))
            continue
        d = [r["max_abs_diff"] for r in rs]
        out.append("  %-44s %-7s passes %3d  max|diff| %.4f (median %.4f, over 3e-2: %d)  drift %.4f  "
                   "bound <= %.3f  near-ties %d (max gap %.3g)" % (
                       w, k, len(rs), max(d), float(np.median(d)), sum(x > TOL for x in d),
                       max(r["oracle_drift"] for r in rs), max(r["bound"] for r in rs),
                       sum(r["id_mismatches"] for r in rs), max(r["max_tie_gap"] for r in rs)))
    return out
