"""One FastRL step's data-parallel core on one GPU, through the C ABI (orchestration only).

    grpo_advantage  ->  grpo_prune  ->  grpo_compact  ->  [host: kept counts, ARS]  ->
    grpo_loss_fwd_bwd over the kept tokens only
    (or, given hidden states and the output layer's weight instead of logits,
    grpo_lmhead_loss_fwd_bwd: logits on the tensor cores, dhidden and dweight out)

This mirrors Algorithm 1's order within a step: advantages (Eq. 5), MDAP pruning (Phase 2),
the ARS update from the kept counts (Phase 1b), then the policy loss over the selected
trajectories.  Every computation is a library kernel; this class only owns the device buffers,
passes pointers and performs the step's single device-to-host read (the kept counts, which the
host needs for ARS and to size the loss launch).
"""
from __future__ import annotations

import dataclasses

import numpy as np

from . import binding as B


@dataclasses.dataclass
class StepParams:
    G: int
    V: int
    ngram_n: int = 1
    tau: float = 0.8
    keep_cap: int | None = None
    dp_divisor: int = 1
    eps_low: float = 0.2
    eps_high: float = 0.2
    beta: float = 0.04
    agg_mode: int = 0
    dlogits_dtype: str = "bf16"
    std_mode: int = 0
    chunk_rows: int = 0  # >0: the loss runs over the kept rows in chunks sharing one dlogits buffer
    class_eps: float = 0.0  # >0: continuous-reward grouping of advantages (the paper uses 1e-4)
    # "token": Eq. 1's token-level ratio (GRPO, DAPO); "sequence": GSPO's length-normalised
    # sequence ratio, clipped per sequence, with the sequence mean (agg_mode is then unused)
    ratio_level: str = "token"
    # output-layer mode (hidden states and weight given): dhidden dtype and rows of dlogits held
    # at a time (0: the library's default)
    dhidden_dtype: str = "bf16"
    lmhead_chunk_rows: int = 0


class GrpoStep:
    """Device buffers and the launch sequence of one step.

    Inputs (device tensors, resident): rewards f32 [P*G], ids i32 [T] (also the sampled tokens y),
    off i64 [P*G+1], logits [T, V] (bf16 or f32, all tokens of all rollouts), old_logp and
    ref_logp f32 [T].  dlogits are produced for the kept tokens only, in compacted order.

    Output-layer mode: pass logits=None with hidden (bf16 [T, D], every token) and weight (bf16
    [V, D]); the loss is then grpo_lmhead_loss_fwd_bwd over the kept tokens, with dhidden (kept
    rows, compacted order) and dweight (f32 [V, D]) as its gradients.  It runs host-synced."""

    def __init__(self, params: StepParams, rewards, ids, off, logits, old_logp, ref_logp,
                 ars_total_steps: int = 1, steps_per_epoch: int = 1, G1: int | None = None,
                 hidden=None, weight=None):
        import torch
        self.torch = torch
        self.p = params
        self.rewards, self.ids, self.off = rewards, ids, off
        self.logits, self.old, self.ref = logits, old_logp, ref_logp
        self.hidden, self.weight = hidden, weight
        if (logits is None) == (hidden is None) or (hidden is None) != (weight is None):
            raise ValueError("give either logits, or hidden states and the output-layer weight")
        dev = rewards.device
        self.dev = dev
        n = rewards.numel()
        self.P = n // params.G
        self.T = ids.numel()
        self.adv = torch.empty(n, dtype=torch.float32, device=dev)
        self.keep = torch.empty(n, dtype=torch.uint8, device=dev)
        self.kpp = torch.empty(max(self.P, 1), dtype=torch.int32, device=dev)
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.kept_idx = torch.empty(max(n, 1), dtype=torch.int32, device=dev)
        self.kept_off = torch.empty(n + 1, dtype=torch.int64, device=dev)
        self.src_token = torch.empty(max(self.T, 1), dtype=torch.int64, device=dev)
        self.token_rollout = torch.empty(max(self.T, 1), dtype=torch.int32, device=dev)
        self.counts = torch.empty(2, dtype=torch.int64, device=dev)
        self.counts_host = torch.empty(2, dtype=torch.int64, pin_memory=True)
        self.kpp_host = torch.empty(max(self.P, 1), dtype=torch.int32, pin_memory=True)
        self.keep_host = torch.empty(max(n, 1), dtype=torch.uint8, pin_memory=True)
        self.kept_off_host = torch.empty(n + 1, dtype=torch.int64, pin_memory=True)
        # numpy views of the pinned buffers: the per-step host reads avoid tensor indexing
        self._stream = torch.cuda.current_stream(dev)
        self._counts_np = self.counts_host.numpy()
        self._kpp_np = self.kpp_host[:max(self.P, 1)].numpy()[:self.P]
        self.loss = torch.empty(1, dtype=torch.float64, device=dev)
        self.logp = torch.empty(max(self.T, 1), dtype=torch.float32, device=dev)
        # per kept row, the weighted Eq. 1 term w_t * l_t whose fixed-order sum is `loss`
        self.row_loss = torch.empty(max(self.T, 1), dtype=torch.float64, device=dev)
        self.out_dtype = torch.bfloat16 if params.dlogits_dtype == "bf16" else torch.float32
        self.dlogits = None
        self.prune_ws = None
        self.ars = B.grpo_ars_init(G1 if G1 is not None else params.G)
        self.ars_total = ars_total_steps
        self.steps_per_epoch = steps_per_epoch
        self.step_index = 0
        self.n_next = params.G
        self.T_kept = 0
        self.K = 0
        if hidden is not None:
            if params.chunk_rows:
                raise ValueError("output-layer mode chunks through lmhead_chunk_rows, not chunk_rows")
            dh_t = torch.bfloat16 if params.dhidden_dtype == "bf16" else torch.float32
            self.dhidden = torch.empty((max(self.T, 1), hidden.shape[1]), dtype=dh_t, device=dev)
            self.dweight = torch.empty(weight.shape, dtype=torch.float32, device=dev)
            self.lm_ws = None
        self.set_workspaces()

    def _ensure_dlogits(self, rows: int):
        if self.dlogits is None or self.dlogits.shape[0] < rows:
            self.dlogits = None
            self.dlogits = self.torch.empty((max(rows, 1), self.p.V), dtype=self.out_dtype,
                                            device=self.dev)

    def select(self):
        """Advantages, pruning and compaction; then the step's one host read (kept counts)."""
        p = self.p
        B.grpo_advantage(self.rewards, p.G, p.std_mode, adv=self.adv)
        B.grpo_prune(self.rewards, self.ids, self.off, p.G, p.V, p.ngram_n, p.tau, p.keep_cap,
                     p.dp_divisor, keep=self.keep, kept_per_prompt=self.kpp, status=self.status,
                     ws=self.prune_ws, adv=self.adv, class_eps=p.class_eps)
        B.grpo_compact(self.keep, self.off, kept_idx=self.kept_idx, kept_off=self.kept_off,
                       src_token=self.src_token, token_rollout=self.token_rollout,
                       counts=self.counts, counts_host=self.counts_host)
        self.kpp_host[:self.P].copy_(self.kpp[:self.P], non_blocking=True)
        self.torch.cuda.current_stream().synchronize()
        return self._read_counts()

    def set_workspaces(self):
        """Allocate persistent workspaces (sizes from the library's queries)."""
        import ctypes
        L = B.lib()
        need = ctypes.c_size_t(0)
        p = self.p
        rc = L.grpo_prune(None, None, float(p.class_eps), None, None, self.P, p.G, self.T, p.V,
                          p.ngram_n, float(p.tau), p.keep_cap or p.G, p.dp_divisor, None, None,
                          None, None, ctypes.byref(need), None)
        B._check(rc)
        self.prune_ws = self.torch.empty(need.value + 256, dtype=self.torch.uint8, device=self.dev)

    def loss_step(self):
        p = self.p
        if self.hidden is not None:
            return self._loss_lmhead()
        if p.ratio_level == "sequence":
            return self._loss_gspo()
        if p.chunk_rows > 0:
            return self._loss_chunked()
        self._ensure_dlogits(self.T_kept)
        return B.grpo_loss_fwd_bwd(
            self.logits, self.ids, self.old, self.ref, self.adv, self.token_rollout,
            V=p.V, row_index=self.src_token, n_rows=self.T_kept, eps_low=p.eps_low,
            eps_high=p.eps_high, beta=p.beta, agg_mode=p.agg_mode,
            denom_tokens=max(self.T_kept, 1), seq_off=self.off, n_seq=max(self.K, 1),
            dlogits=self.dlogits, dlogits_dtype=self.out_dtype, logp_out=self.logp,
            row_loss_out=self.row_loss, loss_out=self.loss, status=self.status)

    def _loss_lmhead(self):
        """The output layer fused with the loss over the kept rows (gathered by src_token): the
        token-level ratio, or with ratio_level "sequence" GSPO's, whose sequences are the kept
        rollouts (kept_off, kept_idx)."""
        p = self.p
        if p.ratio_level == "sequence":
            if getattr(self, "seq_ratio", None) is None:
                self.seq_ratio = self.torch.empty(max(self.keep.numel(), 1),
                                                  dtype=self.torch.float32, device=self.dev)
            out = B.grpo_lmhead_gspo_loss_fwd_bwd(
                self.hidden, self.weight, self.ids, self.old, self.ref, self.adv, self.kept_idx,
                self.kept_off, n_seq_rows=self.K, n_seq=max(self.K, 1), eps_low=p.eps_low,
                eps_high=p.eps_high, beta=p.beta, dhidden=self.dhidden, dweight=self.dweight,
                logp_out=self.logp, seq_ratio_out=self.seq_ratio, loss_out=self.loss,
                status=self.status, chunk_rows=p.lmhead_chunk_rows, row_index=self.src_token,
                n_rows=self.T_kept, ws=self.lm_ws)
            self.lm_ws = out["ws"]
            return out
        out = B.grpo_lmhead_loss_fwd_bwd(
            self.hidden, self.weight, self.ids, self.old, self.ref, self.adv, self.token_rollout,
            row_index=self.src_token, n_rows=self.T_kept, eps_low=p.eps_low, eps_high=p.eps_high,
            beta=p.beta, agg_mode=p.agg_mode, denom_tokens=max(self.T_kept, 1), seq_off=self.off,
            n_seq=max(self.K, 1), dhidden=self.dhidden, dweight=self.dweight, logp_out=self.logp,
            loss_out=self.loss, status=self.status, chunk_rows=p.lmhead_chunk_rows, ws=self.lm_ws)
        self.lm_ws = out["ws"]
        return out

    def _loss_gspo(self):
        """GSPO's sequence-level loss over the kept rollouts: the compaction's kept offsets and
        kept rollout indices are the sequences."""
        p = self.p
        if p.chunk_rows > 0:
            raise ValueError("the sequence-level ratio runs the loss in one call (chunk_rows = 0)")
        self._ensure_dlogits(self.T_kept)
        if getattr(self, "seq_ratio", None) is None:
            self.seq_ratio = self.torch.empty(max(self.keep.numel(), 1), dtype=self.torch.float32,
                                              device=self.dev)
        out = B.grpo_gspo_loss_fwd_bwd(
            self.logits, self.ids, self.old, self.ref, self.adv, self.kept_idx, self.kept_off,
            n_rows=self.T_kept, n_seq_rows=self.K, n_seq=max(self.K, 1), V=p.V,
            row_index=self.src_token, eps_low=p.eps_low, eps_high=p.eps_high, beta=p.beta,
            dlogits=self.dlogits, dlogits_dtype=self.out_dtype, logp_out=self.logp,
            seq_ratio_out=self.seq_ratio, loss_out=self.loss, status=self.status,
            ws=getattr(self, "gspo_ws", None))
        self.gspo_ws = out["ws"]
        return out

    def _loss_chunked(self):
        """Kept rows in chunks of p.chunk_rows; each chunk overwrites the same dlogits buffer
        (a consumer would use it before the next chunk).  Per-row loss terms are kept and summed
        once at the end in the loss's own fixed order, so the total equals a single call's."""
        p = self.p
        torch = self.torch
        self._ensure_dlogits(min(p.chunk_rows, max(self.T_kept, 1)))
        if getattr(self, "chunk_loss", None) is None:
            self.chunk_loss = torch.empty(1, dtype=torch.float64, device=self.dev)
        for c0 in range(0, self.T_kept, p.chunk_rows):
            c1 = min(self.T_kept, c0 + p.chunk_rows)
            B.grpo_loss_fwd_bwd(
                self.logits, self.ids, self.old, self.ref, self.adv, self.token_rollout[c0:c1],
                V=p.V, row_index=self.src_token[c0:c1], n_rows=c1 - c0, eps_low=p.eps_low,
                eps_high=p.eps_high, beta=p.beta, agg_mode=p.agg_mode,
                denom_tokens=max(self.T_kept, 1), seq_off=self.off, n_seq=max(self.K, 1),
                dlogits=self.dlogits, dlogits_dtype=self.out_dtype, logp_out=self.logp[c0:c1],
                row_loss_out=self.row_loss[c0:c1], loss_out=self.chunk_loss, status=self.status)
        B.grpo_sum_f64(self.row_loss, self.T_kept, out=self.loss)
        return dict(loss=self.loss, dlogits=self.dlogits, logp=self.logp)

    # ---- CUDA-graph mode: no host round trip inside the step ----------------------------------

    def _enqueue_select(self):
        p = self.p
        B.grpo_advantage(self.rewards, p.G, p.std_mode, adv=self.adv)
        B.grpo_prune(self.rewards, self.ids, self.off, p.G, p.V, p.ngram_n, p.tau, p.keep_cap,
                     p.dp_divisor, keep=self.keep, kept_per_prompt=self.kpp, status=self.status,
                     ws=self.prune_ws, adv=self.adv, class_eps=p.class_eps)
        B.grpo_compact(self.keep, self.off, kept_idx=self.kept_idx, kept_off=self.kept_off,
                       src_token=self.src_token, token_rollout=self.token_rollout,
                       counts=self.counts)
        self.counts_host.copy_(self.counts, non_blocking=True)
        self.kpp_host[:self.P].copy_(self.kpp[:self.P], non_blocking=True)
        self.keep_host[:self.keep.numel()].copy_(self.keep, non_blocking=True)
        self.kept_off_host.copy_(self.kept_off, non_blocking=True)

    def _enqueue_loss(self):
        p = self.p
        if p.ratio_level == "sequence":
            return self._enqueue_gspo()
        B.grpo_loss_fwd_bwd_dev(
            self.logits, self.ids, self.old, self.ref, self.adv, self.token_rollout, self.counts,
            max_rows=self.T, dlogits=self.dlogits, loss_out=self.loss, ws=None, V=p.V,
            row_index=self.src_token, eps_low=p.eps_low, eps_high=p.eps_high, beta=p.beta,
            agg_mode=p.agg_mode, seq_off=self.off, logp_out=self.logp, row_loss_out=self.row_loss,
            status=self.status)

    def capture(self):
        """Capture the selection (advantage, prune, compact, count copies) and the loss as two
        CUDA graphs.  The loss reads the kept counts on the device (the token-level loss or, with
        ratio_level "sequence", GSPO's), so nothing waits for the host between them; dlogits are
        sized for all T rows."""
        torch = self.torch
        if self.p.chunk_rows > 0:
            raise ValueError("graph mode runs the loss in one call (chunk_rows = 0)")
        if self.hidden is not None:
            raise ValueError("output-layer mode runs host-synced (its launches are sized by T_kept)")
        self._ensure_dlogits(self.T)
        for _ in range(2):  # warm-up outside capture (kernel attributes, occupancy queries)
            self._enqueue_select()
            self._enqueue_loss()
        torch.cuda.synchronize()
        self.g_select, self.g_loss = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.g_select):
            self._enqueue_select()
        with torch.cuda.graph(self.g_loss):
            self._enqueue_loss()
        torch.cuda.synchronize()
        self._stream = torch.cuda.current_stream()

    def _enqueue_gspo(self):
        """GSPO's loss with the kept counts read on the device (graph mode)."""
        torch = self.torch
        p = self.p
        n = self.keep.numel()
        if getattr(self, "seq_ratio", None) is None:
            self.seq_ratio = torch.empty(max(n, 1), dtype=torch.float32, device=self.dev)
        out = B.grpo_gspo_loss_fwd_bwd_dev(
            self.logits, self.ids, self.old, self.ref, self.adv, self.kept_idx, self.kept_off,
            self.counts, max_rows=self.T, max_seqs=n, dlogits=self.dlogits, loss_out=self.loss,
            ws=getattr(self, "gspo_dev_ws", None), V=p.V, row_index=self.src_token,
            eps_low=p.eps_low, eps_high=p.eps_high, beta=p.beta, logp_out=self.logp,
            seq_ratio_out=self.seq_ratio, status=self.status)
        self.gspo_dev_ws = out["ws"]  # sized on the warm-up calls, before capture

    def replay_select(self):
        self.g_select.replay()

    def replay_loss(self):
        self.g_loss.replay()

    def finish(self):
        """After a replayed step: wait for it, read the kept counts and update ARS (Phase 1b)."""
        self._stream.synchronize()
        return self._read_counts()

    def _read_counts(self):
        """Kept counts from the host copies; then Algorithm 1, Phase 1(b) then 1(a): the rollout
        count for the next step."""
        self.K = int(self._counts_np[0])
        self.T_kept = int(self._counts_np[1])
        self.step_index += 1
        s = (self.step_index - 1) % self.ars_total + 1
        self.n_next = B.adaptive_rollout_count(self.ars, self._kpp_np, s, self.ars_total,
                                               s % self.steps_per_epoch == 0)
        return self.T_kept

    def run_graph(self):
        self.replay_select()
        self.replay_loss()
        return self.finish()

    def run(self):
        self.select()
        self.loss_step()
        return self.loss

    # ---- inputs in pinned host memory ---------------------------------------------------------

    SMALL_INPUTS = ("rewards", "ids", "off", "old", "ref")

    def run_from_host(self, host: dict, loss_host=None, overlap_groups: int = 4):
        """One step whose inputs start in host memory (pinned, for asynchronous copies): `host`
        holds tensors 'rewards', 'ids', 'off', 'old', 'ref' and 'logits' (or, in output-layer
        mode, 'hidden') shaped like the device inputs.  The selection inputs and the per-token log-probs are copied whole; after the
        selection, only the kept rollouts' logit rows are copied (grpo_upload_kept), since the
        pruned rollouts take no further part in the step (Sec. 3.2).

        With overlap_groups > 1 (token-level loss in one call), the kept rollouts are uploaded in
        that many groups on a copy stream, and the loss runs over each group's rows as soon as
        they have landed; the per-row terms are summed once at the end in the loss's fixed order,
        so the result equals a single call's bit for bit.  Otherwise the upload completes first
        and the loss runs as in `loss_step` (the captured graph when `capture()` has run).
        The loss is copied into `loss_host` (f64 [1]) if given.  Returns (h2d_bytes, d2h_bytes)
        moved by this step."""
        torch = self.torch
        p = self.p
        dev_of = dict(rewards=self.rewards, ids=self.ids, off=self.off, old=self.old, ref=self.ref)
        h2d = 0
        for k in self.SMALL_INPUTS:
            dev_of[k].copy_(host[k], non_blocking=True)
            h2d += host[k].numel() * host[k].element_size()
        graphed = getattr(self, "g_select", None) is not None
        if graphed:
            self.replay_select()
        else:
            self._enqueue_select()
        self._stream.synchronize()
        self._read_counts()
        n = self.keep.numel()
        lmhead = self.hidden is not None
        overlap = (overlap_groups > 1 and p.chunk_rows == 0 and p.ratio_level == "token"
                   and not lmhead)
        if overlap and self.T_kept > 0:
            h2d += self._upload_and_loss_overlapped(host, overlap_groups)
        else:
            key, dst = ("hidden", self.hidden) if lmhead else ("logits", self.logits)
            up, _ = B.grpo_upload_kept(host[key], dst, self.keep_host[:n], host["off"])
            h2d += up
            if graphed and p.chunk_rows == 0:
                self.replay_loss()
            else:
                self.loss_step()
        d2h = 2 * 8 + 4 * self.P + n + 8 * (n + 1)  # counts, kept per prompt, keep, kept_off
        if loss_host is not None:
            loss_host.copy_(self.loss, non_blocking=True)
            d2h += 8
        self._stream.synchronize()
        return h2d, d2h

    def _upload_and_loss_overlapped(self, host, groups: int) -> int:
        """Upload the kept rollouts' logit rows in `groups` groups of about equal rows on a copy
        stream; the loss over each group's compacted rows waits only for that group."""
        torch = self.torch
        p = self.p
        n = self.keep.numel()
        keep = self.keep_host.numpy()[:n].astype(bool)
        kept = np.flatnonzero(keep)
        # compacted row offset of each kept rollout: grpo_compact's kept_off, read back with the
        # keep flags; then group boundaries by rows
        rows_before = self.kept_off_host.numpy()[:kept.size + 1]
        T = self.T_kept
        bounds = [0]
        for g in range(1, groups):
            k = int(np.searchsorted(rows_before, T * g / groups, side="left"))
            if k > bounds[-1] and k < kept.size:
                bounds.append(k)
        bounds.append(kept.size)
        if getattr(self, "_copy_stream", None) is None:
            self._copy_stream = torch.cuda.Stream(self.dev)
        self._ensure_dlogits(self.T_kept)
        cs = self._copy_stream
        cs.wait_stream(self._stream)  # the previous step's loss is done with the logits buffer
        up = 0
        for g in range(len(bounds) - 1):
            ka, kb = bounds[g], bounds[g + 1]
            ra, rb = int(kept[ka]), int(kept[kb - 1]) + 1  # rollouts covering the group
            with torch.cuda.stream(cs):
                sub_keep = self.keep_host[ra:rb]
                nb, _ = B.grpo_upload_kept(host["logits"], self.logits, sub_keep,
                                           host["off"][ra:rb + 1])
                up += nb
                ev = torch.cuda.Event()
                ev.record(cs)
            self._stream.wait_event(ev)
            c0, c1 = int(rows_before[ka]), int(rows_before[kb])
            if c1 > c0:
                B.grpo_loss_fwd_bwd(
                    self.logits, self.ids, self.old, self.ref, self.adv, self.token_rollout[c0:c1],
                    V=p.V, row_index=self.src_token[c0:c1], n_rows=c1 - c0, eps_low=p.eps_low,
                    eps_high=p.eps_high, beta=p.beta, agg_mode=p.agg_mode,
                    denom_tokens=max(self.T_kept, 1), seq_off=self.off, n_seq=max(self.K, 1),
                    dlogits=self.dlogits[c0:c1], dlogits_dtype=self.out_dtype,
                    logp_out=self.logp[c0:c1], row_loss_out=self.row_loss[c0:c1],
                    loss_out=self.loss, status=self.status)
        B.grpo_sum_f64(self.row_loss, self.T_kept, out=self.loss)
        return up

    def kept_rows(self):
        """(src_token, token_rollout) of the kept rows as host arrays."""
        return (self.src_token[:self.T_kept].cpu().numpy(),
                self.token_rollout[:self.T_kept].cpu().numpy())


def as_device(batch: dict, device):
    """Host arrays of a workloads batch -> device tensors (rewards, ids, off)."""
    import torch
    return (torch.from_numpy(batch["rewards"]).to(device),
            torch.from_numpy(batch["ids"]).to(device),
            torch.from_numpy(batch["off"]).to(device))
