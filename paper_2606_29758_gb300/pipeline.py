"""The PS-PPO LM-head update pass through the C ABI, with buffers held in torch.

UpdatePass owns the device buffers of one batch shape (allocated once with torch,
sized for the worst case N = sum L) and runs the four library calls in order on the
current stream: cutoffs -> packed prefixes -> fused forward -> fused backward. With a
logit store (PassShape.store_rows), a step whose N fits keeps the forward's logits for
the backward instead of recomputing them.
The only host synchronisation is reading N after packing.
CutoffDesign does the same for the cutoff design upstream of the update (score
proxy and top-k next tokens, u_t, and the design into sampler masses).
InputStager copies the next batch's inputs from pinned host memory on its own
stream while the current pass runs.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import torch

from . import _binding as B


@dataclass
class PassShape:
    P: int
    K: int
    T_max: int
    d: int
    V: int
    capacity: int                 # max packed rows (sum of lengths)
    dtype: torch.dtype = torch.bfloat16
    bwd_chunk_rows: int = 32768   # rows of dZ held at once in the backward workspace
    store_rows: int = 0           # rows of the logit store (bf16): a step with N <= store_rows keeps
                                  # its logits from the forward instead of recomputing them (0: never)


class UpdatePass:
    def __init__(self, shape: PassShape, device: str = "cuda", eps: float = 0.2, loss_scale: Optional[float] = None,
                 mode: int = B.PS_MODE_TRUNC, adv_mode: int = B.PS_ADV_GROUP_NORM):
        s = shape
        self.s, self.device, self.eps, self.mode, self.adv_mode = s, device, eps, mode, adv_mode
        self.loss_scale = loss_scale if loss_scale is not None else 1.0 / (s.P * s.K)
        self.dcode = B.dtype_code(torch.empty(0, dtype=s.dtype))
        Bn, cap = s.P * s.K, s.capacity
        i32 = dict(dtype=torch.int32, device=device)
        f32 = dict(dtype=torch.float32, device=device)
        self.H = torch.empty(Bn, **i32)
        self.n = torch.empty(Bn, **i32)
        self.w_tab = torch.empty(s.P, s.T_max, **f32)
        self.cu_seqlens = torch.empty(Bn + 1, **i32)
        self.src_row = torch.empty(cap, **i32)
        self.row_traj = torch.empty(cap, **i32)
        self.row_pos = torch.empty(cap, **i32)
        self.tok = torch.empty(cap, **i32)
        self.oldlogp = torch.empty(cap, **f32)
        self.w = torch.empty(cap, **f32)
        self.adv = torch.empty(cap, **f32)
        self.hid = torch.empty(cap, s.d, dtype=s.dtype, device=device)
        self.lse = torch.empty(cap, **f32)
        self.logp = torch.empty(cap, **f32)
        self.ratio = torch.empty(cap, **f32)
        self.coef = torch.empty(cap, **f32)
        self.row_loss = torch.empty(cap, **f32)
        self.loss = torch.zeros(1, dtype=torch.float64, device=device)
        self.dH = torch.empty(cap, s.d, **f32)
        self.dW = torch.empty(s.V, s.d, **f32)
        u8 = dict(dtype=torch.uint8, device=device)   # zeroed: a status word never written reads clear
        self.ws_samp = torch.zeros(B.ps_sample_cutoffs_workspace_size(s.P, s.K, s.T_max), **u8)
        self.ws_pack = torch.zeros(B.ps_pack_prefixes_workspace_size(s.P, s.K), **u8)
        self.ws_fwd = torch.zeros(B.ps_lmhead_ppo_fwd_workspace_size(cap, s.d, s.V, self.dcode), **u8)
        self.ws_bwd = torch.zeros(B.ps_lmhead_ppo_bwd_workspace_size(cap, s.d, s.V, self.dcode,
                                                                     min(s.bwd_chunk_rows, cap)), **u8)
        self.store = None
        if s.store_rows > 0:
            if s.dtype != torch.bfloat16:
                raise ValueError("the logit store needs a bf16 head")
            self.store = torch.empty(B.ps_lmhead_logit_store_size(min(s.store_rows, cap), s.V), **u8)
        self.N = 0
        self.use_store = True         # False: recompute even where the store would hold the step
        self.stored = False           # the last forward filled the store (its backward reads it)

    def sample(self, q, L, seed, step, traj_base=0):
        s = self.s
        B.ps_sample_cutoffs(s.P, s.K, s.T_max, q, L, seed, step, traj_base, self.mode, self.H, self.n,
                            self.w_tab, self.ws_samp)

    def pack(self, L, R, tok_full, oldlogp_full, hid_full) -> int:
        s = self.s
        self.N = B.ps_pack_prefixes(s.P, s.K, s.T_max, s.d, self.dcode, L, self.n, R, self.adv_mode, self.w_tab,
                                    tok_full, oldlogp_full, hid_full, s.capacity, self.cu_seqlens, self.src_row,
                                    self.row_traj, self.row_pos, self.tok, self.oldlogp, self.w, self.adv, self.hid,
                                    self.ws_pack)
        return self.N

    def forward(self, W):
        s = self.s
        self.stored = self.use_store and self.store is not None and self.N <= s.store_rows
        if self.stored:
            B.ps_lmhead_ppo_fwd_store(self.N, s.d, s.V, self.dcode, self.hid, W, self.tok, self.oldlogp, self.adv,
                                      self.w, self.eps, self.loss_scale, self.loss, self.lse, self.logp, self.ratio,
                                      self.coef, self.row_loss, self.store, self.ws_fwd)
        else:
            B.ps_lmhead_ppo_fwd(self.N, s.d, s.V, self.dcode, self.hid, W, self.tok, self.oldlogp, self.adv, self.w,
                                self.eps, self.loss_scale, self.loss, self.lse, self.logp, self.ratio, self.coef,
                                self.row_loss, self.ws_fwd)

    def backward(self, W, dw_accumulate: bool = False):
        s = self.s
        flags = B.PS_DW_ACCUMULATE if dw_accumulate else B.PS_DW_OVERWRITE
        if self.stored:
            # the store turns into dZ in place: one backward per forward
            self.stored = False
            B.ps_lmhead_ppo_bwd_from_store(self.N, s.d, s.V, self.dcode, self.hid, W, self.tok, self.lse, self.logp,
                                           self.coef, self.store, self.dH, self.dW, flags, self.ws_bwd)
        else:
            B.ps_lmhead_ppo_bwd(self.N, s.d, s.V, self.dcode, self.hid, W, self.tok, self.lse, self.coef, self.dH,
                                self.dW, flags, self.ws_bwd)

    def run(self, q, L, R, tok_full, oldlogp_full, hid_full, W, seed, step, traj_base=0, grads=True) -> int:
        self.sample(q, L, seed, step, traj_base)
        self.pack(L, R, tok_full, oldlogp_full, hid_full)
        self.forward(W)
        if grads:
            self.backward(W)
        return self.N

    def check_status(self):
        """Raise PsppoError if any workspace reports a device-side error."""
        for name, ws in (("sample", self.ws_samp), ("pack", self.ws_pack), ("fwd", self.ws_fwd),
                         ("bwd", self.ws_bwd)):
            rc, bits = B.ps_workspace_status(ws)
            if rc != B.PS_OK:
                raise B.PsppoError(rc, f"{name} (device bits {bits:#x})")


@dataclass(frozen=True)
class PromptShard:
    """One rank's share of a rollout batch in a data-parallel update: the prompts [p0, p1), their
    completions [k0, k1) and their rows [o0, o1) of the unpacked batch (completion after
    completion). Advantages are per group, so a shard holds whole groups; its cutoffs are drawn
    with traj_base = k0, the global index of its first completion, so every completion gets the
    draw it gets in the whole batch; its loss uses the global scale 1/(P K); and dW sums over the
    shards (PS_DW_ACCUMULATE after the first shard on one device, an all-reduce across devices)."""
    p0: int
    p1: int
    k0: int
    k1: int
    o0: int
    o1: int

    @property
    def prompts(self) -> int:
        return self.p1 - self.p0


def prompt_shard(P: int, K: int, L, world: int, rank: int) -> PromptShard:
    """Contiguous prompt ranges of sizes as equal as possible; L: the batch's completion lengths
    (host array, B = P K entries)."""
    if not (0 <= rank < world) or world > P:
        raise ValueError("need 0 <= rank < world <= P")
    p0, p1 = rank * P // world, (rank + 1) * P // world
    k0, k1 = p0 * K, p1 * K
    lens = [int(x) for x in L]
    o0 = sum(lens[:k0])
    return PromptShard(p0, p1, k0, k1, o0, o0 + sum(lens[k0:k1]))


class DataParallelUpdate:
    """One rank's step of a data-parallel update: its prompt shard through an update pass, then the
    sum of dW and of the loss over the ranks of a process group.

    The pass must have been built with the global loss scale 1/(P K) of the whole batch, and
    `traj_base` is the global index of the shard's first completion (PromptShard.k0, or rank * B
    when every rank holds B completions), so that each completion draws the cutoff it draws in the
    whole batch. The summed dW and loss are then the whole batch's (Eq. full_update_G and Eq.
    truncated_update_Ghat: 1/K per prompt, the mean over all prompts). The exchange is one
    all-reduce of dW (V x d f32) and one of the loss, enqueued on the current stream after the
    backward; with one rank, or no initialised process group, there is nothing to exchange.
    `update_pass` needs sample / pack / forward / backward and the tensors dW and loss (UpdatePass).
    """

    def __init__(self, update_pass, traj_base: int, group=None):
        self.up = update_pass
        self.traj_base = int(traj_base)
        self.group = group

    def world(self) -> int:
        import torch.distributed as dist
        if not (dist.is_available() and dist.is_initialized()):
            return 1
        return dist.get_world_size(self.group)

    def exchange(self):
        """Sum dW and the loss over the ranks."""
        if self.world() > 1:
            import torch.distributed as dist
            dist.all_reduce(self.up.dW, group=self.group)
            dist.all_reduce(self.up.loss, group=self.group)

    def run(self, q, L, R, tok_full, oldlogp_full, hid_full, W, seed, step) -> int:
        """Sample, pack, forward and backward on this rank's shard, then the exchange; returns the
        shard's packed rows."""
        up = self.up
        up.sample(q, L, seed, step, traj_base=self.traj_base)
        n = up.pack(L, R, tok_full, oldlogp_full, hid_full)
        up.forward(W)
        up.backward(W)
        self.exchange()
        return n


def vocab_shards(V: int, S: int):
    """S contiguous vocabulary ranges (v0, Vs) of sizes as equal as possible."""
    if not 1 <= S <= V:
        raise ValueError("need 1 <= S <= V")
    return [(r * V // S, (r + 1) * V // S - r * V // S) for r in range(S)]


class VocabParallelHead:
    """The update pass's head split by vocabulary rows (the vocabulary-parallel calls of psppo.h).

    `shards` lists the ranges (v0, Vs) of all S shards, in order; W_shard r is rows [v0, v0 + Vs)
    of W. Per step: `stats(r, ...)` for every local shard, `gather()` (all_gather of the S shards'
    12 bytes per row over `group`; nothing with one process, which then holds every shard), the
    identical `forward(...)` on every process, `backward(r, ...)` for every local shard (its dW rows and
    its term of dH, added into dH by every local shard after the first: PS_DH_ACCUMULATE), and
    `reduce_dH()` (the all_reduce of dH over the processes; nothing with one process).

    With `store`, each shard's statistics call also keeps the shard's logits in a logit store of its
    own (allocated for the shards this process runs, on their first use) and its backward turns them
    into the shard's dZ instead of recomputing them (bf16 heads)."""

    def __init__(self, shards, capacity: int, d: int, V: int, dtype: torch.dtype = torch.bfloat16,
                 device: str = "cuda", eps: float = 0.2, loss_scale: float = 1.0, bwd_chunk_rows: int = 32768,
                 group=None, store: bool = False):
        if store and dtype != torch.bfloat16:
            raise ValueError("the logit store needs a bf16 head")
        self.shards, self.d, self.V, self.eps, self.loss_scale, self.group = list(shards), d, V, eps, loss_scale, group
        self.device, self.use_store, self.stores = device, store, {}
        self.S = len(self.shards)
        self.dcode = B.dtype_code(torch.empty(0, dtype=dtype))
        f32 = dict(dtype=torch.float32, device=device)
        u8 = dict(dtype=torch.uint8, device=device)
        self.stats_all = torch.empty(self.S, capacity, 2, **f32)
        self.ztok_all = torch.empty(self.S, capacity, **f32)
        vmax = max(Vs for _, Vs in self.shards)
        self.ws_stats = torch.zeros(B.ps_lmhead_logit_stats_workspace_size(capacity, d, vmax, self.dcode), **u8)
        self.ws_fin = torch.zeros(B.ps_lmhead_ppo_fwd_from_stats_workspace_size(capacity), **u8)
        self.capacity = capacity
        self.chunk_rows = min(bwd_chunk_rows, capacity)
        self.ws_bwd = torch.zeros(B.ps_lmhead_ppo_bwd_workspace_size(capacity, d, vmax, self.dcode, self.chunk_rows),
                                  **u8)
        self.ws_store = torch.zeros(B.ps_lmhead_ppo_bwd_from_store_workspace_size(), **u8)
        self.lse, self.logp, self.ratio, self.coef, self.row_loss = (torch.empty(capacity, **f32) for _ in range(5))
        self.loss = torch.zeros(1, dtype=torch.float64, device=device)

    def stats(self, r: int, N: int, hid, W_shard, tok):
        v0, Vs = self.shards[r]
        if self.use_store:
            if r not in self.stores:
                self.stores[r] = torch.empty(B.ps_lmhead_logit_store_size(self.capacity, Vs), dtype=torch.uint8,
                                             device=self.device)
            B.ps_lmhead_logit_stats_store(N, self.d, Vs, v0, self.dcode, hid, W_shard, tok, self.stats_all[r],
                                          self.ztok_all[r], self.stores[r], self.ws_stats)
        else:
            B.ps_lmhead_logit_stats(N, self.d, Vs, v0, self.dcode, hid, W_shard, tok, self.stats_all[r],
                                    self.ztok_all[r], self.ws_stats)

    def gather(self, N: int, rank: int):
        """Every shard's statistics on every process (rank = the index of this process's shard)."""
        import torch.distributed as dist
        if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size(self.group) == 1:
            return
        dist.all_gather([self.stats_all[r, :N] for r in range(self.S)], self.stats_all[rank, :N].clone(),
                        group=self.group)
        dist.all_gather([self.ztok_all[r, :N] for r in range(self.S)], self.ztok_all[rank, :N].clone(),
                        group=self.group)

    def forward(self, N: int, tok, oldlogp, adv, w):
        ld = self.stats_all.shape[1]
        B.ps_lmhead_ppo_fwd_from_stats(N, self.S, ld, self.V, self.stats_all, self.ztok_all, tok, oldlogp, adv, w,
                                       self.eps, self.loss_scale,
                                       self.loss, self.lse, self.logp, self.ratio, self.coef, self.row_loss,
                                       self.ws_fin)

    def backward(self, r: int, N: int, hid, W_shard, tok, dH, dW_shard, add_to_dH: bool = False):
        """Shard r's rows of dW (overwritten) and its term of dH (written, or added to dH)."""
        v0, Vs = self.shards[r]
        flags = B.PS_DH_ACCUMULATE if add_to_dH else 0
        if self.use_store:
            # the store of this shard's last statistics call becomes its dZ: one backward per call
            B.ps_lmhead_ppo_bwd_vocab_shard_from_store(N, self.d, Vs, v0, self.V, self.dcode, hid, W_shard, tok,
                                                       self.lse, self.logp, self.coef, self.stores[r], dH, dW_shard,
                                                       flags, self.ws_store)
            return
        # the workspace of chunk_rows rows at this shard's width: every shard (and the whole head with
        # the same chunk_rows) cuts the rows into the same chunks
        nb = B.ps_lmhead_ppo_bwd_workspace_size(self.capacity, self.d, Vs, self.dcode, self.chunk_rows)
        B.ps_lmhead_ppo_bwd_vocab_shard(N, self.d, Vs, v0, self.V, self.dcode, hid, W_shard, tok, self.lse,
                                        self.coef, dH, dW_shard, flags, self.ws_bwd[:nb])

    def reduce_dH(self, dH):
        import torch.distributed as dist
        if dist.is_available() and dist.is_initialized() and dist.get_world_size(self.group) > 1:
            dist.all_reduce(dH, group=self.group)


class InputStager:
    """Double-buffered host -> device staging of the unpacked batch inputs.

    Holds `slots` device copies of a dict of tensors (the per-batch inputs of UpdatePass.sample and
    UpdatePass.pack) and a copy stream. `stage(host)` enqueues the host -> device copies of one batch
    (pinned host tensors, so the copies are asynchronous) into the next slot and returns the slot;
    `acquire(slot, stream)` makes `stream` wait for that slot's copies and returns its tensors;
    `release(slot, stream)` marks the slot free once the work enqueued on `stream` so far is done, and
    a later `stage` into the slot waits for that. Staging batch i + 1 before running the pass on
    batch i lets the copy engine move the next batch while the tensor cores work on this one.
    """

    def __init__(self, like: dict, device: str = "cuda", slots: int = 2):
        if slots < 1:
            raise ValueError("slots must be >= 1")
        self.bufs = [{k: torch.empty(v.shape, dtype=v.dtype, device=device) for k, v in like.items()}
                     for _ in range(slots)]
        self.copy_stream = torch.cuda.Stream(device=device)
        self.ready = [torch.cuda.Event() for _ in range(slots)]
        self.free = [torch.cuda.Event() for _ in range(slots)]
        self.nbytes = sum(v.numel() * v.element_size() for v in like.values())
        self._next = 0

    def stage(self, host: dict) -> int:
        j = self._next
        self._next = (j + 1) % len(self.bufs)
        dst = self.bufs[j]
        with torch.cuda.stream(self.copy_stream):
            self.copy_stream.wait_event(self.free[j])     # no-op until the slot has been released once
            for k, t in host.items():
                dst[k].copy_(t, non_blocking=True)
            self.ready[j].record(self.copy_stream)
        return j

    def acquire(self, j: int, stream=None) -> dict:
        (stream or torch.cuda.current_stream()).wait_event(self.ready[j])
        return self.bufs[j]

    def release(self, j: int, stream=None):
        self.free[j].record(stream or torch.cuda.current_stream())


@dataclass
class DesignShape:
    P: int
    K: int
    T_max: int
    d: int
    V: int
    rows: int                     # rollout tokens (sum of the completions' lengths)
    topk: int = 16                # next tokens kept per rollout token for u_t (0: no u_t)


class CutoffDesign:
    """The cutoff design upstream of the update (Algorithm 1, steps 7-9), with buffers held in torch.

    CutoffDesign owns the device buffers of one batch shape and runs, on the current stream:
    the score proxy (and, with topk > 0, the top-k next tokens) of every rollout token under the
    old-policy head; the reward-uncertainty proxy u_t per prompt and step; and the design of each
    prompt's cutoff distribution into sampler masses `q` [P][T_max] (sample them with
    PS_MODE_TRUNC_ZERO: a design may leave Pr(H = 0) > 0).
    """

    def __init__(self, shape: DesignShape, device: str = "cuda"):
        s = shape
        self.s, self.device = s, device
        f32 = dict(dtype=torch.float32, device=device)
        u8 = dict(dtype=torch.uint8, device=device)
        self.gamma = torch.empty(s.rows, **f32)
        self.logp = torch.empty(s.rows, **f32)
        k = max(s.topk, 0)
        self.top_idx = torch.empty(s.rows, max(k, 1), dtype=torch.int32, device=device)
        self.top_prob = torch.empty(s.rows, max(k, 1), **f32)
        self.u = torch.empty(s.P, s.T_max, **f32)
        self.y = torch.empty(s.P * s.K, **f32)          # reward labels for u_t (continuous rewards)
        self.q = torch.zeros(s.P, s.T_max, dtype=torch.int64, device=device)
        self.xi = torch.zeros(s.P, s.T_max, dtype=torch.float64, device=device)
        self.ws_proxy = torch.zeros(B.ps_lmhead_score_proxy_workspace_size(s.rows, s.d, s.V, B.PS_DTYPE_BF16, k),
                                    **u8)
        self.ws_u = torch.zeros(B.ps_reward_uncertainty_workspace_size(s.P, s.K), **u8) if k > 0 else None
        self.ws_design = torch.zeros(B.ps_design_cutoffs_workspace_size(s.P, s.K, s.T_max), **u8)

    def score(self, hid_full, W_old, tok_full):
        """gamma (and log p(o), and the top-k next tokens) of every rollout token."""
        s = self.s
        k = max(s.topk, 0)
        B.ps_lmhead_score_proxy(s.rows, s.d, s.V, B.PS_DTYPE_BF16, hid_full, W_old, tok_full, self.gamma, self.logp,
                                self.ws_proxy, k, self.top_idx if k else None, self.top_prob if k else None)

    def uncertainty(self, L, R, continuous: bool = False, seed: int = 0, step: int = 0, traj_base: int = 0):
        """u_t per prompt and step. With continuous rewards, each is first turned into a label
        y ~ Bernoulli(sigma(R)) (Appendix G; ps_binarize_rewards) used for u_t only."""
        s = self.s
        if s.topk <= 0:
            raise ValueError("u_t needs the top-k next tokens (topk > 0)")
        labels = R
        if continuous:
            B.ps_binarize_rewards(s.P * s.K, R, seed, step, self.y, traj_base)
            labels = self.y
        B.ps_reward_uncertainty(s.P, s.K, s.T_max, L, labels, s.topk, self.top_idx, self.top_prob, self.u,
                                self.ws_u)

    def design(self, L, budget: float, strategy: int = B.PS_DESIGN_OPTIMIZED, param: float = 0.0,
               use_u: bool = True):
        s = self.s
        B.ps_design_cutoffs(s.P, s.K, s.T_max, L, self.gamma, self.u if (use_u and s.topk > 0) else None, budget,
                            strategy, param, self.q, self.xi, self.ws_design)

    def run(self, hid_full, W_old, tok_full, L, R, budget: float, strategy: int = B.PS_DESIGN_OPTIMIZED,
            param: float = 0.0, continuous: bool = False, seed: int = 0, step: int = 0):
        """Proxy -> u_t -> design; returns the masses q."""
        if strategy in (B.PS_DESIGN_OPTIMIZED, B.PS_DESIGN_HEURISTIC):
            self.score(hid_full, W_old, tok_full)
            if self.s.topk > 0:
                self.uncertainty(L, R, continuous, seed, step)
        self.design(L, budget, strategy, param)
        return self.q

    def check_status(self):
        """Raise PsppoError if any workspace reports a device-side error."""
        for name, ws in (("proxy", self.ws_proxy), ("uncertainty", self.ws_u), ("design", self.ws_design)):
            if ws is None:
                continue
            rc, bits = B.ps_workspace_status(ws)
            if rc != B.PS_OK:
                raise B.PsppoError(rc, f"{name} (device bits {bits:#x})")
