"""Buffer management around the libqk C ABI.

PyTorch supplies device memory and streams; every computation is a libqk call.
``Decoder`` owns the packed weights, KV caches and workspaces (all torch
tensors, so the library itself never allocates) and forwards to the binding.
"""
from __future__ import annotations

import numpy as np
import torch

from . import _binding as B


def _to_device(arr: np.ndarray, device) -> torch.Tensor:
    if arr.dtype == np.uint16:
        t = torch.from_numpy(arr.view(np.int16))
    else:
        t = torch.from_numpy(np.ascontiguousarray(arr))
    return t.to(device, non_blocking=False)


class Decoder:
    """A loaded model plus cached workspaces.

    host_tensors: a sequence (or an iterable) of numpy arrays in the canonical
    order of qk_model_load (bf16 as uint16 bit patterns, or float32).  Tensors
    are uploaded in groups so that the unpacked copy never exceeds ~group_bytes.
    """

    def __init__(self, cfg: B.qk_config, host_tensors, device="cuda", group_bytes=4 << 30):
        self.cfg = cfg
        self.device = torch.device(device)
        n = B.qk_weight_count(cfg)
        self.packed = torch.empty(B.qk_model_packed_bytes(cfg), dtype=torch.uint8, device=self.device)
        tensors = list(host_tensors)
        if len(tensors) != n:
            raise ValueError(f"expected {n} tensors, got {len(tensors)}")
        # The loader repacks all tensors in one call, so every tensor must be resident at once.
        dev = [_to_device(np.asarray(a), self.device) for a in tensors]
        self.handle = B.qk_model_load(cfg, dev, self.packed)
        torch.cuda.current_stream(self.device).synchronize()
        del dev
        self._ws = {}

    def close(self):
        if self.handle:
            B.qk_model_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ------------------------------------------------------------ buffers
    def new_kv(self, max_batch: int, max_seq: int) -> torch.Tensor:
        return torch.empty(B.qk_kv_bytes(self.handle, max_batch, max_seq), dtype=torch.uint8,
                           device=self.device)

    def workspace(self, kind: int, Bn: int, T: int, max_seq: int = 1) -> torch.Tensor:
        need = B.qk_workspace_bytes(self.handle, kind, Bn, T, max_seq)
        ws = self._ws.get(kind)
        if ws is None or ws.numel() < need:
            ws = torch.empty(need, dtype=torch.uint8, device=self.device)
            self._ws[kind] = ws
        return ws

    def kv_view(self, kv: torch.Tensor, max_batch: int, max_seq: int):
        """The cache as [layers, 2, max_batch, n_kv, max_seq, d] in the model dtype."""
        c = self.cfg
        dt = torch.bfloat16 if c.dtype == B.QK_DTYPE_BF16 else torch.float32
        return kv.view(dt).view(c.n_layers, 2, max_batch, c.n_kv_heads, max_seq, c.head_dim)

    # ------------------------------------------------------------ calls
    def prefill(self, kv, max_batch, max_seq, tokens, start_pos=0, last_logits=None, targets=None,
                logprobs=None, argmax=None):
        Bn, T = tokens.shape
        ws = self.workspace(B.QK_CALL_PREFILL, Bn, T, max_seq)
        B.qk_prefill(self.handle, kv, max_batch, max_seq, tokens, Bn, T, start_pos, last_logits,
                     targets, logprobs, argmax, ws)

    def decode_step(self, kv, max_batch, max_seq, tokens, pos, logits=None, targets=None,
                    logprobs=None, argmax=None):
        Bn = tokens.shape[0]
        ws = self.workspace(B.QK_CALL_DECODE, Bn, 1, max_seq)
        B.qk_decode_step(self.handle, kv, max_batch, max_seq, tokens, pos, Bn, logits, targets,
                         logprobs, argmax, ws)

    def decode_layer(self, layer, kv, max_batch, max_seq, x, pos):
        Bn = x.shape[0]
        ws = self.workspace(B.QK_CALL_DECODE, Bn, 1, max_seq)
        B.qk_decode_layer(self.handle, layer, kv, max_batch, max_seq, x, pos, Bn, ws)

    def score(self, tokens, logprobs=None, argmax=None):
        Bn, T = tokens.shape
        if logprobs is None:
            logprobs = torch.empty(Bn, T - 1, dtype=torch.float32, device=self.device)
        ws = self.workspace(B.QK_CALL_SCORE, Bn, T)
        B.qk_score_logprobs(self.handle, tokens, Bn, T, logprobs, argmax, ws)
        return logprobs

    def score_grpo(self, tokens, lp_old, rewards, group, lp_ref=None, mask=None, eps_low=0.2,
                   eps_high=0.28, beta=0.01):
        """Scoring with the GRPO token loss formed in the log-prob epilogue.
        Returns (logprobs [B, T-1], loss_tok [B, T-1], loss_mean [1])."""
        Bn, T = tokens.shape
        logprobs = torch.empty(Bn, T - 1, dtype=torch.float32, device=self.device)
        loss_tok = torch.empty(Bn, T - 1, dtype=torch.float32, device=self.device)
        loss_mean = torch.empty(1, dtype=torch.float32, device=self.device)
        need = (B.qk_workspace_bytes(self.handle, B.QK_CALL_SCORE, Bn, T, T) + 255) // 256 * 256
        need += B.qk_grpo_workspace_bytes(Bn)
        ws = self._ws.get("score_grpo")
        if ws is None or ws.numel() < need:
            ws = torch.empty(need, dtype=torch.uint8, device=self.device)
            self._ws["score_grpo"] = ws
        B.qk_score_grpo(self.handle, tokens, Bn, T, lp_old, lp_ref, rewards, group, mask, eps_low,
                        eps_high, beta, logprobs, loss_tok, loss_mean, ws)
        return logprobs, loss_tok, loss_mean

    def weight_shapes(self):
        """Shapes of the weight tensors in the canonical order of qk_model_load."""
        c = self.cfg
        H, d, nq, nkv, I, V = c.hidden, c.head_dim, c.n_q_heads, c.n_kv_heads, c.intermediate, c.vocab
        layer = [(H,), (nq * d, H), (nkv * d, H), (nkv * d, H), (d,), (d,), (H, nq * d), (H,), (I, H),
                 (I, H), (H, I)]
        return [(V, H)] + layer * c.n_layers + [(H,), (V, H)]

    def new_grads(self):
        """fp32 gradient buffers, one per weight tensor (canonical order)."""
        return [torch.empty(shp, dtype=torch.float32, device=self.device) for shp in self.weight_shapes()]

    def backward(self, tokens, coef, grads, accumulate=False, loss=None):
        """d/d theta of sum coef[b, t] * (-log p(tokens[b, t+1] | tokens[b, <= t])) into grads
        (qk_backward_logprob); returns loss [1]."""
        Bn, T = tokens.shape
        if loss is None:
            loss = torch.empty(1, dtype=torch.float32, device=self.device)
        ws = self.workspace(B.QK_CALL_BACKWARD, Bn, T)
        B.qk_backward_logprob(self.handle, tokens, Bn, T, coef, grads, int(bool(accumulate)), loss, ws)
        return loss

    def prefill_rows(self, kv, max_batch, max_seq, tokens, start, length=None, last_logits=None):
        """Append tokens[b, :length[b]] to row b at positions start[b] .. (rows at different
        positions; entries past length[b] are padding)."""
        Bn, T = tokens.shape
        ws = self.workspace(B.QK_CALL_PREFILL, Bn, T, max_seq)
        B.qk_prefill_rows(self.handle, kv, max_batch, max_seq, tokens, Bn, T, start, length,
                          last_logits, ws)
        return last_logits

    def rollout_sampled(self, kv, max_batch, max_seq, prompt, N, tau=1.0, seed=0):
        """Sampled rollout (Gumbel-max at temperature tau): returns (tokens [B, N+1],
        logprobs [B, N+1]) for the draws c[0..N] after the prompt [B, P]."""
        Bn, P = prompt.shape
        tokens = torch.empty(Bn, N + 1, dtype=torch.int32, device=self.device)
        logprobs = torch.empty(Bn, N + 1, dtype=torch.float32, device=self.device)
        ws = self.workspace(B.QK_CALL_ROLLOUT, Bn, P, max_seq)
        B.qk_rollout_sampled(self.handle, kv, max_batch, max_seq, prompt, Bn, P, N, tau, seed, tokens,
                             logprobs, ws)
        return tokens, logprobs

    def rollout(self, kv, max_batch, max_seq, seq, P, logprobs=None, argmax=None):
        Bn, L = seq.shape
        N = L - P - 1
        if logprobs is None:
            logprobs = torch.empty(Bn, N + 1, dtype=torch.float32, device=self.device)
        ws = self.workspace(B.QK_CALL_ROLLOUT, Bn, P, max_seq)
        B.qk_rollout_teacher_forced(self.handle, kv, max_batch, max_seq, seq, Bn, P, N, logprobs,
                                    argmax, ws)
        return logprobs

    # ------------------------------------------------------------ paged cache
    def new_kv_pages(self, n_pages: int, page_size: int) -> torch.Tensor:
        """A paged cache of n_pages pages of page_size positions (per layer a K pool then a
        V pool, each [n_pages, n_kv, page_size, d])."""
        return torch.empty(B.qk_kv_pages_bytes(self.handle, n_pages, page_size), dtype=torch.uint8,
                           device=self.device)

    def decode_step_paged(self, kv, table, n_pages, page_size, tokens, pos, logits=None, targets=None,
                          logprobs=None, argmax=None):
        """decode_step over a paged cache; table: device int32 [B, per_row] page ids."""
        Bn, per_row = table.shape
        assert table.dtype == torch.int32 and table.is_contiguous()
        ws = self.workspace(B.QK_CALL_DECODE, tokens.shape[0], 1, per_row * page_size)
        B.qk_decode_step_paged(self.handle, kv, table, per_row, n_pages, page_size, tokens, pos,
                               tokens.shape[0], logits, targets, logprobs, argmax, ws)

    def prefill_rows_paged(self, kv, table, n_pages, page_size, tokens, start, length=None,
                           last_logits=None):
        """prefill_rows over a paged cache; table: device int32 [B, per_row] page ids."""
        Bn, T = tokens.shape
        assert table.dtype == torch.int32 and table.is_contiguous()
        per_row = table.shape[1]
        ws = self.workspace(B.QK_CALL_PREFILL, Bn, T, per_row * page_size)
        B.qk_prefill_rows_paged(self.handle, kv, table, per_row, n_pages, page_size, tokens, Bn, T, start,
                                length, last_logits, ws)
        return last_logits

    def rollout_paged(self, kv, table, n_pages, page_size, seq, P, logprobs=None, argmax=None):
        """rollout over a paged cache; table: device int32 [B, per_row] page ids."""
        Bn, L = seq.shape
        N = L - P - 1
        per_row = table.shape[1]
        assert table.dtype == torch.int32 and table.is_contiguous()
        if logprobs is None:
            logprobs = torch.empty(Bn, N + 1, dtype=torch.float32, device=self.device)
        ws = self.workspace(B.QK_CALL_ROLLOUT, Bn, P, per_row * page_size)
        B.qk_rollout_teacher_forced_paged(self.handle, kv, table, per_row, n_pages, page_size, seq, Bn, P, N,
                                          logprobs, argmax, ws)
        return logprobs

    def rollout_sampled_paged(self, kv, table, n_pages, page_size, prompt, N, tau=1.0, seed=0):
        """rollout_sampled over a paged cache; table: device int32 [B, per_row] page ids."""
        Bn, P = prompt.shape
        per_row = table.shape[1]
        assert table.dtype == torch.int32 and table.is_contiguous()
        tokens = torch.empty(Bn, N + 1, dtype=torch.int32, device=self.device)
        logprobs = torch.empty(Bn, N + 1, dtype=torch.float32, device=self.device)
        ws = self.workspace(B.QK_CALL_ROLLOUT, Bn, P, per_row * page_size)
        B.qk_rollout_sampled_paged(self.handle, kv, table, per_row, n_pages, page_size, prompt, Bn, P, N, tau,
                                   seed, tokens, logprobs, ws)
        return tokens, logprobs

    def check_status(self) -> int:
        return B.qk_check_status(self.handle)


def grpo_token_loss(lp, lp_old, rewards, group, lp_ref=None, mask=None, eps_low=0.2, eps_high=0.28,
                    beta=0.01, stream=None):
    """GRPO token loss over precomputed log-probs [B, T] (contiguous rows): returns
    (loss_tok [B, T], loss_mean [1]); every step runs in libqk's kernels."""
    Bn, T = lp.shape
    loss_tok = torch.empty_like(lp)
    loss_mean = torch.empty(1, dtype=torch.float32, device=lp.device)
    ws = torch.empty(B.qk_grpo_workspace_bytes(Bn), dtype=torch.uint8, device=lp.device)
    B.qk_grpo_token_loss(lp, lp_old, lp_ref, Bn, T, T, rewards, group, mask, eps_low, eps_high, beta,
                         loss_tok, loss_mean, ws, stream=stream)
    return loss_tok, loss_mean
