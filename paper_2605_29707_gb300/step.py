"""DraftStep: keeps the device weights, a workspace and output buffers for one shape and
calls the C ABI.  PyTorch only allocates device memory and provides the stream."""
from __future__ import annotations

import torch

from . import binding as B_


def _dev_bf16(a, device):
    """uint16 bf16 bit patterns (numpy) -> bf16 device tensor (the same bytes)."""
    if a is None:
        return None
    t = torch.from_numpy(a.view("int16")).view(torch.bfloat16)
    return t.to(device, non_blocking=False).contiguous()


class DraftStep:
    def __init__(self, weights: dict, B: int, K: int, H: int, V: int, k: int, N: int, Ds: int = 1024,
                 R: int = 256, device="cuda", head_on: bool = True, input_table: bool = False):
        self.B, self.K, self.H, self.V, self.k, self.N = B, K, H, V, k, N
        self.device = torch.device(device)
        self.head_on = head_on and R > 0 and weights.get("w2") is not None
        self.Ds, self.R = (Ds, R) if self.head_on else (0, 0)
        dev = self.device
        self.w = {n: (_dev_bf16(a, dev) if not isinstance(a, torch.Tensor) else a)
                  for n, a in weights.items() if a is not None}
        w = self.w
        self.head = B_.make_head(w.get("emb"), w.get("w_ih"), w.get("w_hh"), w.get("b_ih"), w.get("b_hh"),
                                 w.get("w1"), w.get("b1"), w.get("w2") if self.head_on else None, w.get("b2"),
                                 self.Ds, self.R)
        # optional input-projection table emb . W_ih^T [V, 3 Ds] fp32, built once on the device
        # (every entry point then reads the GRU's input-gate sums from it)
        self.x_table = None
        if input_table and self.head_on:
            self.x_table = torch.empty(B_.domino_input_table_bytes(V, self.Ds) // 4, dtype=torch.float32,
                                       device=dev)
            rc = B_.domino_build_input_table(w["emb"], w["w_ih"], V, H, self.Ds, self.x_table,
                                             torch.cuda.current_stream(dev))
            if rc != B_.DOMINO_OK:
                raise B_.DominoError(rc, "domino_build_input_table")
            self.head.x_table = self.x_table.data_ptr()
        self.ws_bytes = B_.domino_workspace_bytes(B, K, H, V, self.Ds, self.R, k, N)
        if self.ws_bytes == 0:
            raise B_.DominoError(B_.DOMINO_ERR_UNSUPPORTED, "domino_workspace_bytes")
        self.ws_host_bytes = B_.domino_workspace_bytes_host(B, K, H, V, self.Ds, self.R, k, N)
        # zero-filled once: the library expects a zero workspace at its first use
        self.workspace = torch.zeros(self.ws_host_bytes, dtype=torch.uint8, device=dev)
        M = B * K
        self.topk_ids = torch.empty(M * k, dtype=torch.int32, device=dev)
        self.topk_logp = torch.empty(M * k, dtype=torch.float32, device=dev)
        self.tree_parent = torch.empty(B * N, dtype=torch.int32, device=dev)
        self.tree_token = torch.empty(B * N, dtype=torch.int32, device=dev)
        self.tree_depth = torch.empty(B * N, dtype=torch.int32, device=dev)
        self.tree_score = torch.empty(B * N, dtype=torch.float32, device=dev)

    def launches_per_step(self) -> int:
        f = B_.domino_launches_per_step_table if self.x_table is not None else B_.domino_launches_per_step
        return f(self.B, self.K, self.H, self.V, self.Ds, self.R, self.k, self.N)

    def enqueue(self, hidden: torch.Tensor, prefix_ids: torch.Tensor, stream=None) -> int:
        """Enqueue one step on `stream` (default: torch's current stream); returns the C status."""
        if stream is None:
            stream = torch.cuda.current_stream(self.device)
        return B_.domino_draft_step(hidden, prefix_ids, self.w["w_lm"], self.head, self.B, self.K, self.H,
                                    self.V, self.k, self.N, self.topk_ids, self.topk_logp, self.tree_parent,
                                    self.tree_token, self.tree_depth, self.tree_score, self.workspace,
                                    self.ws_bytes, stream)

    def run(self, hidden: torch.Tensor, prefix_ids: torch.Tensor, stream=None) -> dict:
        rc = self.enqueue(hidden, prefix_ids, stream)
        if rc != 0:
            raise B_.DominoError(rc, "domino_draft_step")
        if stream is None:
            stream = torch.cuda.current_stream(self.device)
        rc = B_.domino_check_status(self.workspace, stream)
        if rc != 0:
            raise B_.DominoError(rc, "device status")
        return self.outputs()

    def outputs(self) -> dict:
        B, K, k, N = self.B, self.K, self.k, self.N
        return {
            "topk_ids": self.topk_ids.view(B, K, k).cpu().numpy(),
            "topk_logp": self.topk_logp.view(B, K, k).cpu().numpy(),
            "tree_parent": self.tree_parent.view(B, N).cpu().numpy(),
            "tree_token": self.tree_token.view(B, N).cpu().numpy(),
            "tree_depth": self.tree_depth.view(B, N).cpu().numpy(),
            "tree_score": self.tree_score.view(B, N).cpu().numpy(),
        }

    def run_host(self, hidden_host: torch.Tensor, ids_host: torch.Tensor, out: dict, stream=None) -> int:
        """The host-buffer entry point: inputs and outputs are (pinned) CPU tensors."""
        if stream is None:
            stream = torch.cuda.current_stream(self.device)
        return B_.domino_draft_step_host(hidden_host, ids_host, self.w["w_lm"], self.head, self.B, self.K,
                                         self.H, self.V, self.k, self.N, out["topk_ids"], out["topk_logp"],
                                         out["tree_parent"], out["tree_token"], out["tree_depth"],
                                         out["tree_score"], self.workspace, self.ws_host_bytes, stream)
