"""MQAR capacity smoke study (Section 2.3, Appendix C) with the CUDA kernels under autograd.

A reduced version of the paper's setup: two blocks of vanilla triadic linear attention
(Algorithm 1: no forgetting, no delta rule, RMSNorm per head on the read-out) and SwiGLU
MLPs, d_model 128, 4 heads of D = 16, E slices.  A sequence holds N key-value pairs, one
token each (key and value embeddings concatenated), then the N keys in random order as
read-only queries (key embedding and zeros; their second key is zeroed so they do not
write); the loss is the cross-entropy of the value at the query positions.  Smaller
vocabulary and far fewer steps than the paper (which trains 50k steps of 250k tokens).

Run directly for the small study:  python tests/mqar.py [--steps S] [--n N ...] [--e E ...]
"""
import argparse
import json
import os
import sys
import time

import torch
import torch.nn as nn
import torch.nn.functional as F

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

from paper_2609_36529_gb300.autograd import triadic_linear_attention  # noqa: E402


class RMSNorm(nn.Module):
    def __init__(self, d, eps=1e-6):
        super().__init__()
        self.w = nn.Parameter(torch.ones(d))
        self.eps = eps

    def forward(self, x):
        return x * torch.rsqrt(x.pow(2).mean(-1, keepdim=True) + self.eps) * self.w


class Block(nn.Module):
    def __init__(self, d, H, D, E, mlp):
        super().__init__()
        self.H, self.D, self.E = H, D, E
        self.n1 = RMSNorm(d)
        self.wq, self.wk, self.wv = (nn.Linear(d, H * D, bias=False) for _ in range(3))
        self.wq2, self.wk2 = (nn.Linear(d, H * E, bias=False) for _ in range(2))
        self.on = RMSNorm(D)
        self.wo = nn.Linear(H * D, d, bias=False)
        self.n2 = RMSNorm(d)
        self.gate, self.up = (nn.Linear(d, mlp, bias=False) for _ in range(2))
        self.down = nn.Linear(mlp, d, bias=False)

    def forward(self, x, writes):
        B, T, _ = x.shape
        H, D, E = self.H, self.D, self.E
        u = self.n1(x)
        q = self.wq(u).view(B, T, H, D)
        k = self.wk(u).view(B, T, H, D)
        v = self.wv(u).view(B, T, H, D)
        q2 = self.wq2(u).view(B, T, H, E)
        k2 = (self.wk2(u).view(B, T, H, E) * writes[:, :, None, None]).contiguous()
        g = torch.zeros(B, T, H, E, device=x.device)   # no forgetting
        o, _ = triadic_linear_attention(q, k, v, q2, k2, g, None, None, use_delta=False)
        x = x + self.wo(self.on(o).reshape(B, T, H * D))
        u = self.n2(x)
        return x + self.down(F.silu(self.gate(u)) * self.up(u))


class MQARModel(nn.Module):
    def __init__(self, n_keys, n_vals, E, d=128, H=4, D=16, layers=2, mlp=384):
        super().__init__()
        self.key_emb = nn.Embedding(n_keys, d // 2)
        self.val_emb = nn.Embedding(n_vals, d // 2)
        self.blocks = nn.ModuleList(Block(d, H, D, E, mlp) for _ in range(layers))
        self.norm = RMSNorm(d)
        self.head = nn.Linear(d, n_vals, bias=False)

    def forward(self, keys, vals, is_query):
        ve = self.val_emb(vals) * (~is_query)[..., None].float()
        x = torch.cat([self.key_emb(keys), ve], -1)
        writes = (~is_query).float()
        for blk in self.blocks:
            x = blk(x, writes)
        return self.head(self.norm(x))


def mqar_batch(B, N, n_keys, n_vals, gen, device):
    """Keys and values drawn without replacement; the queries are the keys permuted."""
    keys = torch.stack([torch.randperm(n_keys, generator=gen)[:N] for _ in range(B)])
    vals = torch.stack([torch.randperm(n_vals, generator=gen)[:N] for _ in range(B)])
    perm = torch.stack([torch.randperm(N, generator=gen) for _ in range(B)])
    qkeys, target = torch.gather(keys, 1, perm), torch.gather(vals, 1, perm)
    K = torch.cat([keys, qkeys], 1)
    V = torch.cat([vals, torch.zeros_like(target)], 1)
    isq = torch.cat([torch.zeros(B, N, dtype=torch.bool), torch.ones(B, N, dtype=torch.bool)], 1)
    return K.to(device), V.to(device), isq.to(device), target.to(device)


def train(E, N, steps, batch=64, n_keys=1024, n_vals=1024, lr=1e-3, seed=0, device="cuda",
          eval_batches=4, fixed_batch=False):
    """Returns (loss of the first step, loss of the last step, held-out query accuracy).
    fixed_batch: train on one batch throughout (a memorisation check of the gradients)."""
    torch.manual_seed(seed)
    gen = torch.Generator().manual_seed(seed)
    model = MQARModel(n_keys, n_vals, E).to(device)
    opt = torch.optim.AdamW(model.parameters(), lr=lr, betas=(0.9, 0.999), weight_decay=0.1)
    sched = torch.optim.lr_scheduler.LambdaLR(
        opt, lambda s: 0.5 * (1 + torch.cos(torch.tensor(3.14159265 * s / steps)).item()))
    first = last = None
    fixed = mqar_batch(batch, N, n_keys, n_vals, gen, device) if fixed_batch else None
    for s in range(steps):
        K, V, isq, tgt = fixed if fixed_batch else mqar_batch(batch, N, n_keys, n_vals, gen, device)
        logits = model(K, V, isq)[:, N:]
        loss = F.cross_entropy(logits.reshape(-1, n_vals), tgt.reshape(-1))
        opt.zero_grad(set_to_none=True)
        loss.backward()
        opt.step()
        sched.step()
        if first is None:
            first = float(loss.detach())
        last = float(loss.detach())
    held = torch.Generator().manual_seed(10_000 + seed)
    correct = total = 0
    with torch.no_grad():
        for _ in range(eval_batches):
            K, V, isq, tgt = mqar_batch(batch, N, n_keys, n_vals, held, device)
            pred = model(K, V, isq)[:, N:].argmax(-1)
            correct += int((pred == tgt).sum())
            total += tgt.numel()
    return first, last, correct / total


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--steps", type=int, default=1500)
    ap.add_argument("--n", type=int, nargs="+", default=[64, 256])
    ap.add_argument("--e", type=int, nargs="+", default=[1, 4, 16])
    ap.add_argument("--batch", type=int, default=64)
    ap.add_argument("--vocab", type=int, default=1024)
    ap.add_argument("--lr", type=float, default=1e-3)
    args = ap.parse_args()
    rows = []
    for N in args.n:
        for E in args.e:
            t0 = time.time()
            first, last, acc = train(E, N, args.steps, batch=args.batch, n_keys=args.vocab,
                                     n_vals=args.vocab, lr=args.lr)
            rows.append({"N": N, "E": E, "steps": args.steps, "batch": args.batch,
                         "vocab": args.vocab, "lr": args.lr,
                         "loss_first": round(first, 3), "loss_last": round(last, 3),
                         "accuracy": round(acc, 4), "seconds": round(time.time() - t0, 1)})
            print(json.dumps(rows[-1]), flush=True)


if __name__ == "__main__":
    main()
