"""A Kafila ring emulated on one GPU, serving several users at once.

A session serves the model as a ring (section III): the head embeds a user's token and runs its
blocks, each member runs its contiguous block range in turn, and the hidden state returns to the
head for the final RMSNorm, lm_head and sampler (the head's return leg).  Decoding one user is
sequential around the ring, so at any instant one stage computes and the others wait; several
users' requests fill that bubble, each stage working on one user's token while another stage works
on the next user's (section VII, "Serving several users at once"; Eq. 1's compute term).

Here every member is a stage of the library on this GPU, with its own CUDA stream, and the return
leg is a stage of its own (no blocks, KFL_LOGITS_OUT).  A stage serves one user per call
(kfl_stage_decode_users, batch 1, the user's own KV slot); CUDA events order a user's token from
stage to stage and feed the return leg's greedy token back to the head.  The stages share the
GPU's SMs and HBM, so what overlaps is one stage's latency-bound phases with another's streaming.

Argument marshalling and stream scheduling only: every step of the path runs in the library.
"""
from __future__ import annotations

import dataclasses

import torch

from . import device_inputs as di
from . import stage as K
from . import workload as wl


class Ring:
    """Stages for the given block counts (in ring order, the head first) plus the head's return
    leg, for `users` concurrent users of workload `work`'s model."""

    def __init__(self, work: wl.Workload, counts: list, users: int):
        m = work.model
        if sum(counts) != m.n_layers_total or min(counts) < 1:
            raise ValueError("the block counts must cover the model's blocks, at least one each")
        # one pre-filled context per user (the workload's, cycled)
        ctx = tuple(work.contexts[u % len(work.contexts)] for u in range(users))
        work = dataclasses.replace(work, batch=users, contexts=ctx, l0=0, l1=m.n_layers_total, splits=())
        self.work, self.users, self.d = work, users, m.d_model
        cfg = K.model_cfg(m, work.max_ctx, users)
        self.bounds = [0]
        for n in counts:
            self.bounds.append(self.bounds[-1] + n)
        self.stages = []
        for i in range(len(counts)):
            st = K.kfl_stage_create(cfg, self.bounds[i], self.bounds[i + 1], K.KFL_EMBED_IN if i == 0 else 0)
            di.load_stage_seeded(st, work, self.bounds[i], self.bounds[i + 1])
            self.stages.append(st)
        L = m.n_layers_total
        self.ret = K.kfl_stage_create(cfg, L, L, K.KFL_LOGITS_OUT)
        di.load_stage_seeded(self.ret, work, L, L)
        self.all = self.stages + [self.ret]
        self.streams = [torch.cuda.Stream() for _ in self.all]
        dev = "cuda"
        self.user_ids = [torch.tensor([u], dtype=torch.int32, device=dev) for u in range(users)]
        self.tok = [torch.zeros(1, dtype=torch.int32, device=dev) for _ in range(users)]
        self.hid = [[torch.empty(1, self.d, dtype=torch.float32, device=dev) for _ in range(users)]
                    for _ in self.all]

    def close(self):
        torch.cuda.synchronize()
        for st in self.all:
            if K.kfl_stage_status(st) != 0:
                raise RuntimeError("device reported an error in a ring stage")
            K.kfl_stage_destroy(st)

    def _positions(self, tokens: int, start: int):
        """int32 [tokens][users] device tensors: user u's position at its token t."""
        ctx = self.work.contexts
        return [[torch.tensor([ctx[u] + start + t], dtype=torch.int32, device="cuda")
                 for u in range(self.users)] for t in range(tokens)]

    def run(self, first_ids: list, tokens: int, start: int = 0, sequential: bool = False):
        """Decode `tokens` greedy tokens for every user (user u starts from first_ids[u]); returns
        the generated ids [tokens][users] (a host list).  sequential: every stage's work goes to
        one stream in the same order (no overlap between stages), else each stage has its own."""
        S = len(self.all)
        pos = self._positions(tokens, start)
        for u in range(self.users):
            self.tok[u].fill_(int(first_ids[u]))
        out = [[torch.zeros(1, dtype=torch.int32, device="cuda") for _ in range(self.users)] for _ in range(tokens)]
        streams = [self.streams[0]] * S if sequential else self.streams
        done = {}  # (stage, user) -> event of the user's latest token through that stage
        main = torch.cuda.current_stream()
        for s_ in streams:
            s_.wait_stream(main)
        for t in range(tokens):
            for u in range(self.users):
                for k, st in enumerate(self.all):
                    stream = streams[k]
                    # the user's token from the stage before (the head: the return leg's last id)
                    dep = done.get((k - 1, u)) if k > 0 else done.get((S - 1, u))
                    if dep is not None:
                        stream.wait_event(dep)
                    with torch.cuda.stream(stream):
                        if k == 0:
                            K.kfl_stage_decode_users(st, self.tok[u], None, pos[t][u], self.user_ids[u], 1,
                                                     self.hid[k][u], None, stream.cuda_stream)
                        elif k < S - 1:
                            K.kfl_stage_decode_users(st, None, self.hid[k - 1][u], pos[t][u], self.user_ids[u], 1,
                                                     self.hid[k][u], None, stream.cuda_stream)
                        else:
                            K.kfl_stage_decode_users(st, None, self.hid[k - 1][u], pos[t][u], self.user_ids[u], 1,
                                                     None, self.tok[u], stream.cuda_stream)
                            out[t][u].copy_(self.tok[u])
                    ev = torch.cuda.Event()
                    ev.record(stream)
                    done[(k, u)] = ev
        for s_ in streams:
            main.wait_stream(s_)
        torch.cuda.synchronize()
        return [[int(out[t][u].item()) for u in range(self.users)] for t in range(tokens)]
