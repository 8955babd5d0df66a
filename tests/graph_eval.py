"""Direct evaluation of a front-end Graph IR on the CPU (float64 numpy).

Test infrastructure for the Axon-subset front end: it runs a module's Graph
IR node by node on its own parameter paths, so a test can check that what a
module states (before or after the stacked-experts rewrite) is the function
the lowered model computes -- the oracle run on the checkpoint re-keyed
through the lowering's name map. It runs a pass over new tokens after the
ones a cache already holds (a prompt from an empty cache, then decode
steps), with the cache the module threads through its layer loop, and the
operations the decoder modules use; each follows the library operation's
meaning in the paper's built-ins (Sec. Built-In Libraries):

  Cache.past_length / prepare / index     tokens cached; the work cache; layer i's
  Cache.update / append                   (K, V) so far; keys and values appended
                                          along the sequence; the layer's new entry
  Masking.causal_mask_for_input / causal_mask
                                          causal (and windowed) over cached + new keys

  NN.embedding / NN.rmsnorm / NN.linear   rows of E; x / sqrt(mean x^2 + eps) * g;
                                          x W^T (+ b), W stored [out, in]
  Attention.reshape_heads / merge_heads   [.., n*d] <-> [.., n, d]
  Positions.position_ids / rope           past + i; rotate-half pairs (j, j + d/2),
                                          angle p * theta^(-2j/d)
  Attention.attention                     softmax(q k^T / sqrt(d)) v over keys at
                                          positions <= the query's (and > p - window),
                                          query head h on kv head floor(h / (H/G))
  Act.silu / Act.gelu_tanh                z / (1 + e^-z); tanh form of gelu
  Act.swiglu z                            silu(z[.., :F]) * z[.., F:], F = width / 2
  Attention.split_qkv t heads kv_heads    rows of t cut into q (heads * d), k and v
                                          (kv_heads * d each), each split into heads
  MoE.softmax_topk_router                 p = softmax(x Wr^T); the top_k experts by p
                                          (lower index first on ties) and their p,
                                          divided by their sum with normalize=true
  MoE.expert_weight w idx e               the weight expert e received (0 if none)
  MoE.stacked_experts                     init + sum_e expert_weight(e) * ffn_e(h)
"""
from __future__ import annotations

import math

import numpy as np

from paper_2608_19889_gb300.frontend import graph as gr


class GraphEval:
    """weights: module parameter path + ".weight" / ".bias" -> array."""

    def __init__(self, weights: dict):
        self.W = {k: np.asarray(v, dtype=np.float64) for k, v in weights.items()}

    def run(self, g: gr.Graph, ids, past=None) -> list:
        """The entry's outputs for new tokens ids [B, S] after `past` (None:
        empty; else the cache of the previous run, see next_past)."""
        ids = np.asarray(ids, dtype=np.int64)
        env: dict = {}
        return self._graph(g, [ids, past], env, {})

    @staticmethod
    def next_past(work, ids):
        """The cache after a run that returned `work` for new tokens ids."""
        return {"layers": dict(enumerate(work["out"])), "len": work["len"] + np.asarray(ids).shape[-1]}

    # ------------------------------------------------------------ plumbing
    def _graph(self, g, args, env, loopvars):
        for n in g.nodes:
            if n.op == "input":
                idx = n.attrs["index"]
                env[n.id] = (args[idx] if idx < len(args) else None,)
            else:
                out = self._node(n, env, loopvars)
                env[n.id] = out if n.n_out > 1 else (out,)
        return [self._val(o, env, loopvars) for o in g.outputs]

    def _val(self, x, env, loopvars):
        if isinstance(x, gr.Ref):
            return env[x.node][x.index]
        if isinstance(x, gr.LoopVar):
            return loopvars[x.name]
        return x

    @staticmethod
    def _path(p, loopvars):
        for k, v in loopvars.items():
            p = p.replace("{" + k + "}", str(v))
        return p

    def _w(self, path, loopvars, leaf="weight"):
        return self.W[self._path(path, loopvars) + "." + leaf]

    # ---------------------------------------------------------- operations
    def _node(self, n, env, lv):
        ins = [self._val(x, env, lv) for x in n.inputs]
        at = {k: self._val(v, env, lv) for k, v in n.attrs.items()}
        op = n.op
        if op == "loop":
            vals = ins
            for i in range(at["start"], at["stop"], at.get("step", 1)):
                inner = dict(lv)
                inner[at["var"]] = i
                vals = self._graph(n.body, vals, env, inner)
            return tuple(vals) if n.n_out > 1 else vals[0]
        if op in ("add", "sub", "mul", "div"):
            a, b = ins
            return {"add": np.add, "sub": np.subtract, "mul": np.multiply, "div": np.divide}[op](a, b)
        if op == "NN.embedding":
            return self._w(n.path, lv)[ins[0]]
        if op == "NN.rmsnorm":
            x = ins[0]
            return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + float(at["eps"])) * self._w(n.path, lv)
        if op == "NN.linear":
            y = ins[0] @ self._w(n.path, lv).T
            return y + self._w(n.path, lv, "bias") if at.get("bias") else y
        if op == "Attention.reshape_heads":
            x = ins[0]
            return x.reshape(x.shape[:-1] + (int(at["heads"]), -1))
        if op == "Attention.merge_heads":
            x = ins[0]
            return x.reshape(x.shape[:-2] + (-1,))
        if op == "Cache.past_length":
            return 0 if ins[0] is None else ins[0]["len"]
        if op == "Positions.position_ids":
            ids = ins[0]
            return np.broadcast_to(np.arange(ids.shape[-1]) + int(at.get("past_length") or 0), ids.shape)
        if op in ("Masking.causal_mask_for_input", "Masking.causal_mask"):
            if at.get("padding_mask") is not None:
                raise NotImplementedError("padding masks")
            if op == "Masking.causal_mask":  # from q and k: the keys beyond the queries are cached ones
                return {"window": int(at.get("window", 0) or 0), "past": ins[1].shape[1] - ins[0].shape[1]}
            return {"window": int(at.get("window", 0) or 0), "past": int(ins[1] or 0)}
        if op == "Cache.prepare":
            past = ins[0]
            return {"in": dict(past["layers"]) if past else {}, "out": [], "len": past["len"] if past else 0}
        if op == "Cache.index":
            return ins[0]["in"].get(int(ins[1]))
        if op == "Cache.append":
            work = ins[0]
            return dict(work, out=work["out"] + [ins[1]])
        if op == "Cache.update":
            kv, k, v = ins
            if kv is not None:
                k = np.concatenate([kv[0], k], axis=1)
                v = np.concatenate([kv[1], v], axis=1)
            return k, v, (k, v)
        if op == "Positions.rope":
            return self._rope(ins[0], ins[1], float(at["theta"]), at)
        if op == "Attention.attention":
            if len(ins) < 4 or ins[3] is None:
                raise NotImplementedError("attention without a causal mask")
            return self._attention(ins[0], ins[1], ins[2], ins[3])
        if op == "Act.silu":
            z = ins[0]
            return z / (1.0 + np.exp(-z))
        if op in ("Act.gelu_tanh", "Act.gelu_new", "Activations.gelu_new"):
            z = ins[0]
            return 0.5 * z * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (z + 0.044715 * z ** 3)))
        if op in ("Act.swiglu", "Activations.swiglu"):
            return self._swiglu(ins[0])
        if op == "Attention.split_qkv":
            t, H, G = ins[0], int(at["heads"]), int(at["kv_heads"])
            d = t.shape[-1] // (H + 2 * G)
            q, k, v = t[..., : H * d], t[..., H * d:(H + G) * d], t[..., (H + G) * d:]
            return (q.reshape(q.shape[:-1] + (H, d)), k.reshape(k.shape[:-1] + (G, d)),
                    v.reshape(v.shape[:-1] + (G, d)))
        if op == "Tensor.zeros_like":
            return np.zeros_like(ins[0])
        if op == "MoE.softmax_topk_router":
            return self._route(ins[0], self._w(n.path, lv), int(at["top_k"]), bool(at.get("normalize", False)))
        if op == "MoE.expert_weight":
            w, idx, e = ins
            return np.sum(np.where(idx == e, w, 0.0), axis=-1, keepdims=True)
        if op == "MoE.stacked_experts":
            return self._stacked(ins, at, lv)
        raise NotImplementedError(op)

    @staticmethod
    def _rope(x, pos, theta, at):
        if any(k in at for k in ("factor", "low_freq_factor", "high_freq_factor")):
            raise NotImplementedError("rope frequency scaling")
        d = x.shape[-1]
        inv = theta ** (-2.0 * np.arange(d // 2) / d)
        ang = np.asarray(pos, dtype=np.float64)[..., None, None] * inv  # [B, S, 1, d/2]
        c, s = np.cos(ang), np.sin(ang)
        a, b = x[..., : d // 2], x[..., d // 2:]
        return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)

    @staticmethod
    def _attention(q, k, v, mask):
        B, S, H, d = q.shape
        G = k.shape[2]
        tq = mask.get("past", 0) + np.arange(S)  # query positions after the cached keys
        tk = np.arange(k.shape[1])
        keep = tk[None, :] <= tq[:, None]
        W = mask.get("window", 0)
        if W > 0:
            keep &= tk[None, :] > tq[:, None] - W
        out = np.empty_like(q)
        for b in range(B):
            for h in range(H):
                g = h // (H // G)
                s = q[b, :, h, :] @ k[b, :, g, :].T / math.sqrt(d)
                s = np.where(keep, s, -np.inf)
                s = np.exp(s - s.max(axis=-1, keepdims=True))
                out[b, :, h, :] = (s / s.sum(axis=-1, keepdims=True)) @ v[b, :, g, :]
        return out

    @staticmethod
    def _route(x, Wr, top_k, normalize):
        s = x @ Wr.T
        p = np.exp(s - s.max(axis=-1, keepdims=True))
        p /= p.sum(axis=-1, keepdims=True)
        idx = np.argsort(-p, axis=-1, kind="stable")[..., :top_k]
        w = np.take_along_axis(p, idx, axis=-1)
        if normalize:
            w = w / w.sum(axis=-1, keepdims=True)
        return w, idx

    @staticmethod
    def _swiglu(z):
        F = z.shape[-1] // 2
        g = z[..., :F]
        return g / (1.0 + np.exp(-g)) * z[..., F:]

    def _stacked(self, ins, at, lv):
        init, h, w, idx = ins
        y = np.array(init, dtype=np.float64)
        for e in range(int(at["experts"])):
            inner = dict(lv)
            inner[at["var"]] = e
            if at.get("fused"):
                u = self._swiglu(h @ self._w(at["gate"], inner).T)
            elif at["act"] == "Act.silu":
                g = h @ self._w(at["gate"], inner).T
                u = g / (1.0 + np.exp(-g)) * (h @ self._w(at["up"], inner).T)
            else:
                raise NotImplementedError(at["act"])
            ffn = u @ self._w(at["down"], inner).T
            y = y + np.sum(np.where(idx == e, w, 0.0), axis=-1, keepdims=True) * ffn
        return y
