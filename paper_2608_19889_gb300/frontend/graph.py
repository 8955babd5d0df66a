"""Graph IR of an Axon module: the desugaring and graph-building phases.

An entry definition is evaluated symbolically (Sec. "The Axon Compiler",
Phases 1-2): library references resolve through the module's imports,
calls to the module's own definitions are inlined at their call sites
(definition inlining), relative parameter paths (``@q_proj``, ``f@ln``,
``scope@attn``, ``for@layers``) resolve against the lexical scope into
absolute checkpoint paths, configuration reads (``Config.dim @@key``)
become constants, and nested expressions flatten into a sequence of
single-operation nodes in static single assignment form. A ``for`` loop
becomes one ``loop`` node whose body graph is built once, with the loop
variable left symbolic in its paths (``layers.{i}.attn``).

Nodes:
  op      qualified primitive or library operation ("NN.linear",
          "Attention.attention", "add", "mul", "loop", "input", ...)
  inputs  Ref(node, index) values or Python constants
  attrs   keyword arguments (constants)
  path    absolute parameter path of a parameterised operation, or None
"""
from __future__ import annotations

import itertools
from dataclasses import dataclass, field
from typing import Dict, List, Optional

from . import syntax as sx


class AxonGraphError(ValueError):
    pass


@dataclass(frozen=True)
class Ref:
    node: int
    index: int = 0


@dataclass
class Node:
    id: int
    op: str
    inputs: list
    attrs: dict
    path: Optional[str] = None
    n_out: int = 1
    body: Optional["Graph"] = None


@dataclass
class Graph:
    nodes: List[Node] = field(default_factory=list)
    inputs: List[Ref] = field(default_factory=list)
    outputs: list = field(default_factory=list)

    def node(self, ref: Ref) -> Node:
        for n in self.nodes:
            if n.id == ref.node:
                return n
        raise KeyError(ref)


@dataclass
class LoopVar:
    name: str


@dataclass
class PathVal:
    path: str


@dataclass
class Closure:
    param: str
    body: object
    env: dict


_BIN = {"+": "add", "-": "sub", "*": "mul", "/": "div"}


def _const_bin(op, a, b):
    if op == "+":
        return a + b
    if op == "-":
        return a - b
    if op == "*":
        return a * b
    if op == "/":
        return a // b if isinstance(a, int) and isinstance(b, int) and a % b == 0 else a / b
    if op == "==":
        return a == b
    if op == "!=":
        return a != b
    if op == "<":
        return a < b
    if op == ">":
        return a > b
    if op == "<=":
        return a <= b
    if op == ">=":
        return a >= b
    if op == "and":
        return a and b
    if op == "or":
        return a or b
    raise AxonGraphError(f"operator {op}")


def _is_const(v):
    return v is None or isinstance(v, (int, float, bool, str, PathVal, LoopVar))


class Builder:
    """Evaluates an entry definition of a parsed module into a Graph."""

    def __init__(self, mod: sx.Module, config: Optional[dict] = None):
        self.mod = mod
        self.config = dict(config or {})
        self.ids = itertools.count()
        self.graphs: List[Graph] = []
        self.imports: Dict[str, str] = {}
        for m, names in mod.imports:
            for n in names:
                self.imports[n] = f"{m}.{n}"
        self.globals: dict = {}
        self.config_reads: dict = {}
        self.depth = 0
        self.want = 1  # outputs of the call being bound (multi-target binds)

    # graph emission
    @property
    def g(self) -> Graph:
        return self.graphs[-1]

    def emit(self, op, inputs, attrs=None, path=None, n_out=1, body=None):
        n = Node(next(self.ids), op, list(inputs), dict(attrs or {}), path, n_out, body)
        self.g.nodes.append(n)
        if n_out == 1:
            return Ref(n.id, 0)
        return tuple(Ref(n.id, i) for i in range(n_out))

    # paths
    @staticmethod
    def join(prefix, rel):
        return ".".join([p for p in prefix + rel.split(".") if p])

    def resolve_path(self, prefix, text):
        """`@@abs` -> abs; `@rel` (or `rel`) -> prefix.rel."""
        if text.startswith("@@"):
            return text[2:].strip("'")
        return self.join(prefix, text.lstrip("@").strip("'"))

    # entry
    def build(self, entry: Optional[str] = None, n_inputs: Optional[int] = None) -> Graph:
        for name, e in self.mod.constants:
            self.globals[name] = self.eval(e, {}, [])
        if entry is None:
            entry = self.mod.pragmas.get("ENTRY", "").strip('"') or self.mod.order[-1]
        d = self.mod.definitions.get(entry)
        if d is None or d.body is None:
            raise AxonGraphError(f"no definition named {entry!r}")
        self.graphs.append(Graph())
        params = d.params if n_inputs is None else d.params[:n_inputs]
        env = {}
        for i, p in enumerate(d.params):
            if i < len(params):
                r = self.emit("input", [], {"name": p, "index": i})
                self.g.inputs.append(r)
                env[p] = r
            else:
                env[p] = None  # optional arguments not supplied (e.g. no mask, no past cache)
        prefix = d.scope.split(".") if d.scope else []
        out = self.eval(d.body, env, prefix)
        self.g.outputs = list(out) if isinstance(out, tuple) else [out]
        return self.graphs.pop()

    # evaluation
    def eval(self, e, env, prefix):
        if isinstance(e, sx.Num):
            return e.value
        if isinstance(e, sx.Str):
            return e.value
        if isinstance(e, sx.Const):
            return e.value
        if isinstance(e, sx.PathLit):
            return PathVal(e.path if e.absolute else self.join(prefix, e.path))
        if isinstance(e, sx.Name):
            if e.path is None:
                if e.name in env:
                    return env[e.name]
                if e.name in self.globals:
                    return self.globals[e.name]
            # a name that is neither a local nor a constant: a call without
            # arguments (a library value such as a default config read)
            n_out, self.want = self.want, 1
            return self.call(e, [], {}, env, prefix, n_out)
        if isinstance(e, sx.Call):
            # outputs wanted by a multi-target bind apply to this call only
            n_out, self.want = self.want, 1
            if e.fn.name == "__apply":
                lam = self.eval(e.args[0], env, prefix)
                return self.apply_closure(lam, self.eval(e.args[1], env, prefix), prefix)
            args = [self.eval(a, env, prefix) for a in e.args]
            kwargs = {k: self.eval(v, env, prefix) for k, v in e.kwargs.items()}
            return self.call(e.fn, args, kwargs, env, prefix, n_out)
        if isinstance(e, sx.Lambda):
            return Closure(e.param, e.body, dict(env))
        if isinstance(e, sx.BinOp):
            a = self.eval(e.left, env, prefix)
            b = self.eval(e.right, env, prefix)
            if _is_const(a) and _is_const(b):
                return _const_bin(e.op, a, b)
            if e.op not in _BIN:
                raise AxonGraphError(f"operator {e.op} on tensors is not in this subset")
            return self.emit(_BIN[e.op], [a, b])
        if isinstance(e, sx.Ternary):
            c = self.eval(e.cond, env, prefix)
            if not _is_const(c):
                raise AxonGraphError("a branch condition must be known when the graph is built")
            return self.eval(e.then if c else e.other, env, prefix)
        if isinstance(e, sx.TupleE):
            return tuple(self.eval(x, env, prefix) for x in e.items)
        if isinstance(e, sx.ListE):
            return [self.eval(x, env, prefix) for x in e.items]
        if isinstance(e, sx.Ascribe):
            return self.eval(e.expr, env, prefix)
        if isinstance(e, sx.DoE):
            return self.run_suite(e.body, dict(env), prefix)
        if isinstance(e, sx.ScopeE):
            return self.run_suite(e.body, dict(env), prefix + e.path.split("."))
        if isinstance(e, sx.ForE):
            return self.loop(e, env, prefix)
        raise AxonGraphError(f"cannot evaluate {type(e).__name__}")

    def apply_closure(self, lam, arg, prefix):
        if not isinstance(lam, Closure):
            raise AxonGraphError(">>= needs a lambda on its right")
        env = dict(lam.env)
        env[lam.param] = arg
        return self.eval(lam.body, env, prefix)

    def run_suite(self, stmts, env, prefix, yield_ok=False):
        for st in stmts:
            if isinstance(st, sx.ReturnS):
                vals = [self.eval(x, env, prefix) for x in st.exprs]
                return vals[0] if len(vals) == 1 else tuple(vals)
            if isinstance(st, sx.YieldS):
                if not yield_ok:
                    raise AxonGraphError(f"line {st.line}: yield outside a loop body")
                vals = [self.eval(x, env, prefix) for x in st.exprs]
                return ("__yield__", vals)
            if isinstance(st, sx.IfS):
                # only the taken branch is built; its return (or yield) ends this suite
                c = self.eval(st.cond, env, prefix)
                if not _is_const(c):
                    raise AxonGraphError(f"line {st.line}: a branch condition must be known when the graph "
                                         "is built")
                return self.run_suite(st.then if c else st.other, dict(env), prefix, yield_ok)
            if isinstance(st, sx.BindS):
                self.want = len(st.targets)
                v = self.eval(st.expr, env, prefix)
                self.want = 1
                if len(st.targets) == 1:
                    env[st.targets[0]] = v
                else:
                    if not isinstance(v, tuple) or len(v) != len(st.targets):
                        raise AxonGraphError(f"line {st.line}: {len(st.targets)} targets for a value of "
                                             f"{len(v) if isinstance(v, tuple) else 1}")
                    for t, x in zip(st.targets, v):
                        env[t] = x
                continue
            raise AxonGraphError(f"statement {type(st).__name__}")
        raise AxonGraphError("a do-suite must end with return (or yield in a loop body)")

    def loop(self, e: sx.ForE, env, prefix):
        start = self.eval(e.start, env, prefix)
        stop = self.eval(e.stop, env, prefix)
        if not isinstance(start, int) or not isinstance(stop, int):
            raise AxonGraphError("loop bounds must be known when the graph is built")
        lo = start if e.lo_closed else start + 1
        hi = stop + 1 if e.hi_closed else stop
        step = 1 if e.step is None else self.eval(e.step, env, prefix)
        if not isinstance(step, int) or step < 1:
            raise AxonGraphError("a loop step must be a positive integer known when the graph is built")
        init = [env[c] for c in e.carry]
        body = Graph()
        self.graphs.append(body)
        benv = dict(env)
        for i, c in enumerate(e.carry):
            r = self.emit("input", [], {"name": c, "index": i})
            body.inputs.append(r)
            benv[c] = r
        benv[e.var] = LoopVar(e.var)
        bprefix = prefix + (e.scope.split(".") if e.scope else []) + ["{" + e.var + "}"]
        out = self.run_suite(e.body, benv, bprefix, yield_ok=True)
        self.graphs.pop()
        if not (isinstance(out, tuple) and out and out[0] == "__yield__"):
            raise AxonGraphError("a loop body must end with yield")
        body.outputs = out[1]
        if len(body.outputs) != len(e.carry):
            raise AxonGraphError("yield must give one value per carried name")
        refs = self.emit("loop", init, {"var": e.var, "start": lo, "stop": hi, "step": step,
                                         "scope": e.scope or ""}, n_out=len(e.carry), body=body)
        return refs

    def call(self, fn: sx.Name, args, kwargs, env, prefix, n_out=1):
        name = fn.name
        if name in env and isinstance(env[name], Closure):
            if len(args) != 1:
                raise AxonGraphError(f"{name} takes one argument")
            return self.apply_closure(env[name], args[0], prefix)
        d = self.mod.definitions.get(name)
        if d is not None and d.body is not None:
            return self.inline(d, fn, args, kwargs, prefix)
        if name in ("Config.dim", "Config.value", "Config.float"):
            return self.config_read(name, args, kwargs)
        qual = self.imports.get(name, name)
        if "." not in qual:
            raise AxonGraphError(f"unknown function {name!r} (not defined in the module, not imported)")
        path = self.resolve_path(prefix, fn.path) if fn.path else None
        return self.emit(qual, args, kwargs, path=path, n_out=n_out)

    def config_read(self, name, args, kwargs):
        if not args or not isinstance(args[0], PathVal):
            raise AxonGraphError(f"{name} needs a configuration path")
        key = args[0].path
        if key in self.config:
            v = self.config[key]
        elif "default" in kwargs:
            v = kwargs["default"]
        else:
            raise AxonGraphError(f"configuration key {key!r} missing and no default")
        v = int(v) if name == "Config.dim" else v
        self.config_reads[key] = v
        return v

    def inline(self, d: sx.Definition, fn: sx.Name, args, kwargs, prefix):
        self.depth += 1
        if self.depth > 64:
            raise AxonGraphError("definitions nest deeper than 64 (recursion?)")
        env = {}
        for i, p in enumerate(d.params):
            if i < len(args):
                env[p] = args[i]
            elif p in kwargs:
                env[p] = kwargs.pop(p)
            else:
                env[p] = None
        if kwargs:
            raise AxonGraphError(f"{d.name}: unknown keyword arguments {sorted(kwargs)}")
        scope = fn.path if fn.path else d.scope
        if scope and scope.startswith("@@"):
            inner = scope[2:].split(".")
        else:
            inner = prefix + (scope.split(".") if scope else [])
        out = self.eval(d.body, env, inner)
        self.depth -= 1
        return out


def build_graph(mod: sx.Module, config: Optional[dict] = None, entry: Optional[str] = None) -> Graph:
    """Evaluate the module's entry definition (pragma ENTRY, else the last
    definition) into a Graph IR; `config` supplies the configuration values
    read through Config.dim / Config.value."""
    b = Builder(mod, config)
    g = b.build(entry)
    g.config_reads = dict(b.config_reads)  # type: ignore[attr-defined]
    return g


def dump(g: Graph, indent="") -> str:
    """Readable listing of a graph (one node per line, loop bodies nested)."""
    out = []
    for n in g.nodes:
        ins = ", ".join(f"%{x.node}.{x.index}" if isinstance(x, Ref) else repr(x) for x in n.inputs)
        at = " ".join(f"{k}={v!r}" for k, v in n.attrs.items())
        p = f" @@{n.path}" if n.path else ""
        out.append(f"{indent}%{n.id} = {n.op}{p}({ins}) {at}".rstrip())
        if n.body is not None:
            out.append(dump(n.body, indent + "    "))
    outs = ", ".join(f"%{x.node}.{x.index}" if isinstance(x, Ref) else repr(x) for x in g.outputs)
    out.append(f"{indent}return {outs}")
    return "\n".join(out)
