"""Lexer and parser for a subset of the Axon surface language.

The subset covers what a decoder definition needs (Sec. "The Axon Language":
values, symbolic-dimension types, Haskell-style syntax; appendix
"Operations" paragraphs and the grammar figure):

  * module items: pragmas ``{-# KEY value #-}``, ``import M`` / ``import M (a, b)``,
    ``export a b``, type aliases ``type T[x] = type`` and signatures
    ``name[@scope] :: type`` (both kept as text: types are not checked),
    constants ``NAME <- expr``, definitions ``name[@scope] p1 p2 = expr`` or
    ``= do`` + an indented suite (a scope on the signature applies to the
    definition);
  * statements: ``targets <- expr``, ``return e1, e2``, ``yield e1, e2``,
    ``targets <- for[@scope] i <- [a..b) [step=n] [carry (x, y)] do`` + suite,
    ``targets <- scope@path do`` + suite, and the statement-level
    conditional ``if c then do`` + suite ``else do`` + suite;
  * expressions, lowest precedence first: ``::`` ascription (inside
    parentheses), ``>>=`` with a lambda, ``|>`` pipes, ``if/then/else`` and
    ``c ? a : b``, ``or``, ``and``, comparisons, ``+ -``, ``* /``, bare-call
    application ``f a b key=v``, atoms (numbers, strings, true/false/null,
    names with an optional ``@path`` suffix, path literals ``@rel`` and
    ``@@abs``, tuples, lists, parentheses).

Blocks are delimited by indentation; ``--`` starts a comment. The parser
produces the plain AST classes below, which the Graph IR builder
(``graph.py``) consumes.
"""
from __future__ import annotations

import re
from dataclasses import dataclass, field
from typing import List, Optional


class AxonSyntaxError(ValueError):
    def __init__(self, msg, line=0):
        super().__init__(f"line {line}: {msg}" if line else msg)
        self.line = line


# --------------------------------------------------------------------- AST
@dataclass
class Num:
    value: float
    is_int: bool


@dataclass
class Str:
    value: str


@dataclass
class Const:
    value: object  # True, False, None


@dataclass
class PathLit:
    absolute: bool
    path: str


@dataclass
class Name:
    name: str
    path: Optional[str] = None  # f@path: relative path suffix of a callee


@dataclass
class Call:
    fn: Name
    args: list
    kwargs: dict


@dataclass
class BinOp:
    op: str
    left: object
    right: object


@dataclass
class Ternary:
    cond: object
    then: object
    other: object


@dataclass
class TupleE:
    items: list


@dataclass
class ListE:
    items: list


@dataclass
class Ascribe:
    expr: object
    type_text: str


@dataclass
class Lambda:
    param: str
    body: object


@dataclass
class BindS:
    targets: List[str]
    expr: object
    line: int = 0


@dataclass
class ReturnS:
    exprs: list
    line: int = 0


@dataclass
class IfS:
    """Statement-level conditional between two do suites; the taken suite's
    return (or yield) ends the enclosing suite."""
    cond: object
    then: list
    other: list
    line: int = 0


@dataclass
class YieldS:
    exprs: list
    line: int = 0


@dataclass
class ForE:
    scope: Optional[str]
    var: str
    start: object
    stop: object
    lo_closed: bool
    hi_closed: bool
    carry: List[str]
    body: list
    step: object = None  # `step=n` (an expression), None: 1


@dataclass
class ScopeE:
    path: str
    body: list


@dataclass
class DoE:
    body: list


@dataclass
class Definition:
    name: str
    scope: Optional[str]
    params: List[str]
    body: object  # expression, or DoE
    signature: Optional[str] = None
    line: int = 0


@dataclass
class Module:
    pragmas: dict = field(default_factory=dict)
    imports: list = field(default_factory=list)
    constants: list = field(default_factory=list)  # [(name, expr)] in order
    exports: list = field(default_factory=list)  # exported names
    types: dict = field(default_factory=dict)  # alias -> type text
    definitions: dict = field(default_factory=dict)  # name -> Definition
    order: list = field(default_factory=list)  # definition names in source order


# ------------------------------------------------------------------- lexer
@dataclass
class Tok:
    kind: str  # NAME NUM STR PATH OP NEWLINE INDENT DEDENT EOF PRAGMA
    text: str
    line: int
    glued: bool = False  # no whitespace before this token


_OPS = ["{-#", "#-}", ">>=", "<-", "->", "::", "|>", "==", "!=", "<=", ">=", "..", "\\",
        "(", ")", "[", "]", ",", "=", "?", ":", "+", "-", "*", "/", "<", ">", ";"]
_NAME = re.compile(r"[A-Za-z_][A-Za-z0-9_']*(?:\.[A-Za-z_][A-Za-z0-9_']*)*")
_NUM = re.compile(r"[0-9]+(?:\.[0-9]+)?(?:[eE][+-]?[0-9]+)?")
_PATH = re.compile(r"@@?(?:'(?:[^'\\]|\\.)*'|(?:[A-Za-z_{][A-Za-z0-9_{}]*|[0-9]+)(?:\.(?:[A-Za-z_{][A-Za-z0-9_{}]*|[0-9]+))*)")
_STR = re.compile(r'"(?:[^"\\]|\\.)*"')


def tokenize(src: str) -> List[Tok]:
    toks: List[Tok] = []
    indents = [0]
    depth = 0  # bracket nesting: newlines inside brackets are not layout
    lines = src.split("\n")
    for ln, raw in enumerate(lines, 1):
        line = raw.rstrip()
        stripped = line.split("--", 1)[0] if not line.lstrip().startswith("{-#") else line
        if not stripped.strip():
            continue
        if depth == 0:
            ind = len(stripped) - len(stripped.lstrip(" "))
            if "\t" in stripped[:ind + 1]:
                raise AxonSyntaxError("tabs in indentation", ln)
            if ind > indents[-1]:
                indents.append(ind)
                toks.append(Tok("INDENT", "", ln))
            else:
                while ind < indents[-1]:
                    indents.pop()
                    toks.append(Tok("DEDENT", "", ln))
                if ind != indents[-1]:
                    raise AxonSyntaxError("inconsistent indentation", ln)
        i = len(stripped) - len(stripped.lstrip(" "))
        glued = False
        while i < len(stripped):
            c = stripped[i]
            if c == " ":
                i += 1
                glued = False
                continue
            if stripped.startswith("{-#", i):
                end = stripped.find("#-}", i)
                if end < 0:
                    raise AxonSyntaxError("unterminated pragma", ln)
                toks.append(Tok("PRAGMA", stripped[i + 3:end].strip(), ln))
                i = end + 3
                glued = True
                continue
            m = _STR.match(stripped, i)
            if m:
                toks.append(Tok("STR", m.group(0)[1:-1], ln, glued))
                i = m.end()
                glued = True
                continue
            if c == "@":
                m = _PATH.match(stripped, i)
                if not m:
                    raise AxonSyntaxError(f"bad path at {stripped[i:i + 20]!r}", ln)
                toks.append(Tok("PATH", m.group(0), ln, glued))
                i = m.end()
                glued = True
                continue
            m = _NUM.match(stripped, i)
            if m and not (toks and toks[-1].kind == "NAME" and glued):
                toks.append(Tok("NUM", m.group(0), ln, glued))
                i = m.end()
                glued = True
                continue
            m = _NAME.match(stripped, i)
            if m:
                toks.append(Tok("NAME", m.group(0), ln, glued))
                i = m.end()
                glued = True
                continue
            for op in _OPS:
                if stripped.startswith(op, i):
                    toks.append(Tok("OP", op, ln, glued))
                    if op in "([":
                        depth += 1
                    elif op in ")]":
                        depth = max(0, depth - 1)
                    i += len(op)
                    glued = True
                    break
            else:
                raise AxonSyntaxError(f"unexpected character {c!r}", ln)
        if depth == 0:
            toks.append(Tok("NEWLINE", "", ln))
    while len(indents) > 1:
        indents.pop()
        toks.append(Tok("DEDENT", "", len(lines)))
    toks.append(Tok("EOF", "", len(lines)))
    return toks


# ------------------------------------------------------------------ parser
_ATOM_START = {"NUM", "STR", "PATH", "NAME"}
_KEYWORDS = {"do", "return", "yield", "for", "scope", "carry", "if", "then", "else", "and", "or", "import",
             "true", "false", "null", "step"}


class Parser:
    def __init__(self, toks: List[Tok]):
        self.t = toks
        self.i = 0

    # token helpers
    def peek(self, k=0) -> Tok:
        return self.t[min(self.i + k, len(self.t) - 1)]

    def at(self, kind, text=None, k=0) -> bool:
        tok = self.peek(k)
        return tok.kind == kind and (text is None or tok.text == text)

    def eat(self, kind, text=None) -> Tok:
        tok = self.peek()
        if tok.kind != kind or (text is not None and tok.text != text):
            want = text or kind
            raise AxonSyntaxError(f"expected {want!r}, found {tok.text or tok.kind!r}", tok.line)
        self.i += 1
        return tok

    def opt(self, kind, text=None) -> Optional[Tok]:
        if self.at(kind, text):
            return self.eat(kind, text)
        return None

    def skip_newlines(self):
        while self.at("NEWLINE"):
            self.i += 1

    # module
    def module(self) -> Module:
        mod = Module()
        self.skip_newlines()
        while not self.at("EOF"):
            tok = self.peek()
            if tok.kind == "PRAGMA":
                key, _, val = tok.text.partition(" ")
                mod.pragmas[key] = val.strip()
                self.i += 1
            elif tok.kind == "NAME" and tok.text == "import":
                self.i += 1
                name = self.eat("NAME").text
                names = []
                if self.opt("OP", "("):
                    while not self.at("OP", ")"):
                        names.append(self.eat("NAME").text)
                        self.opt("OP", ",")
                    self.eat("OP", ")")
                mod.imports.append((name, names))
            elif tok.kind == "NAME" and tok.text == "export" and self.at("NAME", None, 1):
                self.i += 1
                while self.at("NAME"):
                    mod.exports.append(self.eat("NAME").text)
            elif tok.kind == "NAME" and tok.text == "type" and self.at("NAME", None, 1):
                self.i += 1
                name = self.eat("NAME").text
                parts = []
                while not self.at("NEWLINE") and not self.at("EOF"):
                    parts.append(self.peek().text)
                    self.i += 1
                if not parts or parts[0] not in ("=", "[") or "=" not in parts:
                    raise AxonSyntaxError(f"type alias {name}: expected [params] = type", tok.line)
                mod.types[name] = " ".join(parts)
            elif tok.kind == "NAME" and self.at("OP", "<-", 1):
                name = self.eat("NAME").text
                self.eat("OP", "<-")
                mod.constants.append((name, self.expr()))
            elif tok.kind == "NAME":
                self.definition_or_signature(mod)
            else:
                raise AxonSyntaxError(f"unexpected {tok.text or tok.kind!r} at module level", tok.line)
            # an item ends at a newline, or where an indented suite closed
            if not self.at("EOF") and self.t[self.i - 1].kind != "DEDENT":
                self.eat("NEWLINE")
            self.skip_newlines()
        return mod

    def definition_or_signature(self, mod: Module):
        start = self.eat("NAME")
        scope = None
        if self.at("PATH") and self.peek().glued:
            scope = self.eat("PATH").text.lstrip("@")
        if self.opt("OP", "::"):
            parts = []
            while not self.at("NEWLINE") and not self.at("EOF"):
                parts.append(self.peek().text)
                self.i += 1
            sig = " ".join(parts)
            d = mod.definitions.get(start.text)
            if d is None:
                mod.definitions[start.text] = Definition(start.text, scope, [], None, sig, start.line)
            else:
                d.signature = sig
            return
        params = []
        while self.at("NAME"):
            params.append(self.eat("NAME").text)
        self.eat("OP", "=")
        body = self.expr()
        d = mod.definitions.get(start.text)
        if d is not None and d.body is not None:
            raise AxonSyntaxError(f"definition {start.text} given twice", start.line)
        sig = d.signature if d else None
        if scope is None and d is not None:
            scope = d.scope  # `name@scope :: type` then `name x = ...`
        mod.definitions[start.text] = Definition(start.text, scope, params, body, sig, start.line)
        if start.text not in mod.order:
            mod.order.append(start.text)

    # suites
    def suite(self) -> list:
        """After `do`: an indented block, or inline statements separated by `;`."""
        if self.at("NEWLINE"):
            self.eat("NEWLINE")
            self.eat("INDENT")
            stmts = []
            while not self.at("DEDENT"):
                stmts.append(self.statement())
                while self.opt("OP", ";"):
                    stmts.append(self.statement())
                if not self.at("DEDENT") and self.t[self.i - 1].kind != "DEDENT":
                    self.eat("NEWLINE")
                self.skip_newlines()
            self.eat("DEDENT")
            return stmts
        stmts = [self.statement()]  # inline: `do s1; s2; return e`
        while self.opt("OP", ";"):
            stmts.append(self.statement())
        return stmts

    def statement(self):
        tok = self.peek()
        if tok.kind == "NAME" and tok.text == "return":
            self.i += 1
            return ReturnS(self.expr_list(), tok.line)
        if tok.kind == "NAME" and tok.text == "yield":
            self.i += 1
            return YieldS(self.expr_list(), tok.line)
        if tok.kind == "NAME" and tok.text == "if":
            self.i += 1
            cond = self.expr()
            self.eat("NAME", "then")
            self.eat("NAME", "do")
            then = self.suite()
            self.skip_newlines()
            if not self.at("NAME", "else"):
                raise AxonSyntaxError("a statement-level if needs an else branch", self.peek().line)
            self.eat("NAME", "else")
            self.eat("NAME", "do")
            return IfS(cond, then, self.suite(), tok.line)
        # targets <- ...
        targets = [self.eat("NAME").text]
        while self.opt("OP", ","):
            targets.append(self.eat("NAME").text)
        self.eat("OP", "<-")
        if self.at("NAME", "for"):
            return BindS(targets, self.for_expr(), tok.line)
        if self.at("NAME", "scope"):
            return BindS(targets, self.scope_expr(), tok.line)
        return BindS(targets, self.expr(), tok.line)

    def for_expr(self) -> ForE:
        self.eat("NAME", "for")
        scope = None
        if self.at("PATH") and self.peek().glued:
            scope = self.eat("PATH").text.lstrip("@")
        var = self.eat("NAME").text
        self.eat("OP", "<-")
        lo = self.eat("OP").text
        if lo not in "[(":
            raise AxonSyntaxError("range must start with [ or (", self.peek().line)
        start = self.arith()
        self.eat("OP", "..")
        stop = self.arith()
        hi = self.eat("OP").text
        if hi not in ")]":
            raise AxonSyntaxError("range must end with ) or ]", self.peek().line)
        carry = []
        step = None
        if self.at("NAME", "step"):
            self.i += 1
            self.eat("OP", "=")
            step = self.atom()
        if self.opt("NAME", "carry"):
            self.eat("OP", "(")
            while not self.at("OP", ")"):
                carry.append(self.eat("NAME").text)
                self.opt("OP", ",")
            self.eat("OP", ")")
        self.eat("NAME", "do")
        return ForE(scope, var, start, stop, lo == "[", hi == "]", carry, self.suite(), step)

    def scope_expr(self) -> ScopeE:
        self.eat("NAME", "scope")
        p = self.eat("PATH").text.lstrip("@")
        self.eat("NAME", "do")
        return ScopeE(p, self.suite())

    # expressions
    def expr_list(self) -> list:
        out = [self.expr()]
        while self.opt("OP", ","):
            out.append(self.expr())
        return out

    def expr(self):
        if self.at("NAME", "do"):
            self.i += 1
            return DoE(self.suite())
        e = self.pipe()
        if self.opt("OP", ">>="):
            self.eat("OP", "\\")
            param = self.eat("NAME").text
            self.eat("OP", "->")
            e = Call(Name("__apply"), [Lambda(param, self.expr()), e], {})
        return e

    def pipe(self):
        e = self.ternary()
        while self.opt("OP", "|>"):
            rhs = self.ternary()
            if isinstance(rhs, Name):
                e = Call(rhs, [e], {})
            elif isinstance(rhs, Call):
                e = Call(rhs.fn, [e] + rhs.args, rhs.kwargs)
            else:
                raise AxonSyntaxError("the right side of |> must be a function or call", self.peek().line)
        return e

    def ternary(self):
        if self.opt("NAME", "if"):
            c = self.expr()
            self.eat("NAME", "then")
            a = self.expr()
            self.eat("NAME", "else")
            return Ternary(c, a, self.expr())
        c = self.or_()
        if self.opt("OP", "?"):
            a = self.pipe()
            self.eat("OP", ":")
            return Ternary(c, a, self.pipe())
        return c

    def or_(self):
        e = self.and_()
        while self.opt("NAME", "or"):
            e = BinOp("or", e, self.and_())
        return e

    def and_(self):
        e = self.cmp()
        while self.opt("NAME", "and"):
            e = BinOp("and", e, self.cmp())
        return e

    def cmp(self):
        e = self.arith()
        while self.peek().kind == "OP" and self.peek().text in ("==", "!=", "<=", ">=", "<", ">"):
            op = self.eat("OP").text
            e = BinOp(op, e, self.arith())
        return e

    def arith(self):
        e = self.term()
        while self.peek().kind == "OP" and self.peek().text in ("+", "-"):
            op = self.eat("OP").text
            e = BinOp(op, e, self.term())
        return e

    def term(self):
        e = self.app()
        while self.peek().kind == "OP" and self.peek().text in ("*", "/"):
            op = self.eat("OP").text
            e = BinOp(op, e, self.app())
        return e

    def app(self):
        if self.at("NAME") and self.peek().text not in _KEYWORDS:
            fn = self.callee()
            args, kwargs = [], {}
            while True:
                tok = self.peek()
                if tok.kind == "NAME" and self.at("OP", "=", 1) and tok.text not in _KEYWORDS:
                    self.i += 2
                    kwargs[tok.text] = self.atom()
                elif tok.kind in _ATOM_START and not (tok.kind == "NAME" and tok.text in _KEYWORDS - {
                        "true", "false", "null"}):
                    args.append(self.atom())
                elif tok.kind == "OP" and tok.text in ("(", "["):
                    args.append(self.atom())
                else:
                    break
            if args or kwargs:
                return Call(fn, args, kwargs)
            return fn
        if self.at("OP", "-"):
            self.i += 1
            return BinOp("-", Num(0, True), self.app())
        return self.atom()

    def callee(self) -> Name:
        name = self.eat("NAME").text
        path = None
        if self.at("PATH") and self.peek().glued and not self.peek().text.startswith("@@"):
            path = self.eat("PATH").text[1:]
        elif self.at("PATH") and self.peek().glued:
            path = self.eat("PATH").text  # absolute: keeps its @@
        return Name(name, path)

    def atom(self):
        tok = self.peek()
        if tok.kind == "NUM":
            self.i += 1
            is_int = re.fullmatch(r"[0-9]+", tok.text) is not None
            return Num(int(tok.text) if is_int else float(tok.text), is_int)
        if tok.kind == "STR":
            self.i += 1
            return Str(tok.text)
        if tok.kind == "PATH":
            self.i += 1
            absolute = tok.text.startswith("@@")
            body = tok.text[2:] if absolute else tok.text[1:]
            if body.startswith("'"):
                body = body[1:-1]
            return PathLit(absolute, body)
        if tok.kind == "NAME":
            if tok.text in ("true", "false", "null"):
                self.i += 1
                return Const({"true": True, "false": False, "null": None}[tok.text])
            return self.callee()
        if self.opt("OP", "("):
            if self.opt("OP", ")"):
                return TupleE([])
            e = self.expr()
            if self.opt("OP", "::"):
                parts, depth = [], 0
                while not (depth == 0 and self.at("OP", ")")):
                    t = self.peek()
                    if t.kind == "EOF":
                        raise AxonSyntaxError("unterminated type ascription", t.line)
                    depth += t.text in ("(", "[")
                    depth -= t.text in (")", "]")
                    parts.append(t.text)
                    self.i += 1
                self.eat("OP", ")")
                return Ascribe(e, " ".join(parts))
            if self.at("OP", ","):
                items = [e]
                while self.opt("OP", ","):
                    if self.at("OP", ")"):
                        break
                    items.append(self.expr())
                self.eat("OP", ")")
                return TupleE(items)
            self.eat("OP", ")")
            return e
        if self.opt("OP", "["):
            items = []
            while not self.at("OP", "]"):
                items.append(self.expr())
                if not self.opt("OP", ","):
                    break
            self.eat("OP", "]")
            return ListE(items)
        raise AxonSyntaxError(f"unexpected {tok.text or tok.kind!r}", tok.line)


def parse_module(src: str) -> Module:
    """Parse an Axon module (the subset described in this file's docstring)."""
    return Parser(tokenize(src)).module()
