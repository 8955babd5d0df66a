"""Axon-subset front end: parse a decoder written in (a subset of) the Axon
language, build its Graph IR, and lower it onto this library's fused GB300
kernels (Sec. "The Axon Language"; Sec. "The Axon Compiler", the three
phases). Host-side Python; the model it describes runs entirely in the
CUDA library.

    mod = parse_module(text)                  # syntax.py
    g = build_graph(mod, config)              # graph.py: inlining, paths, loops
    stack_experts(g)                          # rewrite.py: loops over experts -> stacked experts
    low = lower_decoder(g)                    # lower.py: shape + checkpoint names (runs the rewrite too)
    model = create_model(low, checkpoint, max_batch=..., max_context=...)
"""
from .graph import AxonGraphError, Graph, Node, Ref, build_graph, dump
from .lower import LoweredDecoder, LoweringError, lower_decoder
from .rewrite import stack_experts
from .syntax import AxonSyntaxError, parse_module


def compile_decoder(text: str, config: dict | None = None) -> LoweredDecoder:
    """Parse, build and lower a module in one call."""
    return lower_decoder(build_graph(parse_module(text), config), config)


def create_model(lowered: LoweredDecoder, checkpoint: dict, max_batch: int, max_context: int, stream=None,
                 **config_kw):
    """axon_model_create for a lowered module: `checkpoint` maps the
    module's parameter paths (+ ".weight" / ".bias") to tensors; extra
    keywords go to make_config (kv_layout, precision, ...)."""
    import paper_2608_19889_gb300 as ax
    cfg = ax.make_config(lowered.shape, max_batch, max_context, **config_kw)
    return ax.axon_model_create(cfg, lowered.library_weights(checkpoint), stream=stream)


__all__ = ["AxonGraphError", "AxonSyntaxError", "Graph", "LoweredDecoder", "LoweringError", "Node", "Ref",
           "build_graph", "compile_decoder", "create_model", "dump", "lower_decoder", "parse_module",
           "stack_experts"]
