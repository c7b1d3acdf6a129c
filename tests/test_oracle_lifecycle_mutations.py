"""Plant plausible mistakes in copies of the oracle's cache-lifecycle model
(oracle/oracle.py: the page allocator, truncation, rewind, eviction,
reconciliation and swap) and of its Algorithm 2 router, and check that the
lifecycle pins of tests/test_oracle_session.py and the hand-derived routing
trace of tests/test_alg2_routing.py catch every one of them (no GPU).

Each mutation is a text substitution in the module's source; the copy is
executed as a module of its own (sharing the already-loaded C library, whose
RoPE and attention are pinned by tests/test_oracle_mutations.py) and every
session pin runs against it.  A mutation counts as caught when at least one
pin fails or raises.
"""
import inspect
import os
import sys
import types

import pytest

import test_alg2_routing
import test_oracle_session as session_pins

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "oracle.py")

MUTATIONS = {
    # the allocator hands out the largest free id instead of the smallest
    "allocator_largest_free": ("pid = min(self.free)", "pid = max(self.free)"),
    # truncation keeps the suffix's pages
    "truncate_keeps_pages": ("        keep = self._pages_for(ver.length)\n",
                             "        keep = len(ver.pages)\n"),
    # truncation drops one cached segment too many
    "truncate_drops_chunk": ("        ver.segments.pop()\n        keep",
                             "        ver.segments.pop()\n        ver.segments.pop()\n        keep"),
    # a block is placed one position past the cached length
    "positions_off_by_one": ("pos = np.arange(L, L + n, dtype=np.int64)",
                             "pos = np.arange(L + 1, L + n + 1, dtype=np.int64)"),
    # rewind forgets to drop the later segments
    "rewind_keeps_segments": ("        ver.segments = ver.segments[:keep]\n", "        pass\n"),
    # eviction drops the newest chunks instead of the oldest
    "evict_drops_newest": ("        for s in chunks:\n            if dropped >= evict_tokens:",
                           "        for s in reversed(chunks):\n            if dropped >= evict_tokens:"),
    # retained chunks keep their old positions instead of being renumbered
    "rebuild_keeps_old_positions": (
        'Segment("chunk", s.ident, np.arange(start, start + m, dtype=np.int64)))',
        'Segment("chunk", s.ident, s.pos.copy()))'),
    # the full prefix pages are copied to fresh pages instead of shared
    "prefix_pages_not_shared": ("            self.alloc.share(pid)\n            new.pages.append(pid)\n",
                                "            new.pages.append(self.alloc.take())\n"),
    # the rebuilt chunks keep the keys rotated at their old positions
    "rebuild_reuses_old_keys": ("        k_rot = rope(k, pos, self.base)\n        ver.segments[idx]",
                                "        k_rot = rope(k, pos - pos[0] + self.sources_pos0(cid), self.base)\n"
                                "        ver.segments[idx]"),
    # the chunks that arrived during the reconciliation are not caught up
    "catchup_skipped": ("for cid in self.retained_ids + list(self.buffer):",
                        "for cid in self.retained_ids:"),
    # the rebuilt version's pages are reserved before the active version's
    "reservation_order_swapped": (
        "        out = self._add(self.active, \"chunk\", cid, q, k, v)\n",
        "        if was_reconciling:\n"
        "            self._grow(self.pending, self.pending.length + q.shape[0])\n"
        "        out = self._add(self.active, \"chunk\", cid, q, k, v)\n"),
    # the swap keeps the old version's pages referenced
    "swap_leaks_old_pages": ("        for pid in old.pages:\n            self.alloc.release(pid)\n"
                             "        self.active = self.pending",
                             "        self.active = self.pending"),
}

# "rebuild_reuses_old_keys" needs each chunk's original first position: the
# copy records it when the chunk is appended.
_EXTRA = {
    "rebuild_reuses_old_keys": (
        "        was_reconciling = self.is_reconciling\n",
        "        was_reconciling = self.is_reconciling\n"
        "        self.__dict__.setdefault('_pos0', {})[cid] = self.active.length\n"),
}
_HELPER = '''

def _sources_pos0(self, cid):
    return self._pos0[cid]


OracleCSR.sources_pos0 = _sources_pos0
'''


ROUTER_MUTATIONS = {
    # the swap does not exchange the primary and secondary resources
    "router_no_resource_exchange": (
        "            self.primary, self.secondary = self.secondary, self.primary\n", ""),
    # the bridge condition is off by one version (queries of the rebuilt
    # version that must be bridged are swapped in too early)
    "router_bridge_condition_shifted": ("            if k_t > self.k_ready:",
                                        "            if k_t > self.k_ready - 1:"),
    # the eviction cursor is not advanced after a bridged query
    "router_cursor_not_advanced": ("                self.j_eps = j_t\n                return \"bridge\"",
                                   "                return \"bridge\""),
    # the cursor is taken from whichever query comes first after the eviction
    # (the active version's own length included)
    "router_cursor_set_by_any_query": ("        j_t = len(x_static)\n",
                                       "        j_t = len(x_static)\n"
                                       "        if self.j_eps is None:\n            self.j_eps = j_eps_t\n"),
    # a bridged query does not extend the reconciliation state
    "router_bridge_drops_recon_extension": ("                self.x_recon = self.x_recon + delta\n", ""),
    # a bridged chunk is not buffered for the catch-up
    "router_bridge_not_buffered": ("                self.buffer.append(delta)\n", ""),
    # stragglers while reconciling go to the secondary (the cache being rebuilt)
    "router_straggler_to_secondary": (
        '                return "straggler_primary", self.primary, self.x_recon + x_dyn',
        '                return "straggler_primary", self.secondary, self.x_recon + x_dyn'),
    # stragglers while reconciling keep their own stale static state
    "router_straggler_not_stitched": (
        '                return "straggler_primary", self.primary, self.x_recon + x_dyn',
        '                return "straggler_primary", self.primary, x_static + x_dyn'),
    # case 3 reached by falling through instead of by k_t < k
    "router_case3_unguarded": ("        if k_t < self.k:\n", "        if True:\n"),
    # Reconcile never authorises the swap
    "router_no_k_ready": ("        self.k_ready = k_target\n", "        pass\n"),
    # a continuation does not advance the active length
    "router_continuation_keeps_j": ("                self.x_recon = x_static\n                self.j = j_t\n",
                                    "                self.x_recon = x_static\n"),
    # the catch-up hands the buffer to the secondary but keeps it buffered
    "router_catch_up_keeps_buffer": ("        taken = \"\".join(self.buffer)\n        self.buffer = []\n",
                                     "        taken = \"\".join(self.buffer)\n"),
}


def _pins():
    return [(name, fn) for name, fn in inspect.getmembers(session_pins, inspect.isfunction)
            if name.startswith("test_")]


def _run_pin(fn, mod):
    params = inspect.signature(fn).parameters
    if "prefix_len" in params:
        for prefix_len in (32, 37):
            fn(mod, prefix_len)
    else:
        fn(mod)


def _mutant(oracle_mod, name):
    old, new = {**MUTATIONS, **ROUTER_MUTATIONS}[name]
    text = open(SRC).read()
    assert text.count(old) == 1, f"mutation anchor for {name} not found exactly once"
    text = text.replace(old, new)
    if name in _EXTRA:
        a, b = _EXTRA[name]
        assert text.count(a) == 1
        text = text.replace(a, b) + _HELPER
    return _load(text, "oracle.oracle_mutant_" + name, oracle_mod)


def _load(text, modname, oracle_mod):
    """Execute `text` as a module of the oracle package (registered while it
    is built: dataclasses look their module up)."""
    mod = types.ModuleType(modname)
    mod.__file__ = SRC
    mod.__package__ = "oracle"
    sys.modules[modname] = mod
    try:
        exec(compile(text, SRC, "exec"), mod.__dict__)
    finally:
        del sys.modules[modname]
    mod._LIB = oracle_mod._lib()   # the pinned C routines
    return mod


def test_unmutated_copy_passes_every_pin(oracle_mod):
    """The harness itself: an unmodified copy passes all lifecycle pins."""
    mod = _load(open(SRC).read(), "oracle.oracle_copy", oracle_mod)
    for _, fn in _pins():
        _run_pin(fn, mod)


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_lifecycle_mistake_is_caught(oracle_mod, name):
    mod = _mutant(oracle_mod, name)
    caught = []
    for pin_name, fn in _pins():
        try:
            _run_pin(fn, mod)
        except Exception as e:  # noqa: BLE001 (an exception or a failed assert: caught)
            caught.append((pin_name, type(e).__name__))
    assert caught, f"no lifecycle pin caught the planted mistake {name}"


def test_unmutated_copy_passes_the_routing_trace(oracle_mod):
    test_alg2_routing.run_hand_trace(_load(open(SRC).read(), "oracle.oracle_copy_r", oracle_mod))


@pytest.mark.parametrize("name", sorted(ROUTER_MUTATIONS))
def test_planted_router_mistake_is_caught(oracle_mod, name):
    mod = _mutant(oracle_mod, name)
    with pytest.raises(AssertionError):
        test_alg2_routing.run_hand_trace(mod)
