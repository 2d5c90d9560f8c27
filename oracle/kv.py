"""Plain-Python model of the paged KV-cache maintenance around a verification step.

TEST INFRASTRUCTURE ONLY: only tests/ may use this module.  It shares nothing with the CUDA library.

What it models (Sec. 4.5: PageAttention pages and a prefix cache updated in place; the semantics
are the ones include/wisp_kv.h states): before a step every request gets the pages covering tokens
0 .. c + k, served in request order from the top of a free stack (a request the remaining pool cannot
serve, and every later valid one, gets nothing), and its k + 1 new K/V rows are written at positions
c .. c + k; after acceptance c becomes c + 1 + L (Eq. 2's L) and the pages past the new length among
those the step could use return to the stack in table order.  Written as loops over requests.
"""
from __future__ import annotations

PAGE = 16
OK, BAD_LENGTH, BAD_BLOCK, NO_BLOCKS = 0, 1, 2, 7


def _pages(n_tokens: int) -> int:
    return (n_tokens + PAGE - 1) // PAGE


def reserve_append(tables, free_stack, free_count, ctx, draft, num_blocks, k_new=None, v_new=None,
                   k_cache=None, v_cache=None):
    """Mutates tables (list of lists), free_stack (list), k_cache / v_cache (numpy, [nb, Hkv, 16, D]);
    returns (new free_count, per-request codes)."""
    B = len(draft)
    cap = len(tables[0]) * PAGE if B else 0
    codes = [OK] * B
    F = free_count
    before = 0
    taken = 0
    row = 0
    for r in range(B):
        k, c = int(draft[r]), int(ctx[r])
        bad = OK
        if k < 0:
            bad, k = BAD_LENGTH, 0
        if bad == OK and (c < 0 or c + k + 1 > cap):
            bad = BAD_LENGTH
        need = 0
        if bad == OK:
            for b in range(_pages(c + k + 1)):
                if tables[r][b] < 0:
                    need += 1
                elif tables[r][b] >= num_blocks:
                    bad = BAD_BLOCK
        if bad != OK:
            need = 0
        served = bad == OK and before + need <= F
        codes[r] = bad if bad != OK else (OK if served else NO_BLOCKS)
        if served:
            t = 0
            for b in range(_pages(c + k + 1)):
                if tables[r][b] < 0:
                    tables[r][b] = free_stack[F - 1 - before - t]
                    t += 1
            taken = before + need
            if k_new is not None:
                for j in range(k + 1):
                    pos = c + j
                    page = tables[r][pos // PAGE]
                    k_cache[page, :, pos % PAGE, :] = k_new[row + j]
                    v_cache[page, :, pos % PAGE, :] = v_new[row + j]
        before += need
        row += k + 1
    return F - taken, codes


def commit(tables, free_stack, free_count, ctx, draft, accepted):
    """Mutates tables, free_stack, ctx; returns (new free_count, per-request codes)."""
    B = len(draft)
    cap = len(tables[0]) * PAGE if B else 0
    codes = [OK] * B
    F = free_count
    for r in range(B):
        k, c, L = int(draft[r]), int(ctx[r]), int(accepted[r])
        if k < 0 or c < 0 or L < 0 or L > k or c + k + 1 > cap:
            codes[r] = BAD_LENGTH
            continue
        cnew = c + 1 + L
        for b in range(_pages(cnew), _pages(c + k + 1)):
            if tables[r][b] >= 0:
                if F < len(free_stack):
                    free_stack[F] = tables[r][b]
                else:
                    free_stack.append(tables[r][b])
                F += 1
                tables[r][b] = -1
        ctx[r] = cnew
    return F, codes
