"""KV page pool accounting (oracle side).

The paper's engine pre-allocates the KV cache to the largest size that fits
and runs a rejection round each time the accelerator is about to run out of
memory (Section 4.2; Section 5, "Setup").  The paper fixes no page size or
allocation order; the reading implemented here (and by the GPU pool) is:

  * a page holds ``page_tokens`` (16) consecutive positions of one sequence,
    all layers, K and V;  pool pages = floor(pool_bytes / (16 * kv_bytes_per_token));
  * the free list is a LIFO stack initialised with ids 0..n-1 in ascending
    order, so the first pop returns n-1;
  * full prompt pages (floor(P / 16)) are popped once and shared by every
    candidate; a non-empty prompt tail (P mod 16 positions) gets one private
    page per candidate, popped in ascending candidate id;
  * at a decode step every live candidate whose next position starts a page
    pops one page, in ascending candidate id;
  * pages are released in ascending (candidate id, page index) order and
    pushed in that order, so the next pop returns the last one released.

Pinned in tests/test_oracle_pool.py (closed-form first trigger step for
uniform lengths; LIFO order).
"""


class PagePool:
    def __init__(self, n_pages: int):
        self.n_pages = n_pages
        self.stack = list(range(n_pages))      # top of stack = end of list

    @property
    def n_free(self) -> int:
        return len(self.stack)

    def pop(self) -> int:
        if not self.stack:
            raise MemoryError("KV page pool exhausted")
        return self.stack.pop()

    def push(self, pages):
        self.stack.extend(pages)


def pool_pages(pool_bytes: int, kv_bytes_per_token: int, page_tokens: int = 16) -> int:
    return pool_bytes // (page_tokens * kv_bytes_per_token)


def private_pages_full(P: int, max_new: int, page_tokens: int = 16) -> int:
    """Private pages a candidate holds when it reaches max_new tokens.

    KV is stored for positions 0 .. P + max_new - 2 (the last sampled token is
    never fed back)."""
    last = P + max_new - 2
    return last // page_tokens + 1 - P // page_tokens


def auto_b_init(n_pages: int, P: int, tau_min: int, n_max: int, page_tokens: int = 16) -> int:
    """Initial batch size of Algorithm 1's first step ("based on the GPU memory capacity and the prompt
    length"), read as: the largest N <= n_max whose candidates can all generate tau_min tokens before the pool
    runs out, i.e. before the first memory-triggered round.  The prompt's full pages are shared; each candidate
    then holds private_pages_full(P, tau_min) pages.  0 when not even one candidate fits."""
    avail = n_pages - P // page_tokens
    per = private_pages_full(P, tau_min, page_tokens)
    if avail < 0:
        return 0
    if per == 0:
        return n_max
    return min(n_max, avail // per)
