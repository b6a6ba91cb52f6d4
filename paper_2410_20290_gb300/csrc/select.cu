// Rejection rounds and KV page accounting, entirely on the device.
//
// Section 4.2: the partial rewards R_partial of the round batch (Eq. partial.reward.set), the
// cut-off r_cut = q_alpha(R_partial) (Eq. cutoff.threshold), the accepted set
// I_accepted = {k : r_k >= r_cut} (Eq. accepted.set); completed candidates join I; the batch
// shrinks to the accepted live candidates (Algorithm 1).  q_alpha is read as the order
// statistic of index k = min(floor(alpha b), b - 1) (0-based, ascending), found by a 4-pass
// 8-bit radix select over order-preserving uint32 keys; ties at r_cut are all accepted.
//
// Page accounting (the pre-allocated KV cache of the Section 5 engine, paged): a LIFO free stack
// initialised 0..n-1 (top = n-1); pages are taken in ascending candidate id and released in
// ascending (candidate id, page index) order, via block-wide exclusive scans, so the page tables
// and the free stack are a deterministic function of the inputs.
//
// Batches are at most 4096 candidates, so each kernel here is one 1024-thread block, with each
// thread owning 4 consecutive batch slots (scan order == slot order == ascending id).
#include "common.cuh"

namespace sr {

namespace {

constexpr int CT = 1024;  // control-kernel block size
constexpr int PER = MAX_BATCH / CT;

__device__ __forceinline__ int priv_pages(int P, int n_sh, int len) {
  // KV positions 0 .. P + len - 2 are stored; pages n_sh .. (P + len - 2) / 16 are private
  const int last = P + len - 2;
  const int c = last / PAGE + 1 - n_sh;
  return (last < 0 || c < 0) ? 0 : c;
}

__device__ void note_peak(int* ctrl) {
  const int used = ctrl[C_NPOOL] - ctrl[C_TOP];
  if (used > ctrl[C_PEAK]) ctrl[C_PEAK] = used;
}

__global__ void k_pool_init(int* free_stack, int n_pages, int* ctrl) {
  pdl_entry();
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n_pages; i += gridDim.x * blockDim.x) free_stack[i] = i;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    for (int c = 0; c < C_N; ++c) ctrl[c] = 0;
    ctrl[C_TOP] = n_pages;
    ctrl[C_NPOOL] = n_pages;
  }
}

// Pop the n_sh shared prompt pages into prompt_row; the template page (outside the stack) holds
// the prompt tail until it is copied into each candidate's first private page.
__global__ void k_prompt_pages(int* free_stack, int* ctrl, int n_sh, int has_tail, int template_page,
                               int* prompt_row) {
  pdl_entry();
  if (threadIdx.x != 0) return;
  int top = ctrl[C_TOP];
  if (top < n_sh) {
    ctrl[C_ERR] = E_POOL_EMPTY;
    return;
  }
  for (int j = 0; j < n_sh; ++j) prompt_row[j] = free_stack[top - 1 - j];
  top -= n_sh;
  if (has_tail) prompt_row[n_sh] = template_page;
  ctrl[C_TOP] = top;
  note_peak(ctrl);
}

// Admit candidates start .. start+count-1: shared prompt pages, one tail page each (ascending id).
__global__ void __launch_bounds__(CT) k_admit(int start, int count, int n_sh, int has_tail,
                                              const int* __restrict__ prompt_row, int* pt, int max_pages, int* len,
                                              int* status, int* live, int* rset, const int* free_stack, int* ctrl,
                                              int* tail_dst) {
  pdl_entry();
  const int top = ctrl[C_TOP];
  if (has_tail && top < count) {
    if (threadIdx.x == 0) ctrl[C_ERR] = E_POOL_EMPTY;
    return;
  }
  for (int i = threadIdx.x; i < count; i += CT) {
    const int id = start + i;
    int* row = pt + (size_t)id * max_pages;
    for (int j = 0; j < n_sh; ++j) row[j] = prompt_row[j];
    if (has_tail) {
      const int page = free_stack[top - 1 - i];
      row[n_sh] = page;
      tail_dst[i] = page;
    }
    len[id] = 0;
    status[id] = ST_LIVE;
    live[i] = id;
    rset[i] = id;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (has_tail) ctrl[C_TOP] = top - count;
    ctrl[C_NLIVE] = count;
    ctrl[C_NRSET] = count;
    note_peak(ctrl);
  }
}

// Before a decode step: every live candidate whose next position (P + len - 1) opens a page pops
// one, in slot order; also gathers the step's input token and position per slot.
__global__ void __launch_bounds__(CT) k_step_begin(int P, const int* __restrict__ live, int* ctrl, const int* len,
                                                   int* pt, int max_pages, const int* free_stack,
                                                   const int* __restrict__ tok, int max_new, int* tok_in,
                                                   int* pos_in, int* kv_len) {
  pdl_entry();
  __shared__ int tmp[40];
  __shared__ int s_total;
  const int n = ctrl[C_NLIVE];
  const int top = ctrl[C_TOP];
  int need[PER], ids[PER], pos[PER];
  int mine = 0;
#pragma unroll
  for (int j = 0; j < PER; ++j) {
    const int s = threadIdx.x * PER + j;
    need[j] = 0;
    if (s < n) {
      ids[j] = live[s];
      const int g = len[ids[j]];
      pos[j] = P + g - 1;
      need[j] = (pos[j] % PAGE == 0) ? 1 : 0;
      tok_in[s] = tok[(size_t)ids[j] * max_new + g - 1];
      pos_in[s] = pos[j];
      kv_len[s] = pos[j] + 1;
    }
    mine += need[j];
  }
  int total;
  int off = block_excl_scan(mine, tmp, &total);
  if (threadIdx.x == 0) s_total = total;
  __syncthreads();
  if (s_total > top) {
    if (threadIdx.x == 0) ctrl[C_ERR] = E_POOL_EMPTY;
    return;
  }
#pragma unroll
  for (int j = 0; j < PER; ++j) {
    const int s = threadIdx.x * PER + j;
    if (s < n && need[j]) {
      pt[(size_t)ids[j] * max_pages + pos[j] / PAGE] = free_stack[top - 1 - off];
      ++off;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    ctrl[C_TOP] = top - s_total;
    note_peak(ctrl);
  }
}

// After sampling: candidates that completed this step release their private pages (ascending
// id, ascending page index) and leave the live list (stable compaction).
__global__ void __launch_bounds__(CT) k_step_end(int P, int n_sh, int* live, int* ctrl, const int* len,
                                                 const int* status, const int* pt, int max_pages, int* free_stack) {
  pdl_entry();
  __shared__ int tmp[40];
  __shared__ int s_rel, s_keep;
  const int n = ctrl[C_NLIVE];
  const int top = ctrl[C_TOP];
  int ids[PER], cnt[PER], keep[PER];
  int rel = 0, kept = 0;
#pragma unroll
  for (int j = 0; j < PER; ++j) {
    const int s = threadIdx.x * PER + j;
    cnt[j] = 0;
    keep[j] = 0;
    if (s < n) {
      ids[j] = live[s];
      const bool fin = status[ids[j]] == ST_PENDING;
      cnt[j] = fin ? priv_pages(P, n_sh, len[ids[j]]) : 0;
      keep[j] = fin ? 0 : 1;
    }
    rel += cnt[j];
    kept += keep[j];
  }
  int total_rel, total_keep;
  int off = block_excl_scan(rel, tmp, &total_rel);
  if (threadIdx.x == 0) s_rel = total_rel;
  int koff = block_excl_scan(kept, tmp, &total_keep);
  if (threadIdx.x == 0) s_keep = total_keep;
  __syncthreads();  // every slot id is in registers before the list is rewritten
#pragma unroll
  for (int j = 0; j < PER; ++j) {
    const int s = threadIdx.x * PER + j;
    if (s >= n) continue;
    const int* row = pt + (size_t)ids[j] * max_pages + n_sh;
    for (int q = 0; q < cnt[j]; ++q) free_stack[top + off + q] = row[q];
    off += cnt[j];
    if (keep[j]) live[koff++] = ids[j];
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    ctrl[C_TOP] = top + s_rel;
    ctrl[C_NLIVE] = s_keep;
  }
}

// k-th smallest (0-based) of keys[0..n) by 4 passes of 8-bit radix select; block-uniform result.
__device__ uint32_t radix_select(const uint32_t* keys, int n, int k, int* hist, int* sh) {
  uint32_t prefix = 0, mask = 0;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
      const uint32_t key = keys[i];
      if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int c = 0, d = 0;
      for (; d < 255; ++d) {
        if (c + hist[d] > k) break;
        c += hist[d];
      }
      sh[0] = d;
      sh[1] = k - c;
    }
    __syncthreads();
    prefix |= (uint32_t)sh[0] << shift;
    mask |= 255u << shift;
    k = sh[1];
    __syncthreads();
  }
  return prefix;
}

__device__ __forceinline__ int cut_index(float alpha, int b) {
  long long k = (long long)floor((double)alpha * (double)b);
  if (k < 0) k = 0;
  if (k > b - 1) k = b - 1;
  return (int)k;
}

__global__ void __launch_bounds__(CT) k_rcut(const float* __restrict__ rewards, int b, float alpha, int k_override,
                                             float* r_cut_out, uint8_t* mask_out) {
  pdl_entry();
  __shared__ uint32_t keys[MAX_BATCH];
  __shared__ int hist[256];
  __shared__ int sh[4];
  for (int i = threadIdx.x; i < b; i += CT) keys[i] = float_key(rewards[i]);
  __syncthreads();
  const int k = k_override >= 0 ? min(k_override, b - 1) : cut_index(alpha, b);
  const uint32_t kc = radix_select(keys, b, k, hist, sh);
  for (int i = threadIdx.x; i < b; i += CT) mask_out[i] = keys[i] >= kc ? 1 : 0;
  if (threadIdx.x == 0) *r_cut_out = key_float(kc);
}

// One rejection round over the round batch rset[0..b) with partial rewards rewards[0..b).
// pool_need: the next decode step needs a page for every live candidate (memory trigger), in
// which case k is raised, if needed, to the smallest index whose rejections free enough pages.
__global__ void __launch_bounds__(CT) k_round(int P, int n_sh, float alpha, int pool_need,
                                              const float* __restrict__ rewards, int* rset, int* live, int* ctrl,
                                              float* ctrlf, int* status, const int* len, float* reward_final,
                                              const int* pt, int max_pages, int* free_stack, uint8_t* mask_out) {
  pdl_entry();
  __shared__ uint32_t keys[MAX_BATCH];
  __shared__ int hist[256];
  __shared__ int sh[4];
  __shared__ int tmp[40];
  __shared__ int s_a, s_b;
  const int b = ctrl[C_NRSET];
  const int top = ctrl[C_TOP];
  for (int i = threadIdx.x; i < b; i += CT) keys[i] = float_key(rewards[i]);
  __syncthreads();
  const int k0 = cut_index(alpha, b);
  int k = k0;
  uint32_t kc = radix_select(keys, b, k0, hist, sh);
  if (pool_need) {
    // cond(k): live accepted <= free pages + pages released by live rejected
    auto cond = [&](uint32_t kcut) -> bool {
      int acc = 0, freed = 0;
      for (int i = threadIdx.x; i < b; i += CT) {
        const int id = rset[i];
        if (status[id] != ST_LIVE) continue;
        if (keys[i] >= kcut) acc += 1;
        else freed += priv_pages(P, n_sh, len[id]);
      }
      int ta, tf;
      block_excl_scan(acc, tmp, &ta);
      if (threadIdx.x == 0) s_a = ta;
      block_excl_scan(freed, tmp, &tf);
      if (threadIdx.x == 0) s_b = tf;
      __syncthreads();
      const bool ok = s_a <= top + s_b;
      __syncthreads();
      return ok;
    };
    if (!cond(kc)) {
      int lo = k0, hi = b - 1;
      const uint32_t k_hi = radix_select(keys, b, hi, hist, sh);
      if (!cond(k_hi)) {
        k = hi;
        kc = k_hi;
      } else {
        uint32_t kc_hi = k_hi;
        while (hi - lo > 1) {
          const int mid = (lo + hi) / 2;
          const uint32_t kmid = radix_select(keys, b, mid, hist, sh);
          if (cond(kmid)) hi = mid, kc_hi = kmid;
          else lo = mid;
        }
        k = hi;
        kc = kc_hi;
      }
    }
  }
  // apply: completed -> I with their reward; rejected live release pages; accepted live survive
  int ids[PER], cnt[PER], keep[PER];
  int rel = 0, kept = 0, nacc = 0;
#pragma unroll
  for (int j = 0; j < PER; ++j) {
    const int s = threadIdx.x * PER + j;
    cnt[j] = 0;
    keep[j] = 0;
    if (s < b) {
      ids[j] = rset[s];
      const bool acc = keys[s] >= kc;
      if (mask_out) mask_out[s] = acc ? 1 : 0;
      nacc += acc ? 1 : 0;
      const int st = status[ids[j]];
      if (st == ST_PENDING) {
        status[ids[j]] = ST_DONE;
        reward_final[ids[j]] = rewards[s];
      } else if (st == ST_LIVE) {
        if (acc) keep[j] = 1;
        else {
          status[ids[j]] = ST_REJECTED;
          cnt[j] = priv_pages(P, n_sh, len[ids[j]]);
        }
      }
    }
    rel += cnt[j];
    kept += keep[j];
  }
  int total_rel, total_keep, total_acc;
  int off = block_excl_scan(rel, tmp, &total_rel);
  if (threadIdx.x == 0) s_a = total_rel;
  int koff = block_excl_scan(kept, tmp, &total_keep);
  if (threadIdx.x == 0) s_b = total_keep;
  block_excl_scan(nacc, tmp, &total_acc);
  __syncthreads();
#pragma unroll
  for (int j = 0; j < PER; ++j) {
    const int s = threadIdx.x * PER + j;
    if (s >= b) continue;
    const int* row = pt + (size_t)ids[j] * max_pages + n_sh;
    for (int q = 0; q < cnt[j]; ++q) free_stack[top + off + q] = row[q];
    off += cnt[j];
    if (keep[j]) {
      rset[koff] = ids[j];
      live[koff] = ids[j];
      ++koff;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    ctrl[C_TOP] = top + s_a;
    ctrl[C_NLIVE] = s_b;
    ctrl[C_NRSET] = s_b;
    ctrl[C_K] = k;
    ctrl[C_KRAISED] = (k != k0) ? 1 : 0;
    ctrl[C_NACC] = total_acc;
    ctrlf[0] = key_float(kc);
  }
}

// Final scores of completed candidates not yet scored: ids[j] -> DONE with r[j].
__global__ void k_mark_done(const int* ids, const float* r, int n, int* status, float* reward_final) {
  pdl_entry();
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < n; j += gridDim.x * blockDim.x) {
    status[ids[j]] = ST_DONE;
    reward_final[ids[j]] = r[j];
  }
}

// Eq. output.SBoN: k* = argmax over I (status DONE) of the final reward, ties to the lowest id;
// copy Y_{k*} to the outputs.
__global__ void __launch_bounds__(CT) k_final(int N, const int* status, const float* reward_final, const int* tok,
                                              int max_new, const int* len, int* out_tokens, int* out_len,
                                              float* out_score, int* ctrl) {
  pdl_entry();
  __shared__ unsigned long long best_s;
  if (threadIdx.x == 0) best_s = 0ull;
  __syncthreads();
  unsigned long long best = 0ull;  // (key + 1) << 32 | ~id : larger is better, lower id wins ties
  for (int i = threadIdx.x; i < N; i += CT) {
    if (status[i] != ST_DONE) continue;
    const unsigned long long v =
        ((unsigned long long)float_key(reward_final[i]) + 1ull) << 32 | (unsigned long long)(0xFFFFFFFFu - (uint32_t)i);
    if (v > best) best = v;
  }
  atomicMax(&best_s, best);
  __syncthreads();
  if (best_s == 0ull) {
    if (threadIdx.x == 0) {
      ctrl[C_ERR] = E_STATE;
      ctrl[C_BEST] = -1;
      *out_len = 0;
    }
    return;
  }
  const int id = (int)(0xFFFFFFFFu - (uint32_t)(best_s & 0xFFFFFFFFull));
  const int L = len[id];
  for (int t = threadIdx.x; t < L; t += CT) out_tokens[t] = tok[(size_t)id * max_new + t];
  if (threadIdx.x == 0) {
    *out_len = L;
    *out_score = reward_final[id];
    ctrl[C_BEST] = id;
  }
}

}  // namespace

// ---- launchers used by the runtime ----
sr_status ctl_pool_init(int* free_stack, int n_pages, int* ctrl, cudaStream_t st) {
  launch_k(k_pool_init, (n_pages + 1023) / 1024 > 0 ? (n_pages + 1023) / 1024 : 1, 1024, 0, st, free_stack, n_pages, ctrl);
  SR_LAUNCH();
  return SR_OK;
}
sr_status ctl_prompt_pages(int* free_stack, int* ctrl, int n_sh, int has_tail, int template_page, int* prompt_row,
                           cudaStream_t st) {
  launch_k(k_prompt_pages, 1, 32, 0, st, free_stack, ctrl, n_sh, has_tail, template_page, prompt_row);
  SR_LAUNCH();
  return SR_OK;
}
sr_status ctl_admit(int start, int count, int n_sh, int has_tail, const int* prompt_row, int* pt, int max_pages,
                    int* len, int* status, int* live, int* rset, const int* free_stack, int* ctrl, int* tail_dst,
                    cudaStream_t st) {
  launch_k(k_admit, 1, CT, 0, st, start, count, n_sh, has_tail, prompt_row, pt, max_pages, len, status, live, rset,
                            free_stack, ctrl, tail_dst);
  SR_LAUNCH();
  return SR_OK;
}
sr_status ctl_step_begin(int P, const int* live, int* ctrl, const int* len, int* pt, int max_pages,
                         const int* free_stack, const int* tok, int max_new, int* tok_in, int* pos_in, int* kv_len,
                         cudaStream_t st) {
  launch_k(k_step_begin, 1, CT, 0, st, P, live, ctrl, len, pt, max_pages, free_stack, tok, max_new, tok_in, pos_in,
                                 kv_len);
  SR_LAUNCH();
  return SR_OK;
}
sr_status ctl_step_end(int P, int n_sh, int* live, int* ctrl, const int* len, const int* status, const int* pt,
                       int max_pages, int* free_stack, cudaStream_t st) {
  launch_k(k_step_end, 1, CT, 0, st, P, n_sh, live, ctrl, len, status, pt, max_pages, free_stack);
  SR_LAUNCH();
  return SR_OK;
}
sr_status ctl_round(int P, int n_sh, float alpha, int pool_need, const float* rewards, int* rset, int* live,
                    int* ctrl, float* ctrlf, int* status, const int* len, float* reward_final, const int* pt,
                    int max_pages, int* free_stack, uint8_t* mask_out, cudaStream_t st) {
  launch_k(k_round, 1, CT, 0, st, P, n_sh, alpha, pool_need, rewards, rset, live, ctrl, ctrlf, status, len, reward_final,
                            pt, max_pages, free_stack, mask_out);
  SR_LAUNCH();
  return SR_OK;
}
sr_status ctl_mark_done(const int* ids, const float* r, int n, int* status, float* reward_final, cudaStream_t st) {
  if (n == 0) return SR_OK;
  launch_k(k_mark_done, (n + 255) / 256, 256, 0, st, ids, r, n, status, reward_final);
  SR_LAUNCH();
  return SR_OK;
}
sr_status ctl_final(int N, const int* status, const float* reward_final, const int* tok, int max_new, const int* len,
                    int* out_tokens, int* out_len, float* out_score, int* ctrl, cudaStream_t st) {
  launch_k(k_final, 1, CT, 0, st, N, status, reward_final, tok, max_new, len, out_tokens, out_len, out_score, ctrl);
  SR_LAUNCH();
  return SR_OK;
}

sr_status launch_rcut(const float* rewards, int b, float alpha, int k_override, float* r_cut_out, uint8_t* mask_out,
                      cudaStream_t st) {
  if (b <= 0 || b > MAX_BATCH) return set_err(SR_ERR_INVALID_ARG, "rcut: b must be in [1, %d]", MAX_BATCH);
  launch_k(k_rcut, 1, CT, 0, st, rewards, b, alpha, k_override, r_cut_out, mask_out);
  SR_LAUNCH();
  return SR_OK;
}

}  // namespace sr
