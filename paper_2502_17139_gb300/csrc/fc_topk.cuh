// Block-wide ranking of counted continuations, shared by the datastore
// retrieval and the CACHE search (Section III-A: the top-k most frequent
// continuations; ties by token order).
//
// Input: the occurrences of the match, sorted so that equal continuations
// are adjacent and runs appear in ascending token order, described by head
// flags work[e] = 1 where occurrence e starts a run (e < nocc <= FC_MAX_OCC).
// Output: runs[0..R] the run starts (runs[R] = nocc) and order[0..ks) the
// kept runs ranked by (count descending, run ascending), ks = min(k, R).
//
// Top-k: a histogram of run counts finds the k-th largest count c*; the runs
// above it and the first runs equal to it (in token order) are kept, then
// ranked by counting, for each kept run, the kept runs ahead of it.
#pragma once

#include "fc_common.cuh"

template <int NT>
__device__ __forceinline__ uint32_t block_excl_scan(uint32_t x, uint32_t* total, uint32_t* wsum) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t inc = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    uint32_t y = __shfl_up_sync(0xFFFFFFFFu, inc, o);
    if (lane >= o) inc += y;
  }
  if (lane == 31) wsum[warp] = inc;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t run = 0;
    for (int w = 0; w < NT / 32; ++w) {
      uint32_t c = wsum[w];
      wsum[w] = run;
      run += c;
    }
    *total = run;
  }
  __syncthreads();
  uint32_t r = wsum[warp] + inc - x;
  __syncthreads();
  return r;
}

struct RunsScratch {
  uint32_t n_runs, cstar, n_greater, n_sel, total;
};

// Run starts from head flags: work[e] (e < nocc <= FC_MAX_OCC) is 1 where
// occurrence e starts a run.  Writes runs[0..R] (runs[R] = nocc) and returns
// R.  Ends with the block synchronised.
template <int NT>
__device__ uint32_t runs_from_heads(uint32_t nocc, uint32_t* runs, const uint32_t* work, uint32_t* wsum,
                                    RunsScratch& sc) {
  constexpr int ITEMS = FC_MAX_OCC / NT;
  static_assert(ITEMS * NT == FC_MAX_OCC, "FC_MAX_OCC must be a multiple of the block size");
  const int tid = threadIdx.x;
  uint32_t head[ITEMS];
  uint32_t local = 0;
#pragma unroll
  for (int it = 0; it < ITEMS; ++it) {
    uint32_t e = tid * ITEMS + it;
    head[it] = (e < nocc) ? work[e] : 0u;
    local += head[it];
  }
  uint32_t run_id = block_excl_scan<NT>(local, &sc.total, wsum);
#pragma unroll
  for (int it = 0; it < ITEMS; ++it) {
    uint32_t e = tid * ITEMS + it;
    if (head[it]) runs[run_id] = e;
    run_id += head[it];
  }
  if (tid == 0) {
    runs[sc.total] = nocc;
    sc.n_runs = sc.total;
  }
  __syncthreads();
  return sc.n_runs;
}

// Top-k of R runs given by their starts runs[0..R] (counts runs[r+1] -
// runs[r], between 1 and FC_MAX_OCC), in token order.  Writes order[0..ks),
// the kept runs ranked by (count descending, run ascending), and returns
// ks = min(k, R).  work, sel: scratch.  Ends with the block synchronised.
template <int NT>
__device__ uint32_t topk_runs(uint32_t R, int k, const uint32_t* runs, uint32_t* work, uint32_t* sel,
                              uint32_t* order, uint32_t* wsum, RunsScratch& sc) {
  constexpr int ITEMS = FC_MAX_OCC / NT;
  const int tid = threadIdx.x;
  auto run_count = [&](uint32_t r) { return runs[r + 1] - runs[r]; };

  if (R <= (uint32_t)k) {
    for (uint32_t r = tid; r < R; r += NT) sel[r] = r;
    if (tid == 0) sc.n_sel = R;
  } else {
    // histogram of counts (1..FC_MAX_OCC), bin q = FC_MAX_OCC - count so that
    // a prefix over q counts the runs with a larger count
    for (uint32_t q = tid; q < FC_MAX_OCC; q += NT) work[q] = 0;
    __syncthreads();
    for (uint32_t r = tid; r < R; r += NT) atomicAdd(&work[FC_MAX_OCC - run_count(r)], 1u);
    __syncthreads();
    uint32_t hq[ITEMS];
    uint32_t hsum = 0;
#pragma unroll
    for (int it = 0; it < ITEMS; ++it) {
      hq[it] = work[tid * ITEMS + it];
      hsum += hq[it];
    }
    uint32_t above = block_excl_scan<NT>(hsum, &sc.total, wsum);  // runs with a larger count than this chunk's bins
#pragma unroll
    for (int it = 0; it < ITEMS; ++it) {
      if (above < (uint32_t)k && above + hq[it] >= (uint32_t)k) {  // the k-th largest count lives here
        sc.cstar = FC_MAX_OCC - (tid * ITEMS + it);
        sc.n_greater = above;
      }
      above += hq[it];
    }
    __syncthreads();
    const uint32_t cstar = sc.cstar, room = (uint32_t)k - sc.n_greater;
    // keep: count > c*, or count == c* among the first `room` such runs in token order
    uint32_t fl[ITEMS], eq_local = 0;
#pragma unroll
    for (int it = 0; it < ITEMS; ++it) {
      uint32_t r = tid * ITEMS + it;
      fl[it] = (r < R) ? (run_count(r) > cstar ? 2u : (run_count(r) == cstar ? 1u : 0u)) : 0u;
      eq_local += (fl[it] == 1u);
    }
    uint32_t eq_before = block_excl_scan<NT>(eq_local, &sc.total, wsum);
    uint32_t keep_local = 0;
#pragma unroll
    for (int it = 0; it < ITEMS; ++it) {
      if (fl[it] == 1u) {
        fl[it] = (eq_before < room) ? 2u : 0u;
        ++eq_before;
      }
      keep_local += (fl[it] == 2u);
    }
    uint32_t kept_before = block_excl_scan<NT>(keep_local, &sc.total, wsum);
#pragma unroll
    for (int it = 0; it < ITEMS; ++it) {
      if (fl[it] == 2u) sel[kept_before++] = tid * ITEMS + it;
    }
    if (tid == 0) sc.n_sel = sc.total;
  }
  __syncthreads();
  const uint32_t ks = sc.n_sel;  // == min(k, R)
  // rank the kept runs by (count descending, run ascending)
  for (uint32_t t = tid; t < ks; t += NT) {
    const uint32_t r = sel[t], c = run_count(r);
    uint32_t rank = 0;
    for (uint32_t u = 0; u < ks; ++u) {
      const uint32_t ru = sel[u], cu = run_count(ru);
      rank += (cu > c || (cu == c && ru < r)) ? 1u : 0u;
    }
    order[rank] = r;
  }
  __syncthreads();
  return ks;
}

// Both steps: head flags in work -> runs -> top-k (runs: FC_MAX_OCC + 1
// words; work: FC_MAX_OCC words; sel, order: FC_MAX_TOPK words; wsum: NT / 32).
template <int NT>
__device__ uint32_t rank_runs(uint32_t nocc, int k, uint32_t* runs, uint32_t* work, uint32_t* sel, uint32_t* order,
                              uint32_t* wsum, RunsScratch& sc) {
  const uint32_t R = runs_from_heads<NT>(nocc, runs, work, wsum, sc);
  return topk_runs<NT>(R, k, runs, work, sel, order, wsum, sc);
}
