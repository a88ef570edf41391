// fc_tree_attn: tree-masked verification attention (Section IV-D, Eq. 4).
// Every draft-tree node attends to the whole KV cache of its sequence and to
// its tree ancestors (and itself), so one forward verifies every draft.
//
// GB300 design.  One CTA serves one (sequence, kv head) group and up to 256
// query rows of it, as two 128-row tiles A and B:
//   * GQA packing: rows are (query head in group, tree node) pairs over the
//     group's H/Hkv heads and the sequence's n_nodes nodes, packed densely, so
//     small trees waste no tensor-core rows and each K/V tile loaded from HBM
//     serves every query head that shares it (and both tiles).
//   * K/V tiles of 128 keys x 128 dims stream in with TMA (128-byte swizzle,
//     two K stages and two V stages, released separately: a K stage as soon
//     as both tiles' QK MMAs are done, a V stage after both PV MMAs).  The
//     tree's own K/V form one last tile.
//   * tcgen05.mma (bf16 in, fp32 accumulate): S_X = Q_X K^T into tensor
//     memory; the softmax writes P_X (bf16) over the first half of S_X in
//     tensor memory, and O_X += P_X V takes P_X straight from tensor memory
//     (A operand) with V as an MN-major shared-memory operand.  One warp
//     issues every MMA (warp-uniform, one lane elected inside each
//     instruction), in the order PV_X(j-1) -> QK_X(j) per tile, so S_X is
//     never overwritten before PV_X has read P_X from it.
//   * two softmax warpgroups, one per tile, one row per thread: tile A's
//     softmax runs while the tensor cores do tile B's PV and QK, and the
//     other way round.  The tree mask and the ragged cache tail are applied in
//     registers; the online softmax is in base 2 with lazy rescaling of O.
//   * every mbarrier wait is bounded; a wait that runs out raises
//     FC_ERR_TIMEOUT, the CTA drains its in-flight copies and MMAs (bounded
//     again), frees its tensor memory and returns.
#include <algorithm>
#include <cmath>
#include <mutex>

#include "fc_common.cuh"

FC_DEFINE_ERROR_WORD(attn)

namespace {

constexpr int TA_THREADS = 384;  // warp 0 TMA, warp 1 MMA, warps 4-7 softmax A, warps 8-11 softmax B
constexpr int BM = 128;          // query rows per tile
constexpr int TILES = 2;         // tiles per CTA
constexpr int BN = 128;          // keys per block
constexpr int HD = 128;          // head dim
constexpr int MAX_PARTS = 4;     // most CTAs one unit's KV blocks are split over
constexpr uint32_t HALF_BYTES = BN * 64 * 2;  // one 64-dim half of a 128-row tile
constexpr uint32_t TILE_BYTES = 2 * HALF_BYTES;
constexpr uint32_t OFF_Q = 0;                              // Q_A, Q_B
constexpr uint32_t OFF_K = OFF_Q + TILES * TILE_BYTES;     // 2 stages
constexpr uint32_t OFF_V = OFF_K + 2 * TILE_BYTES;         // 2 stages
constexpr uint32_t OFF_BAR = OFF_V + 2 * TILE_BYTES;
constexpr uint32_t SMEM_BYTES = OFF_BAR + 256 + 1024;      // + alignment slack
constexpr uint32_t TMEM_COLS = 512;                        // S_A, S_B, O_A, O_B (128 columns each)
constexpr uint64_t WAIT_CYCLES = 4000000000ull;            // ~2 s
constexpr uint64_t DRAIN_CYCLES = 400000000ull;            // ~0.2 s
// Lazy rescaling: O and l are rescaled only when a row's running maximum
// (base-2 logits) grows by more than this; until then probabilities may reach
// 2^RESCALE_THRESHOLD, harmless in bf16/fp32.
constexpr float RESCALE_THRESHOLD = 8.f;
// Register split (setmaxnreg): the kernel launches with REGS_LAUNCH per
// thread; the TMA/MMA warpgroup drops to REGS_PRODUCER and the two softmax
// warpgroups rise to REGS_SOFTMAX, enough to hold a row's 128 scores.  The
// shares must add up to the launch's allocation or the increase never returns;
// the host checks the compiled register count before launching.
constexpr int REGS_LAUNCH = 168, REGS_PRODUCER = 48, REGS_SOFTMAX = 224;
static_assert(128 * REGS_PRODUCER + 256 * REGS_SOFTMAX <= TA_THREADS * REGS_LAUNCH, "register split");

// barrier slots (8 bytes each)
enum {
  B_KFULL = 0,   // [2] K tile landed
  B_VFULL = 2,   // [2] V tile landed
  B_KEMPTY = 4,  // [2] K tile consumed by both QK MMAs
  B_VEMPTY = 6,  // [2] V tile consumed by both PV MMAs
  B_SFULL = 8,   // [2 tiles] S_X ready
  B_PFULL = 10,  // [2 tiles] P_X written (128 arrivals)
  B_ODONE = 12,  // one-tile CTAs: a PV into O done (one completion per block)
  B_DRAIN = 14,  // MMA drain on abort
  B_OFIN = 15,   // [2 tiles] the last PV into O_X done
  N_BARS = 17
};

struct AttnArgs {
  const __nv_bfloat16* q;
  const int32_t* kv_len;
  const uint64_t* mask;
  const int32_t* n_nodes;
  __nv_bfloat16* out;
  int B, n_pad, H, Hkv, G, kv_cap, ctas;  // ctas = row chunks (units) per group
  int u_split;     // units [0, u_split) run whole, one CTA each; the rest ...
  int parts;       // ... have their KV blocks split over this many CTAs (1..MAX_PARTS)
  int* ws_cnt;     // [split units][2]: arrival tickets, finished partials (zeroed before the launch)
  float2* ws_ml;   // [split units][parts][256 rows]: (m, l) of a partial, by part
  float* ws_o;     // [split units][parts][256 rows][128]: unnormalised O of a partial, by part
  unsigned int* err;  // the launch's error word (NULL: this file's own)
  float scale_log2;
  const int32_t* pos;  // [B][n_pad] node positions: rotate Q by them (RoPE), or nullptr
  double rope_nl2f;    // -2 log2(base) / D: pair i turns by pos * 2^(i * rope_nl2f)
};

// Rotates the two pairs held by one 32-bit word of each half: l holds
// dimensions i, i + 1 and h the same dimensions + D/2.
__device__ __forceinline__ void rope_word(uint32_t& l, uint32_t& h, float pos, const float2* tab, int i) {
  __nv_bfloat162 lb = *reinterpret_cast<__nv_bfloat162*>(&l), hb = *reinterpret_cast<__nv_bfloat162*>(&h);
  const float2 xl = __bfloat1622float2(lb), xh = __bfloat1622float2(hb);
  float s0, c0, s1, c1;
  fc_rope_sincos(pos, tab[i], s0, c0);
  fc_rope_sincos(pos, tab[i + 1], s1, c1);
  lb = __float22bfloat162_rn(make_float2(xl.x * c0 - xh.x * s0, xl.y * c1 - xh.y * s1));
  hb = __float22bfloat162_rn(make_float2(xh.x * c0 + xl.x * s0, xh.y * c1 + xl.y * s1));
  l = *reinterpret_cast<uint32_t*>(&lb);
  h = *reinterpret_cast<uint32_t*>(&hb);
}

// Rotates the 8 pairs held by two 16-byte chunks: lo = dimensions
// i0 .. i0 + 7, hi = the same dimensions + D/2.
__device__ __forceinline__ void rope_chunks(uint4& lo, uint4& hi, float pos, const float2* tab, int i0) {
  rope_word(lo.x, hi.x, pos, tab, i0);
  rope_word(lo.y, hi.y, pos, tab, i0 + 2);
  rope_word(lo.z, hi.z, pos, tab, i0 + 4);
  rope_word(lo.w, hi.w, pos, tab, i0 + 6);
}

// The Q tiles of a CTA with RoPE fused into the staging: a 16-byte chunk of
// the first 64 dimensions and its partner chunk of the second 64 are rotated
// together and land at the same swizzled offset of the two halves.
__device__ __forceinline__ void stage_q_rope(unsigned char* sq, const __nv_bfloat16* q, const int32_t* pos,
                                             const float2* tab, int b, int g, int G, int H, int n_pad, int nn,
                                             int row0, int rows_total, int tid) {
  for (int e = tid; e < TILES * BM * 8; e += TA_THREADS) {
    const int r = e >> 3, gran = e & 7;
    const int tile = r / BM, rt = r - tile * BM;
    const int rg = row0 + r;
    uint4 lo = make_uint4(0, 0, 0, 0), hi = lo;
    if (rg < rows_total) {
      const int hh = rg / nn, i = rg - hh * nn;
      const uint4* src = reinterpret_cast<const uint4*>(q + (((size_t)b * n_pad + i) * H + g * G + hh) * HD);
      lo = src[gran];
      hi = src[gran + 8];
      const int p = pos[(size_t)b * n_pad + i];
      if (p >= 0) rope_chunks(lo, hi, (float)p, tab, 8 * gran);
    }
    unsigned char* dst = sq + tile * TILE_BYTES + rt * 128 + ((gran ^ (rt & 7)) << 4);
    *reinterpret_cast<uint4*>(dst) = lo;
    *reinterpret_cast<uint4*>(dst + HALF_BYTES) = hi;
  }
}

// 2^x on the MUFU unit.  The flush-to-zero form is a single instruction; the
// results it flushes (below 2^-126) are probabilities that cannot move an
// fp32 row sum whose largest term is >= 1.
__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// ---- packed fp32 pairs (sm_100 family f32x2 arithmetic) ----
__device__ __forceinline__ uint64_t f2_pack(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t v, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

template <int N>
__device__ __forceinline__ void regs_dec() {
  asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(N));
}
template <int N>
__device__ __forceinline__ void regs_inc() {
  asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(N));
}

// Named barrier among `count` threads (the softmax warpgroups use id 1).
__device__ __forceinline__ void named_sync(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// All 32 lanes wait; the result is warp-uniform.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort) {
  return __all_sync(0xFFFFFFFFu, mbar_wait_bounded(bar, parity, abort, WAIT_CYCLES));
}

// An L2 prefetch of a tensor-map tile (no shared memory, no barrier).
__device__ __forceinline__ void tma_prefetch_l2_3d(const CUtensorMap* map, int x, int y, int z) {
  asm volatile("cp.async.bulk.prefetch.tensor.3d.L2.global.tile [%0, {%1, %2, %3}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(z)
               : "memory");
}
// One-tile CTAs are bound by their K/V delivery: they prefetch the cache
// blocks this far ahead of their loads into L2.
constexpr int PF_ONE_TILE = 2;

// 16-byte asynchronous global -> shared copies (cp.async, no mbarrier): a
// thread issues all of its copies before it waits once for them.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;\n" ::: "memory"); }

// ROPE: the queries arrive unrotated and are rotated by a.pos while staged
// (a separate instance, so the plain kernel's code is unchanged).
template <bool ROPE>
__global__ void __launch_bounds__(TA_THREADS, 1)
    k_tree_attn(const __grid_constant__ CUtensorMap tm_kc, const __grid_constant__ CUtensorMap tm_vc,
                const __grid_constant__ CUtensorMap tm_kt, const __grid_constant__ CUtensorMap tm_vt, AttnArgs a) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  __shared__ int s_ticket, s_ready;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // Units (group, row chunk) in launch order, so the row chunks of a group,
  // which stream the same K/V blocks, run together and share them through
  // L2.  The units of the last, partial wave are split over `parts` CTAs each
  // (launched last: whole units first, the short split CTAs fill the tail).
  int unit, part, nparts;
  if ((int)blockIdx.x < a.u_split) {
    unit = blockIdx.x;
    part = 0;
    nparts = 1;
  } else {
    const int k = blockIdx.x - a.u_split;
    unit = a.u_split + k / a.parts;
    part = k - (unit - a.u_split) * a.parts;
    nparts = a.parts;
  }
  const int su = unit - a.u_split;  // index among the split units
  const int bg = unit / a.ctas, c = unit - bg * a.ctas;
  const int b = bg / a.Hkv, g = bg - b * a.Hkv;
  const int nn_raw = a.n_nodes[b], kvl = a.kv_len[b];
  const bool bad = nn_raw < 1 || nn_raw > a.n_pad || kvl < 0 || kvl > a.kv_cap;
  const int nn = bad ? 0 : nn_raw;
  if (bad && c == 0 && part == 0 && tid == 0) fc_flag(FC_ERR_WORD(a.err), FC_EBIT_INVALID);

  // Zero the padding rows (nodes >= n_nodes) of this group: the group's part-0
  // CTAs share them (row r of the G x pad padding rows goes to CTA r mod ctas),
  // threads [t0, t0 + nthr) of this CTA take its rows.
  auto zero_pad = [&](int t0, int nthr) {
    if (part != 0 || tid < t0 || tid >= t0 + nthr) return;
    const int pad = a.n_pad - nn;
    const int my_rows = (a.G * pad - c + a.ctas - 1) / a.ctas;  // rows c, c + ctas, ...
    for (int e = tid - t0; e < my_rows * (HD / 8); e += nthr) {
      const int r = c + (e / (HD / 8)) * a.ctas, ch = e % (HD / 8);
      const int hh = r / pad, i = nn + (r - hh * pad);
      reinterpret_cast<uint4*>(a.out + (((size_t)b * a.n_pad + i) * a.H + g * a.G + hh) * HD)[ch] =
          make_uint4(0, 0, 0, 0);
    }
  };
  const int rows_total = a.G * nn;
  const int row0 = c * (TILES * BM);
  if (row0 >= rows_total) {
    zero_pad(0, TA_THREADS);
    return;
  }
  const bool has_b = row0 + BM < rows_total;

  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase + OFF_Q, sK = sbase + OFF_K, sV = sbase + OFF_V;
  const uint32_t bar0 = sbase + OFF_BAR;
  auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };

  const int nblk_c = (kvl + BN - 1) / BN;
  const int nblk_all = nblk_c + 1;  // + the tree block (always the unit's last block)
  // This CTA's share of the unit's blocks: [kb, kb + nblk).  Parts may be
  // empty when a unit has fewer blocks than parts.
  const int kb = part * nblk_all / nparts;
  const int nblk = (part + 1) * nblk_all / nparts - kb;
  int n_contrib = 0;
  for (int h = 0; h < nparts; ++h) n_contrib += ((h + 1) * nblk_all / nparts > h * nblk_all / nparts);
  if (nblk == 0) {
    zero_pad(0, TA_THREADS);
    return;
  }

  // K and V of block j into stage j & 1 (the tree's own K/V form the last
  // block; the tree maps' box is 128 rows, so rows >= n_pad arrive as zeros)
  auto load_kv = [&](int j, bool k_part) {
    const int st = j & 1;
    const bool tree = kb + j >= nblk_c;
    const CUtensorMap* m = k_part ? (tree ? &tm_kt : &tm_kc) : (tree ? &tm_vt : &tm_vc);
    const int y = tree ? 0 : (kb + j) * BN;
    const uint32_t dst = (k_part ? sK : sV) + st * TILE_BYTES, fb = bar((k_part ? B_KFULL : B_VFULL) + st);
    mbar_expect_tx(fb, TILE_BYTES);
    tma_load_3d(dst, m, 0, y, bg, fb);
    tma_load_3d(dst + HALF_BYTES, m, 64, y, bg, fb);
  };
  const int n_early = min(2, nblk);  // blocks whose loads start before Q is staged
  if (tid == 0) {
    s_abort = 0;
    for (int i = 0; i < N_BARS; ++i) mbar_init(bar(i), (i == B_PFULL || i == B_PFULL + 1) ? 128u : 1u);
    fence_mbar_init();
    prefetch_tmap(&tm_kc);
    prefetch_tmap(&tm_vc);
    prefetch_tmap(&tm_kt);
    prefetch_tmap(&tm_vt);
    for (int j = 0; j < n_early; ++j) {  // the stages are free: start the first copies now
      load_kv(j, true);
      load_kv(j, false);
    }
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), TMEM_COLS);
    tmem_relinquish();
  }
  // Q tiles: rows (head in group, node) packed densely, 128-byte swizzled, K-major.
  if constexpr (ROPE) {
    __shared__ float2 s_rope[HD / 2];
    fc_rope_table(s_rope, HD / 2, a.rope_nl2f);
    __syncthreads();
    stage_q_rope(smem + OFF_Q, a.q, a.pos, s_rope, b, g, a.G, a.H, a.n_pad, nn, row0, rows_total, tid);
  } else {
    // asynchronous 16-byte copies: all of a thread's rows in flight at once
    for (int e = tid; e < TILES * BM * 16; e += TA_THREADS) {
      const int r = e >> 4, ch = e & 15, half = ch >> 3, gran = ch & 7;
      const int tile = r / BM, rt = r - tile * BM;
      const int rg = row0 + r;
      const uint32_t off = OFF_Q + tile * TILE_BYTES + half * HALF_BYTES + rt * 128 + ((gran ^ (rt & 7)) << 4);
      if (rg < rows_total) {
        const int hh = rg / nn, i = rg - hh * nn;
        cp_async16(sbase + off, a.q + (((size_t)b * a.n_pad + i) * a.H + g * a.G + hh) * HD + ch * 8);
      } else {
        *reinterpret_cast<uint4*>(smem + off) = make_uint4(0, 0, 0, 0);
      }
    }
    cp_async_wait_all();
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  if (warp < 4) {
    regs_dec<REGS_PRODUCER>();  // the whole warpgroup (warps 2 and 3 only wait)
    if (warp == 0) {
      // ---------------- TMA producer ----------------
      if (lane == 0) {
        int issued = n_early;  // blocks 0 and 1 were issued at setup
        for (int j = n_early; j < nblk; ++j) {
          const int st = j & 1;
          if (!mbar_wait_bounded(bar(B_KEMPTY + st), ((j >> 1) - 1) & 1, &s_abort, WAIT_CYCLES)) break;
          load_kv(j, true);
          if (!mbar_wait_bounded(bar(B_VEMPTY + st), ((j >> 1) - 1) & 1, &s_abort, WAIT_CYCLES)) {
            issued = j + 1;  // the K copy of this block is in flight
            break;
          }
          load_kv(j, false);
          issued = j + 1;
          const int jp = kb + j + PF_ONE_TILE;
          if (!has_b && j + PF_ONE_TILE < nblk && jp < nblk_c) {  // a cache block of this CTA's share
            tma_prefetch_l2_3d(&tm_kc, 0, jp * BN, bg);
            tma_prefetch_l2_3d(&tm_kc, 64, jp * BN, bg);
            tma_prefetch_l2_3d(&tm_vc, 0, jp * BN, bg);
            tma_prefetch_l2_3d(&tm_vc, 64, jp * BN, bg);
          }
        }
        if (s_abort) {  // let the copies already issued land before the CTA exits
          volatile int dummy = 0;
          for (int j = max(0, issued - 2); j < issued; ++j) {
            mbar_wait_bounded(bar(B_KFULL + (j & 1)), (j >> 1) & 1, &dummy, DRAIN_CYCLES);
            mbar_wait_bounded(bar(B_VFULL + (j & 1)), (j >> 1) & 1, &dummy, DRAIN_CYCLES);
          }
        }
      }
      __syncwarp();
    } else if (warp >= 2) {
      zero_pad(64, 64);  // warps 2-3: the padding output rows, while the pipeline runs
    } else if (warp == 1) {
      // ---------------- MMA issuer (+ ragged V rows zeroed by the warp) -------
      constexpr uint32_t IDESC_QK = idesc_bf16_f32(BM, BN, 0);
      constexpr uint32_t IDESC_PV = idesc_bf16_f32(BM, HD, 1);
      // S buffer sb (TMEM columns sb*128..) <- Q tile x . K(j)^T; arrives on S_FULL[sb]
      auto issue_qk = [&](int j, int x, int sb) {
        const uint32_t kb = sK + (j & 1) * TILE_BYTES, qb = sQ + x * TILE_BYTES;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint32_t off = (kk >> 2) * HALF_BYTES + (kk & 3) * 32;
          tc_mma_f16(tmem + sb * 128, smem_desc_sw128(qb + off, 16, 1024), smem_desc_sw128(kb + off, 16, 1024),
                     IDESC_QK, kk > 0);
        }
        tc_commit(bar(B_SFULL + sb));
      };
      // O tile x += P (bf16 pairs in the first 64 columns of S buffer sb) . V(jj)
      auto issue_pv = [&](int jj, int x, int sb, int) {
        const uint32_t vb = sV + (jj & 1) * TILE_BYTES;
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk)  // 8 packed columns per 16 keys
          tc_mma_f16_tmem_a(tmem + 256 + x * 128, tmem + sb * 128 + kk * 8,
                            smem_desc_sw128(vb + kk * 2048, HALF_BYTES, 1024), IDESC_PV, (jj > 0 || kk > 0));
      };
      // Never let garbage (possibly NaN) V rows meet a zero probability: the
      // cache's rows past kv_len and the tree's rows past n_nodes (the tree
      // tile's rows >= n_pad arrived as zeros).
      auto zero_ragged_v = [&](int jj) {
        const int gj = kb + jj;
        const bool tree = gj >= nblk_c;
        const int nv = tree ? nn : min(BN, kvl - gj * BN), top = tree ? a.n_pad : BN;
        if (nv < top) {
          unsigned char* vt = smem + OFF_V + (jj & 1) * TILE_BYTES;
          for (int e = lane; e < (top - nv) * 16; e += 32) {
            const int r = nv + (e >> 4), ch = e & 15;
            *reinterpret_cast<uint4*>(vt + (ch >> 3) * HALF_BYTES + r * 128 + (ch & 7) * 16) = make_uint4(0, 0, 0, 0);
          }
          fence_proxy_async_smem();
        }
        __syncwarp();
      };
      bool ok = true;
      if (has_b) {
        // Two tiles, one S buffer each: per tile PV_X(j-1) -> QK_X(j); the
        // other tile's softmax runs meanwhile.
        ok = warp_wait(bar(B_KFULL), 0, &s_abort);
        if (ok) {
          tc_fence_after();
          for (int x = 0; x < 2; ++x) issue_qk(0, x, x);
          tc_commit(bar(B_KEMPTY));
        }
        for (int j = 1; ok && j <= nblk; ++j) {
          const int jj = j - 1, st = jj & 1;
          if (!(ok = warp_wait(bar(B_VFULL + st), (jj >> 1) & 1, &s_abort))) break;
          zero_ragged_v(jj);
          for (int x = 0; ok && x < 2; ++x) {
            if (!(ok = warp_wait(bar(B_PFULL + x), jj & 1, &s_abort))) break;
            tc_fence_after();
            issue_pv(jj, x, x, x);
            if (j < nblk) {
              if (x == 0 && !(ok = warp_wait(bar(B_KFULL + (j & 1)), (j >> 1) & 1, &s_abort))) break;
              issue_qk(j, x, x);
            } else {
              tc_commit(bar(B_OFIN + x));
            }
          }
          if (!ok) break;
          if (j < nblk) tc_commit(bar(B_KEMPTY + (j & 1)));
          tc_commit(bar(B_VEMPTY + st));
        }
      } else {
        // One tile, S double-buffered in both S regions: QK(j+1) runs during
        // softmax(j); PV(j) reads P from S(j&1) before QK(j+2) overwrites it.
        for (int j = 0; ok && j < min(2, nblk); ++j) {
          if (!(ok = warp_wait(bar(B_KFULL + j), 0, &s_abort))) break;
          tc_fence_after();
          issue_qk(j, 0, j);
          tc_commit(bar(B_KEMPTY + j));
        }
        for (int jj = 0; ok && jj < nblk; ++jj) {
          const int v = jj & 1;
          if (!(ok = warp_wait(bar(B_VFULL + v), (jj >> 1) & 1, &s_abort))) break;
          zero_ragged_v(jj);
          if (!(ok = warp_wait(bar(B_PFULL + v), (jj >> 1) & 1, &s_abort))) break;
          tc_fence_after();
          issue_pv(jj, 0, v, 0);
          tc_commit(bar(B_ODONE));
          tc_commit(bar(B_VEMPTY + v));
          if (jj == nblk - 1) tc_commit(bar(B_OFIN));
          if (jj + 2 < nblk) {
            if (!(ok = warp_wait(bar(B_KFULL + v), ((jj + 2) >> 1) & 1, &s_abort))) break;
            tc_fence_after();
            issue_qk(jj + 2, 0, v);
            tc_commit(bar(B_KEMPTY + v));
          }
        }
      }
      if (__any_sync(0xFFFFFFFFu, s_abort)) {  // let issued MMAs retire before the tensor memory is freed
        tc_commit(bar(B_DRAIN));
        volatile int dummy = 0;
        mbar_wait_bounded(bar(B_DRAIN), 0, &dummy, DRAIN_CYCLES);
      }
    }
  } else {
    regs_inc<REGS_SOFTMAX>();
    // ---------------- softmax warpgroups: tile x, thread = row ----------------
    const int x = (warp - 4) >> 2;  // 0: warps 4-7, 1: warps 8-11
    const int q4 = warp & 3;        // TMEM lane quarter of this warp
    const bool active = (x == 0 || has_b);
    const int r = q4 * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const uint32_t tO = tmem + 256 + x * 128 + lane_off;
    const int rg = row0 + x * BM + r;
    const bool row_ok = active && rg < rows_total;
    const int hh = row_ok ? rg / nn : 0, i = row_ok ? rg - hh * nn : 0;
    __nv_bfloat16* dst = a.out + (((size_t)b * a.n_pad + i) * a.H + g * a.G + hh) * HD;
    float m_run = -INFINITY, l_run = 0.f;
    bool fin = false;  // warp-uniform: the row's O is complete in tensor memory
    if (active) {
      const int nw = a.n_pad / 64;
      const uint64_t* mrow = a.mask + ((size_t)b * a.n_pad + i) * nw;
      const uint64_t m0 = mrow[0], m1 = (nw > 1) ? mrow[1] : 0ull;
      bool ok = true;
      for (int j = 0; j < nblk; ++j) {
        // two tiles: S buffer x, one phase per block; one tile: S buffers alternate
        const int sb = has_b ? x : (j & 1);
        const uint32_t par = has_b ? (j & 1) : ((j >> 1) & 1);
        const uint32_t tS = tmem + sb * 128 + lane_off;
        if (!(ok = warp_wait(bar(B_SFULL + sb), par, &s_abort))) break;
        tc_fence_after();
        const bool tree = (kb + j == nblk_all - 1);
        const int nv = tree ? BN : min(BN, kvl - (kb + j) * BN);
        const bool masked = tree || nv < BN;  // block-uniform
        // keep-bits of 32-column chunk q: the tree mask row, or the ragged cache tail
        auto keep_bits = [&](int q) -> uint32_t {
          if (tree) return (uint32_t)((q < 2 ? m0 : m1) >> (32 * (q & 1)));
          const int lo = nv - 32 * q;
          return lo >= 32 ? 0xFFFFFFFFu : (lo <= 0 ? 0u : ((1u << lo) - 1u));
        };
        // The block's 128 scores of this row stay in registers from here on.
        uint32_t sv[128];
#pragma unroll
        for (int c4 = 0; c4 < 4; ++c4) tmem_ld32(tS + c4 * 32, *reinterpret_cast<uint32_t(*)[32]>(&sv[c4 * 32]));
        tc_wait_ld();
        if (masked) {  // masked scores become -inf (exp2 turns them into exact zeros)
#pragma unroll
          for (int c4 = 0; c4 < 4; ++c4) {
            const uint32_t kb = keep_bits(c4);
#pragma unroll
            for (int cc = 0; cc < 32; ++cc)
              if (!(kb & (1u << cc))) sv[c4 * 32 + cc] = __float_as_uint(-INFINITY);
          }
        }
        // raw row maximum over the block (scale > 0 commutes with max)
        float pm[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) pm[u] = -INFINITY;
#pragma unroll
        for (int cc = 0; cc < 128; cc += 2)
          pm[(cc >> 1) & 7] = fmax3(pm[(cc >> 1) & 7], __uint_as_float(sv[cc]), __uint_as_float(sv[cc + 1]));
        const float mx = fmaxf(fmaxf(fmaxf(pm[0], pm[1]), fmaxf(pm[2], pm[3])),
                               fmaxf(fmaxf(pm[4], pm[5]), fmaxf(pm[6], pm[7]))) * a.scale_log2;
        // lazy rescale: keep the old reference unless the maximum grew a lot
        const float m_new = (mx > m_run + RESCALE_THRESHOLD) ? mx : m_run;
        const float m_use = (m_new == -INFINITY) ? 0.f : m_new;
        const float alpha = fast_exp2(m_run - m_use);
        // Two tiles: O_X is stable here (PV_X(j-1) was issued before QK_X(j) and
        // MMAs retire in order).  One tile: PV(j-1) may still run; wait for it.
        if (j > 0 && __any_sync(0xFFFFFFFFu, alpha != 1.f)) {  // warp-uniform: tcgen05.ld/st are collective
          if (!has_b && !(ok = warp_wait(bar(B_ODONE), (j - 1) & 1, &s_abort))) break;
          tc_fence_after();
#pragma unroll
          for (int cc = 0; cc < HD / 32; ++cc) {
            uint32_t o[32];
            tmem_ld32(tO + cc * 32, o);
            tc_wait_ld();
#pragma unroll
            for (int u = 0; u < 32; ++u) o[u] = __float_as_uint(__uint_as_float(o[u]) * alpha);
            tmem_st32(tO + cc * 32, o);
          }
        }
        // P = exp2(s * scale - m), bf16 pairs written over S's first 64 columns
        uint64_t ps2[4] = {0ull, 0ull, 0ull, 0ull};  // packed partial row sums
        const uint64_t sc2 = f2_pack(a.scale_log2, a.scale_log2), nm2 = f2_pack(-m_use, -m_use);
#pragma unroll
        for (int c4 = 0; c4 < 4; ++c4) {
          uint32_t pk[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const int cc = c4 * 32 + 2 * q;
            float x0, x1;
            f2_unpack(f2_fma(f2_pack(__uint_as_float(sv[cc]), __uint_as_float(sv[cc + 1])), sc2, nm2), x0, x1);
            const float p0 = fast_exp2(x0), p1 = fast_exp2(x1);
            ps2[q & 3] = f2_add(ps2[q & 3], f2_pack(p0, p1));
            pk[q] = pack_bf16x2(p0, p1);
          }
          tmem_st16(tS + c4 * 16, pk);
        }
        tc_wait_st();
        float ps[8];
        f2_unpack(ps2[0], ps[0], ps[1]);
        f2_unpack(ps2[1], ps[2], ps[3]);
        f2_unpack(ps2[2], ps[4], ps[5]);
        f2_unpack(ps2[3], ps[6], ps[7]);
        const float sum = ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
        l_run = l_run * alpha + sum;
        m_run = m_new;
        tc_fence_before();
        mbar_arrive(bar(B_PFULL + sb));
      }
      fin = ok && warp_wait(bar(B_OFIN + x), 0, &s_abort);
      if (fin) tc_fence_after();
    }
    if (n_contrib == 1) {
      if (fin) {
        const float inv = 1.f / l_run;
#pragma unroll
        for (int cc = 0; cc < HD / 32; ++cc) {
          uint32_t o[32];
          tmem_ld32(tO + cc * 32, o);
          tc_wait_ld();
          if (row_ok) {
#pragma unroll
            for (int u = 0; u < 32; u += 8) {
              uint4 v;
              v.x = pack_bf16x2(__uint_as_float(o[u + 0]) * inv, __uint_as_float(o[u + 1]) * inv);
              v.y = pack_bf16x2(__uint_as_float(o[u + 2]) * inv, __uint_as_float(o[u + 3]) * inv);
              v.z = pack_bf16x2(__uint_as_float(o[u + 4]) * inv, __uint_as_float(o[u + 5]) * inv);
              v.w = pack_bf16x2(__uint_as_float(o[u + 6]) * inv, __uint_as_float(o[u + 7]) * inv);
              *reinterpret_cast<uint4*>(dst + cc * 32 + u) = v;
            }
          }
        }
      }
    } else {
      // The unit's KV blocks are split over n_contrib CTAs.  Softmax
      // attention over a key set is a ratio of two sums over its keys, so the
      // parts' (m, l, O) over disjoint key ranges merge exactly:
      //   m* = max m_t,  l* = sum l_t 2^(m_t - m*),  O = sum O_t 2^(m_t - m*) / l*.
      // Each CTA takes a ticket when done; all but the last store their rows
      // in their part's slot, the last waits (bounded) until they have, then
      // merges and writes out.  The CTAs it waits for are resident: they took
      // their tickets before it.  The merge sums the parts in part order,
      // whichever CTA merges, so the result does not depend on timing.
      named_sync(1, 256);
      if (tid == 128) s_ticket = atomicAdd(a.ws_cnt + 2 * su, 1);
      named_sync(1, 256);
      const int t = s_ticket;
      const size_t slot0 = (size_t)su * a.parts * (TILES * BM);  // the unit's first slot row
      const int lr = x * BM + r;                                          // row within the unit
      if (t < n_contrib - 1) {
        if (fin) {
          float* od = a.ws_o + (slot0 + (size_t)part * (TILES * BM) + lr) * HD;
#pragma unroll
          for (int cc = 0; cc < HD / 32; ++cc) {
            uint32_t o[32];
            tmem_ld32(tO + cc * 32, o);
            tc_wait_ld();
            if (row_ok) {
#pragma unroll
              for (int u = 0; u < 32; u += 4)
                __stcg(reinterpret_cast<float4*>(od + cc * 32 + u),
                       make_float4(__uint_as_float(o[u]), __uint_as_float(o[u + 1]), __uint_as_float(o[u + 2]),
                                   __uint_as_float(o[u + 3])));
            }
          }
          if (row_ok) __stcg(a.ws_ml + slot0 + (size_t)part * (TILES * BM) + lr, make_float2(m_run, l_run));
        }
        named_sync(1, 256);
        if (tid == 128) {
          __threadfence();
          atomicAdd(a.ws_cnt + 2 * su + 1, 1);
        }
      } else {
        if (tid == 128) {
          const volatile int* done = a.ws_cnt + 2 * su + 1;
          const long long t0 = clock64();
          int ready;
          while (!(ready = (*done >= n_contrib - 1)) && !s_abort && (uint64_t)(clock64() - t0) < WAIT_CYCLES)
            __nanosleep(128);
          if (!ready) s_abort = 1;
          __threadfence();
          s_ready = ready;
        }
        named_sync(1, 256);
        if (fin && s_ready) {
          // the parts with keys, in part order; this CTA's own partial at its index
          auto contributes = [&](int h) { return (h + 1) * nblk_all / nparts > h * nblk_all / nparts; };
          float mt[MAX_PARTS], wt[MAX_PARTS];
          float mstar = -INFINITY;
#pragma unroll
          for (int h = 0; h < MAX_PARTS; ++h) {
            mt[h] = -INFINITY;
            wt[h] = 0.f;
            if (h >= nparts || !contributes(h)) continue;
            const float2 ml = h == part ? make_float2(m_run, l_run)
                                        : (row_ok ? __ldcg(a.ws_ml + slot0 + (size_t)h * (TILES * BM) + lr)
                                                  : make_float2(m_run, 0.f));
            mt[h] = ml.x;
            wt[h] = ml.y;  // l for now
            mstar = fmaxf(mstar, ml.x);
          }
          float lstar = 0.f;
#pragma unroll
          for (int h = 0; h < MAX_PARTS; ++h) {
            if (h >= nparts || !contributes(h)) continue;
            const float w = exp2f(mt[h] - mstar);
            lstar += wt[h] * w;
            wt[h] = w;
          }
          const float inv = 1.f / lstar;
#pragma unroll
          for (int cc = 0; cc < HD / 32; ++cc) {
            uint32_t o[32];
            tmem_ld32(tO + cc * 32, o);
            tc_wait_ld();
            if (row_ok) {
              float acc[32];
#pragma unroll
              for (int u = 0; u < 32; ++u) acc[u] = 0.f;
#pragma unroll
              for (int h = 0; h < MAX_PARTS; ++h) {
                if (h >= nparts || !contributes(h)) continue;
                if (h == part) {
#pragma unroll
                  for (int u = 0; u < 32; ++u) acc[u] += __uint_as_float(o[u]) * wt[h];
                } else {
                  const float* os = a.ws_o + (slot0 + (size_t)h * (TILES * BM) + lr) * HD + cc * 32;
#pragma unroll
                  for (int u = 0; u < 32; u += 4) {
                    const float4 v = __ldcg(reinterpret_cast<const float4*>(os + u));
                    acc[u] += v.x * wt[h];
                    acc[u + 1] += v.y * wt[h];
                    acc[u + 2] += v.z * wt[h];
                    acc[u + 3] += v.w * wt[h];
                  }
                }
              }
#pragma unroll
              for (int u = 0; u < 32; u += 8) {
                uint4 v;
                v.x = pack_bf16x2(acc[u + 0] * inv, acc[u + 1] * inv);
                v.y = pack_bf16x2(acc[u + 2] * inv, acc[u + 3] * inv);
                v.z = pack_bf16x2(acc[u + 4] * inv, acc[u + 5] * inv);
                v.w = pack_bf16x2(acc[u + 6] * inv, acc[u + 7] * inv);
                *reinterpret_cast<uint4*>(dst + cc * 32 + u) = v;
              }
            }
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (tid == 0 && s_abort) fc_flag(FC_ERR_WORD(a.err), FC_EBIT_TIMEOUT);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// Streaming variant for short one-tile units: every group's rows fit one
// 128-row tile (G * n_pad <= 128) and the caches are short, so a unit is a
// handful of K/V blocks and a CTA per unit would pay its set-up (barriers,
// tensor memory, Q staging, pipeline fill) and its epilogue for each few
// blocks.  Here a CTA serves units blockIdx.x, blockIdx.x + gridDim.x, ... in
// turn and keeps the pipeline full across them: one K/V stage ring runs over
// the concatenated blocks of all its units, and Q and O alternate between two
// buffers per unit (Q_A / Q_B in shared memory, O_A / O_B in tensor memory),
// so warps 2-3 stage unit t + 1's queries and the MMA warp multiplies its
// first blocks while the softmax warps still write unit t's output.  The
// arithmetic per block is k_tree_attn's one-tile path, block for block, so the
// results are the same.
struct StreamUnit {
  int b, g, nn, kvl, nblk_c, nblk;  // nblk = 0: no work (a length out of range, recorded)
  bool bad;
};

__device__ __forceinline__ StreamUnit stream_unit(const AttnArgs& a, int u) {
  StreamUnit su;
  su.b = u / a.Hkv;
  su.g = u - su.b * a.Hkv;
  const int nn = a.n_nodes[su.b], kvl = a.kv_len[su.b];
  su.bad = nn < 1 || nn > a.n_pad || kvl < 0 || kvl > a.kv_cap;
  su.nn = su.bad ? 0 : nn;
  su.kvl = su.bad ? 0 : kvl;
  su.nblk_c = (su.kvl + BN - 1) / BN;
  su.nblk = su.bad ? 0 : su.nblk_c + 1;  // + the tree block, the unit's last
  return su;
}

// Walks a CTA's blocks in order: unit t (the t-th of this CTA), its block j,
// and `live` = how many units with work came before (it picks the Q and O
// buffers and their barrier phases).
struct StreamCursor {
  int t, j, live, n_units;
  StreamUnit su;
  __device__ __forceinline__ bool valid() const { return t < n_units; }
  __device__ __forceinline__ void skip_empty(const AttnArgs& a) {
    while (t < n_units && su.nblk == 0) {
      ++t;
      if (t < n_units) su = stream_unit(a, (int)blockIdx.x + t * (int)gridDim.x);
    }
  }
  __device__ __forceinline__ void start(const AttnArgs& a, int n) {
    t = 0, j = 0, live = 0, n_units = n;
    if (n > 0) su = stream_unit(a, (int)blockIdx.x);
    skip_empty(a);
  }
  __device__ __forceinline__ void next(const AttnArgs& a) {
    if (++j < su.nblk) return;
    j = 0;
    ++live;
    ++t;
    if (t < n_units) su = stream_unit(a, (int)blockIdx.x + t * (int)gridDim.x);
    skip_empty(a);
  }
};

// Shared-memory layout and barrier slots of the streaming kernel with NST K/V
// stages.  With three stages the Q buffers hold 64 rows (the launch's groups
// have G * n_pad <= 64 rows): the 128-row MMA then reads 64 rows past each
// buffer, rows whose scores no output row uses.
template <int NST>
struct StreamLayout {
  static constexpr int QROWS = NST == 3 ? 64 : 128;
  static constexpr uint32_t QHALF = QROWS * 128, QTILE = 2 * QHALF;
  static constexpr uint32_t OFF_Q = 0;                           // Q buffers 0, 1
  static constexpr uint32_t OFF_K = OFF_Q + 2 * QTILE;           // NST stages
  static constexpr uint32_t OFF_V = OFF_K + NST * TILE_BYTES;    // NST stages
  static constexpr uint32_t OFF_BAR = OFF_V + NST * TILE_BYTES;
  static constexpr uint32_t SMEM = OFF_BAR + 256 + 1024;         // + alignment slack
  // barrier slots (8 bytes each)
  static constexpr int KFULL = 0, VFULL = NST, KEMPTY = 2 * NST, VEMPTY = 3 * NST;  // [NST] each
  static constexpr int SFULL = 4 * NST;       // [2] S buffer ready
  static constexpr int PFULL = SFULL + 2;     // [2] P written into S buffer (128 arrivals)
  static constexpr int ODONE = PFULL + 2;     // a PV into O done (one completion per block)
  static constexpr int DRAIN = ODONE + 1;     // MMA drain on abort
  static constexpr int OFIN = DRAIN + 1;      // [2] the last PV of a unit into O buffer done
  static constexpr int OFREE = OFIN + 2;      // [2] the softmax warps have read O buffer out (128 arrivals)
  static constexpr int QFULL = OFREE + 2;     // [2] Q buffer staged (64 arrivals, warps 2-3)
  static constexpr int QFREE = QFULL + 2;     // [2] the last QK reading Q buffer done
  static constexpr int NBARS = QFREE + 2;
  static_assert(NBARS * 8 <= 256, "barrier area");
  static_assert(SMEM + 1024 <= 232448, "shared memory per CTA (the kernel's static part is 1024 bytes)");
};
// Register split of the streaming kernel: the softmax warpgroup rises to
// REGS_SOFTMAX, warps 8-11 (idle) keep the launch's count, and the producer
// warpgroup (two block cursors in the MMA warp) drops to what is left.
constexpr int REGS_PRODUCER_STREAM = 96;
static_assert(128 * REGS_PRODUCER_STREAM + 128 * REGS_SOFTMAX + 128 * REGS_LAUNCH <= TA_THREADS * REGS_LAUNCH,
              "register split");

template <int NST>
__global__ void __launch_bounds__(TA_THREADS, 1)
    k_tree_attn_stream(const __grid_constant__ CUtensorMap tm_kc, const __grid_constant__ CUtensorMap tm_vc,
                       const __grid_constant__ CUtensorMap tm_kt, const __grid_constant__ CUtensorMap tm_vt,
                       AttnArgs a) {
  using L = StreamLayout<NST>;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int U = a.B * a.Hkv;
  const int n_units = max(0, (U - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x);
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase + L::OFF_Q, sK = sbase + L::OFF_K, sV = sbase + L::OFF_V;
  const uint32_t bar0 = sbase + L::OFF_BAR;
  auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };

  // warps 2-3: a unit's queries into Q buffer q (rows past the unit's G * nn
  // are zeros), every row's copy in flight at once; the caller waits
  // (cp_async_wait_all) before it signals the buffer staged
  auto stage_q = [&](const StreamUnit& su, int q) {
    const int t0 = tid - 64, rows_total = a.G * su.nn;
    const uint32_t qt = sQ + q * L::QTILE;
    for (int e = t0; e < L::QROWS * 16; e += 64) {
      const int r = e >> 4, ch = e & 15, half = ch >> 3, gran = ch & 7;
      const uint32_t d = qt + half * L::QHALF + r * 128 + ((gran ^ (r & 7)) << 4);
      if (r < rows_total) {
        const int hh = r / su.nn, i = r - hh * su.nn;
        cp_async16(d, a.q + (((size_t)su.b * a.n_pad + i) * a.H + su.g * a.G + hh) * HD + ch * 8);
      } else {
        *reinterpret_cast<uint4*>(smem + (d - sbase)) = make_uint4(0, 0, 0, 0);
      }
    }
  };
  // The first unit's queries are requested before anything else, so that they
  // do not queue behind every CTA's first K/V stages.
  bool q_pre = false;
  if ((warp == 2 || warp == 3) && n_units > 0) {
    const StreamUnit su0 = stream_unit(a, (int)blockIdx.x);
    if (su0.nblk > 0) {
      stage_q(su0, 0);
      q_pre = true;
    }
  }

  // K or V of global block J (block j of unit su) into stage J % NST.  The tree
  // maps' box is 128 rows: rows >= n_pad arrive as zeros.
  auto load_kv = [&](int J, const StreamUnit& su, int j, bool k_part) {
    const int st = J % NST;
    const bool tree = j >= su.nblk_c;
    const CUtensorMap* m = k_part ? (tree ? &tm_kt : &tm_kc) : (tree ? &tm_vt : &tm_vc);
    const int y = tree ? 0 : j * BN, z = su.b * a.Hkv + su.g;
    const uint32_t dst = (k_part ? sK : sV) + st * TILE_BYTES, fb = bar((k_part ? L::KFULL : L::VFULL) + st);
    mbar_expect_tx(fb, TILE_BYTES);
    tma_load_3d(dst, m, 0, y, z, fb);
    tma_load_3d(dst + HALF_BYTES, m, 64, y, z, fb);
  };
  if (tid == 0) {
    s_abort = 0;
    for (int i = 0; i < L::NBARS; ++i) {
      const bool p128 = i == L::PFULL || i == L::PFULL + 1 || i == L::OFREE || i == L::OFREE + 1;
      const bool q64 = i == L::QFULL || i == L::QFULL + 1;
      mbar_init(bar(i), p128 ? 128u : (q64 ? 64u : 1u));
    }
    fence_mbar_init();
    prefetch_tmap(&tm_kc);
    prefetch_tmap(&tm_vc);
    prefetch_tmap(&tm_kt);
    prefetch_tmap(&tm_vt);
    StreamCursor c;
    c.start(a, n_units);
    for (int J = 0; J < NST && c.valid(); ++J, c.next(a)) {  // the stages are free: start the first copies now
      load_kv(J, c.su, c.j, true);
      load_kv(J, c.su, c.j, false);
    }
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  if (warp < 4) {
    regs_dec<REGS_PRODUCER_STREAM>();
    if (warp == 0) {
      // ---------------- TMA producer: the CTA's blocks in order ----------------
      if (lane == 0) {
        StreamCursor c;
        c.start(a, n_units);
        int J = 0, issued = 0;
        for (; c.valid(); ++J, c.next(a)) {
          if (J < NST) {
            issued = J + 1;
            continue;
          }
          const int st = J % NST;
          const uint32_t par = ((J / NST) - 1) & 1;
          if (!mbar_wait_bounded(bar(L::KEMPTY + st), par, &s_abort, WAIT_CYCLES)) break;
          load_kv(J, c.su, c.j, true);
          if (!mbar_wait_bounded(bar(L::VEMPTY + st), par, &s_abort, WAIT_CYCLES)) {
            issued = J + 1;  // the K copy of this block is in flight
            break;
          }
          load_kv(J, c.su, c.j, false);
          issued = J + 1;
        }
        if (s_abort) {  // let the copies already issued land before the CTA exits
          volatile int dummy = 0;
          for (int j = max(0, issued - NST); j < issued; ++j) {
            mbar_wait_bounded(bar(L::KFULL + j % NST), (j / NST) & 1, &dummy, DRAIN_CYCLES);
            mbar_wait_bounded(bar(L::VFULL + j % NST), (j / NST) & 1, &dummy, DRAIN_CYCLES);
          }
        }
      }
      __syncwarp();
    } else if (warp >= 2) {
      // ---------------- warps 2-3: each unit's queries into its Q buffer, and
      // the zero rows of nodes >= n_nodes ----------------
      const int t0 = tid - 64;  // 0..63
      int live = 0;
      bool ok = true;
      for (int t = 0; t < n_units && ok; ++t) {
        const StreamUnit su = stream_unit(a, (int)blockIdx.x + t * (int)gridDim.x);
        if (su.bad && t0 == 0) fc_flag(FC_ERR_WORD(a.err), FC_EBIT_INVALID);
        const int pad = a.n_pad - su.nn;
        for (int e = t0; e < a.G * pad * (HD / 8); e += 64) {  // padding rows (all rows of a bad unit)
          const int r = e / (HD / 8), ch = e % (HD / 8);
          const int hh = r / pad, i = su.nn + (r - hh * pad);
          reinterpret_cast<uint4*>(a.out + (((size_t)su.b * a.n_pad + i) * a.H + su.g * a.G + hh) * HD)[ch] =
              make_uint4(0, 0, 0, 0);
        }
        if (su.nblk == 0) continue;
        const int q = live & 1;
        if (live >= 2 && !(ok = warp_wait(bar(L::QFREE + q), ((live >> 1) - 1) & 1, &s_abort))) break;
        if (!(t == 0 && q_pre)) stage_q(su, q);
        cp_async_wait_all();
        fence_proxy_async_smem();
        mbar_arrive(bar(L::QFULL + q));
        ++live;
      }
    } else {
      // ---------------- MMA issuer (+ padding V rows of tree blocks zeroed) -------
      constexpr uint32_t IDESC_QK = idesc_bf16_f32(BM, BN, 0);
      constexpr uint32_t IDESC_PV = idesc_bf16_f32(BM, HD, 1);
      bool ok = true;
      // S buffer J & 1 <- Q buffer q . K(stage J % NST)^T
      auto issue_qk = [&](int J, int q) {
        const uint32_t kb = sK + (J % NST) * TILE_BYTES, qb = sQ + q * L::QTILE;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          tc_mma_f16(tmem + (J & 1) * 128, smem_desc_sw128(qb + (kk >> 2) * L::QHALF + (kk & 3) * 32, 16, 1024),
                     smem_desc_sw128(kb + (kk >> 2) * HALF_BYTES + (kk & 3) * 32, 16, 1024), IDESC_QK, kk > 0);
        }
        tc_commit(bar(L::SFULL + (J & 1)));
      };
      // the QK of the block under cursor c (global index J), once its Q and K are there
      auto qk_step = [&](const StreamCursor& c, int J) -> bool {
        const int q = c.live & 1;
        if (c.j == 0 && !warp_wait(bar(L::QFULL + q), (c.live >> 1) & 1, &s_abort)) return false;
        if (!warp_wait(bar(L::KFULL + J % NST), (J / NST) & 1, &s_abort)) return false;
        tc_fence_after();
        issue_qk(J, q);
        tc_commit(bar(L::KEMPTY + J % NST));
        if (c.j == c.su.nblk - 1) tc_commit(bar(L::QFREE + q));  // the unit's last QK: its Q buffer frees
        return true;
      };
      StreamCursor cq, cp;
      cq.start(a, n_units);
      cp = cq;
      int Jq = 0;
      for (; ok && Jq < 2 && cq.valid(); ++Jq, cq.next(a)) ok = qk_step(cq, Jq);
      for (int J = 0; ok && cp.valid(); ++J, cp.next(a)) {
        const int st = J % NST, o = cp.live & 1;
        if (!(ok = warp_wait(bar(L::VFULL + st), (J / NST) & 1, &s_abort))) break;
        {  // never let garbage (possibly NaN) V rows meet a zero probability: the
           // cache's rows past kv_len and the tree's rows past n_nodes (the tree
           // tile's rows >= n_pad arrived as zeros)
          const bool tree = cp.j >= cp.su.nblk_c;
          const int nv = tree ? cp.su.nn : min(BN, cp.su.kvl - cp.j * BN);
          const int top = tree ? a.n_pad : BN;
          if (nv < top) {
            unsigned char* vt = smem + L::OFF_V + st * TILE_BYTES;
            for (int e = lane; e < (top - nv) * 16; e += 32) {
              const int r = nv + (e >> 4), ch = e & 15;
              *reinterpret_cast<uint4*>(vt + (ch >> 3) * HALF_BYTES + r * 128 + (ch & 7) * 16) =
                  make_uint4(0, 0, 0, 0);
            }
            fence_proxy_async_smem();
          }
          __syncwarp();
        }
        if (!(ok = warp_wait(bar(L::PFULL + (J & 1)), (J >> 1) & 1, &s_abort))) break;
        // a unit's first PV overwrites its O buffer: the unit two back must be read out
        if (cp.j == 0 && cp.live >= 2 && !(ok = warp_wait(bar(L::OFREE + o), ((cp.live >> 1) - 1) & 1, &s_abort)))
          break;
        tc_fence_after();
        {
          const uint32_t vb = sV + st * TILE_BYTES;
#pragma unroll
          for (int kk = 0; kk < BN / 16; ++kk)  // 8 packed columns per 16 keys
            tc_mma_f16_tmem_a(tmem + 256 + o * 128, tmem + (J & 1) * 128 + kk * 8,
                              smem_desc_sw128(vb + kk * 2048, HALF_BYTES, 1024), IDESC_PV, (cp.j > 0 || kk > 0));
        }
        tc_commit(bar(L::ODONE));
        tc_commit(bar(L::VEMPTY + st));
        if (cp.j == cp.su.nblk - 1) tc_commit(bar(L::OFIN + o));
        if (cq.valid()) {  // QK two blocks ahead, into the S buffer PV(J) has just read
          ok = qk_step(cq, Jq);
          ++Jq;
          cq.next(a);
        }
      }
      if (__any_sync(0xFFFFFFFFu, s_abort)) {  // let issued MMAs retire before the tensor memory is freed
        tc_commit(bar(L::DRAIN));
        volatile int dummy = 0;
        mbar_wait_bounded(bar(L::DRAIN), 0, &dummy, DRAIN_CYCLES);
      }
    }
  } else {
    if (warp < 8) {
      regs_inc<REGS_SOFTMAX>();
      // ---------------- softmax warpgroup: thread = row of the unit's tile ----------------
      const int q4 = warp & 3;
      const int r = q4 * 32 + lane;
      const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
      StreamCursor c;
      c.start(a, n_units);
      bool ok = true;
      const int nw = a.n_pad / 64;
      bool row_ok = false;
      __nv_bfloat16* dst = nullptr;
      uint64_t m0 = 0, m1 = 0;
      float m_run = -INFINITY, l_run = 0.f;
      // A unit's output is written once the next unit's first P is handed
      // over: its last PV then runs while this warpgroup already works on the
      // next unit's scores, instead of being waited for.
      bool pend = false, pend_row_ok = false;
      int pend_o = 0;
      uint32_t pend_par = 0;
      float pend_l = 1.f;
      __nv_bfloat16* pend_dst = nullptr;
      auto flush = [&]() -> bool {  // the pending unit's O: normalise, store, free the buffer
        if (!pend) return true;
        pend = false;
        if (!warp_wait(bar(L::OFIN + pend_o), pend_par, &s_abort)) return false;
        tc_fence_after();
        const uint32_t tP = tmem + 256 + pend_o * 128 + lane_off;
        const float inv = 1.f / pend_l;
#pragma unroll
        for (int cc = 0; cc < HD / 32; ++cc) {
          uint32_t ov[32];
          tmem_ld32(tP + cc * 32, ov);
          tc_wait_ld();
          if (pend_row_ok) {
#pragma unroll
            for (int u = 0; u < 32; u += 8) {
              uint4 v;
              v.x = pack_bf16x2(__uint_as_float(ov[u + 0]) * inv, __uint_as_float(ov[u + 1]) * inv);
              v.y = pack_bf16x2(__uint_as_float(ov[u + 2]) * inv, __uint_as_float(ov[u + 3]) * inv);
              v.z = pack_bf16x2(__uint_as_float(ov[u + 4]) * inv, __uint_as_float(ov[u + 5]) * inv);
              v.w = pack_bf16x2(__uint_as_float(ov[u + 6]) * inv, __uint_as_float(ov[u + 7]) * inv);
              *reinterpret_cast<uint4*>(pend_dst + cc * 32 + u) = v;
            }
          }
        }
        tc_fence_before();
        mbar_arrive(bar(L::OFREE + pend_o));
        return true;
      };
      for (int J = 0; ok && c.valid(); ++J, c.next(a)) {
        const int o = c.live & 1;
        const uint32_t tO = tmem + 256 + o * 128 + lane_off;
        if (c.j == 0) {  // a new unit: its row, mask row (first read in its last block) and running state
          row_ok = r < a.G * c.su.nn;
          const int hh = row_ok ? r / c.su.nn : 0, i = row_ok ? r - hh * c.su.nn : 0;
          dst = a.out + (((size_t)c.su.b * a.n_pad + i) * a.H + c.su.g * a.G + hh) * HD;
          const uint64_t* mrow = a.mask + ((size_t)c.su.b * a.n_pad + i) * nw;
          m0 = mrow[0];
          m1 = (nw > 1) ? mrow[1] : 0ull;
          m_run = -INFINITY;
          l_run = 0.f;
        }
        const int sb = J & 1;
        const uint32_t tS = tmem + sb * 128 + lane_off;
        if (!(ok = warp_wait(bar(L::SFULL + sb), (J >> 1) & 1, &s_abort))) break;
        tc_fence_after();
        const bool tree = c.j == c.su.nblk - 1;
        if (q4 * 32 >= L::QROWS) {  // lanes past the Q buffer's rows: no output row, keep the phases only
          tc_fence_before();
          mbar_arrive(bar(L::PFULL + sb));
          if (tree) {
            if (!(ok = warp_wait(bar(L::OFIN + o), (c.live >> 1) & 1, &s_abort))) break;
            tc_fence_after();
            tc_fence_before();
            mbar_arrive(bar(L::OFREE + o));
          }
          continue;
        }
        const int nv = tree ? BN : min(BN, c.su.kvl - c.j * BN);
        const bool masked = tree || nv < BN;  // block-uniform
        auto keep_bits = [&](int q) -> uint32_t {
          if (tree) return (uint32_t)((q < 2 ? m0 : m1) >> (32 * (q & 1)));
          const int lo = nv - 32 * q;
          return lo >= 32 ? 0xFFFFFFFFu : (lo <= 0 ? 0u : ((1u << lo) - 1u));
        };
        uint32_t sv[128];
#pragma unroll
        for (int c4 = 0; c4 < 4; ++c4) tmem_ld32(tS + c4 * 32, *reinterpret_cast<uint32_t(*)[32]>(&sv[c4 * 32]));
        tc_wait_ld();
        if (masked) {
#pragma unroll
          for (int c4 = 0; c4 < 4; ++c4) {
            const uint32_t kbits = keep_bits(c4);
#pragma unroll
            for (int cc = 0; cc < 32; ++cc)
              if (!(kbits & (1u << cc))) sv[c4 * 32 + cc] = __float_as_uint(-INFINITY);
          }
        }
        float pm[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) pm[u] = -INFINITY;
#pragma unroll
        for (int cc = 0; cc < 128; cc += 2)
          pm[(cc >> 1) & 7] = fmax3(pm[(cc >> 1) & 7], __uint_as_float(sv[cc]), __uint_as_float(sv[cc + 1]));
        const float mx = fmaxf(fmaxf(fmaxf(pm[0], pm[1]), fmaxf(pm[2], pm[3])),
                               fmaxf(fmaxf(pm[4], pm[5]), fmaxf(pm[6], pm[7]))) * a.scale_log2;
        const float m_new = (mx > m_run + RESCALE_THRESHOLD) ? mx : m_run;
        const float m_use = (m_new == -INFINITY) ? 0.f : m_new;
        const float alpha = fast_exp2(m_run - m_use);
        // PV of the unit's previous block may still run: wait for it
        if (c.j > 0 && __any_sync(0xFFFFFFFFu, alpha != 1.f)) {
          if (!(ok = warp_wait(bar(L::ODONE), (J - 1) & 1, &s_abort))) break;
          tc_fence_after();
#pragma unroll
          for (int cc = 0; cc < HD / 32; ++cc) {
            uint32_t ov[32];
            tmem_ld32(tO + cc * 32, ov);
            tc_wait_ld();
#pragma unroll
            for (int u = 0; u < 32; ++u) ov[u] = __float_as_uint(__uint_as_float(ov[u]) * alpha);
            tmem_st32(tO + cc * 32, ov);
          }
        }
        uint64_t ps2[4] = {0ull, 0ull, 0ull, 0ull};
        const uint64_t sc2 = f2_pack(a.scale_log2, a.scale_log2), nm2 = f2_pack(-m_use, -m_use);
#pragma unroll
        for (int c4 = 0; c4 < 4; ++c4) {
          uint32_t pk[16];
#pragma unroll
          for (int qq = 0; qq < 16; ++qq) {
            const int cc = c4 * 32 + 2 * qq;
            float x0, x1;
            f2_unpack(f2_fma(f2_pack(__uint_as_float(sv[cc]), __uint_as_float(sv[cc + 1])), sc2, nm2), x0, x1);
            const float p0 = fast_exp2(x0), p1 = fast_exp2(x1);
            ps2[qq & 3] = f2_add(ps2[qq & 3], f2_pack(p0, p1));
            pk[qq] = pack_bf16x2(p0, p1);
          }
          tmem_st16(tS + c4 * 16, pk);
        }
        tc_wait_st();
        float ps[8];
        f2_unpack(ps2[0], ps[0], ps[1]);
        f2_unpack(ps2[1], ps[2], ps[3]);
        f2_unpack(ps2[2], ps[4], ps[5]);
        f2_unpack(ps2[3], ps[6], ps[7]);
        const float sum = ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
        l_run = l_run * alpha + sum;
        m_run = m_new;
        tc_fence_before();
        mbar_arrive(bar(L::PFULL + sb));
        if (c.j == 0 && !(ok = flush())) break;  // the previous unit's output
        if (tree) {  // the unit's last block: its output follows the next unit's first P
          pend = true;
          pend_o = o;
          pend_par = (c.live >> 1) & 1;
          pend_l = l_run;
          pend_row_ok = row_ok;
          pend_dst = dst;
        }
      }
      if (ok) ok = flush();  // the last unit's output
    }
  }
  tc_fence_before();
  __syncthreads();
  if (tid == 0 && s_abort) fc_flag(FC_ERR_WORD(a.err), FC_EBIT_TIMEOUT);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// bf16 tensor [outer][rows][128] as a 3-D map with a (64, box_rows, 1) box.
bool make_map(CUtensorMap* m, const void* base, uint64_t rows, uint64_t outer, uint32_t box_rows) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)HD, (cuuint64_t)rows, (cuuint64_t)outer};
  cuuint64_t strides[2] = {(cuuint64_t)HD * 2, (cuuint64_t)rows * HD * 2};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Workspace layout for `parts` KV parts per unit (units = batch * Hkv * row chunks).
struct WsLayout {
  size_t cnt, ml, o, total;
};
WsLayout ws_layout(uint64_t units, int parts) {
  WsLayout w;
  const uint64_t slots = units * (uint64_t)parts * (TILES * BM);
  w.cnt = 0;
  w.ml = (units * 2 * sizeof(int) + 255) / 256 * 256;
  w.o = w.ml + (slots * sizeof(float2) + 255) / 256 * 256;
  w.total = w.o + slots * HD * sizeof(float);
  return w;
}

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 0;
  return n;
}

// Tail split: with U units on P SMs, the first U - R units (R = U mod P)
// fill whole waves and run unsplit; the R units of the last, partial wave are
// split into the most parts that still fit one wave (R * parts <= P), as long
// as each part keeps at least MIN_PART_BLOCKS blocks (the block count is
// bounded by kv_cap; the actual lengths live on the device) and the
// workspace holds their partial sums.
constexpr int MIN_PART_BLOCKS = 8;
struct SplitPlan {
  uint64_t u_split;
  int parts;
};
SplitPlan choose_split(uint64_t units, int kv_cap, size_t ws_bytes) {
  SplitPlan sp{units, 1};
  const int sms = sm_count();
  if (sms <= 0 || units <= (uint64_t)sms) return sp;
  const uint64_t rem = units % (uint64_t)sms;
  if (rem == 0) return sp;
  const int nb = (kv_cap + BN - 1) / BN + 1;
  int parts = (int)std::min<uint64_t>((uint64_t)MAX_PARTS, (uint64_t)sms / rem);
  parts = std::min(parts, nb / MIN_PART_BLOCKS);
  while (parts > 1 && ws_bytes < ws_layout(rem, parts).total) --parts;
  if (parts > 1) sp = SplitPlan{units - rem, parts};
  return sp;
}

// Which kernel serves a launch of one-tile units (G * n_pad <= 128, caches
// of at most STREAM_MAX_KV keys; RoPE launches keep the per-unit kernel).
// Per-unit CTAs pay a unit's set-up and epilogue, about
// STREAM_OVERHEAD_BLOCKS blocks' time, on top of its nb blocks; streaming
// CTAs pay them once but each serves ceil(units / SMs) whole units, where
// per-unit CTAs spread units / SMs (and split the last wave's keys).  The
// streaming kernel is chosen when its estimate is no longer.
constexpr int STREAM_MAX_KV = 4096;
constexpr int STREAM_OVERHEAD_BLOCKS = 3;
bool use_stream(uint64_t units, int G, int n_pad, int kv_cap, bool rope) {
  if (rope || G * n_pad > BM || kv_cap > STREAM_MAX_KV) return false;
  const int sms = sm_count();
  if (sms <= 0 || units <= (uint64_t)sms) return false;
  const uint64_t nb = (uint64_t)(kv_cap + BN - 1) / BN + 1;
  const uint64_t waves = (units + sms - 1) / sms;
  return waves * nb * (uint64_t)sms <= units * (nb + STREAM_OVERHEAD_BLOCKS);
}

uint64_t attn_units(int batch, int n_pad, int H, int Hkv) {
  return (uint64_t)batch * Hkv * (((uint64_t)(H / Hkv) * n_pad + TILES * BM - 1) / (TILES * BM));
}

// fc_rope: rows of bf16 vectors rotated by their node's position.  layout 0
// is node-major [B][n_pad][heads][D] (queries), layout 1 head-major
// [B][heads][n_pad][D] (tree keys).  One thread per pair of partner chunks.
__global__ void k_rope(const uint4* __restrict__ in, uint4* __restrict__ out, int B, int n_pad, int heads, int D,
                       int layout, const int32_t* __restrict__ pos, double nl2f) {
  __shared__ float2 tab[FC_ROPE_MAX_HALF];
  fc_rope_table(tab, D / 2, nl2f);
  __syncthreads();
  const int ch = D / 16;  // 16-byte chunks per half row
  const size_t items = (size_t)B * n_pad * heads * ch;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < items; e += (size_t)gridDim.x * blockDim.x) {
    const int gran = (int)(e % ch);
    const size_t row = e / ch;
    int bb, i;
    if (layout == 0) {
      const size_t bi = row / heads;
      bb = (int)(bi / n_pad);
      i = (int)(bi % n_pad);
    } else {
      i = (int)(row % n_pad);
      bb = (int)(row / ((size_t)heads * n_pad));
    }
    const uint4* src = in + row * (D / 8);
    uint4 lo = src[gran], hi = src[gran + ch];
    const int p = pos[(size_t)bb * n_pad + i];
    if (p >= 0) rope_chunks(lo, hi, (float)p, tab, 8 * gran);
    out[row * (D / 8) + gran] = lo;
    out[row * (D / 8) + gran + ch] = hi;
  }
}

}  // namespace

extern "C" size_t fc_tree_attn_workspace(int batch, int n_pad, int H, int Hkv) {
  if (batch < 1 || H < 1 || Hkv < 1 || H % Hkv != 0 || (n_pad != 64 && n_pad != 128)) return 0;
  // only the units of the last partial wave are ever split (fewer than the SM count)
  const uint64_t units = attn_units(batch, n_pad, H, Hkv);
  const int sms = sm_count();
  return ws_layout(std::min<uint64_t>(units, (uint64_t)std::max(sms, 1)), MAX_PARTS).total;
}

extern "C" int fc_tree_attn_streamed(int batch, int n_pad, int H, int Hkv, int kv_cap) {
  if (batch < 1 || H < 1 || Hkv < 1 || kv_cap < 1 || H % Hkv != 0 || (n_pad != 64 && n_pad != 128)) return 0;
  return use_stream(attn_units(batch, n_pad, H, Hkv), H / Hkv, n_pad, kv_cap, false) ? 1 : 0;
}

extern "C" int fc_tree_attn_parts(int batch, int n_pad, int H, int Hkv, int kv_cap, size_t ws_bytes) {
  if (batch < 1 || H < 1 || Hkv < 1 || kv_cap < 1 || H % Hkv != 0 || (n_pad != 64 && n_pad != 128)) return 0;
  const uint64_t units = attn_units(batch, n_pad, H, Hkv);
  if (use_stream(units, H / Hkv, n_pad, kv_cap, false)) return 1;  // no key split there
  return choose_split(units, kv_cap, ws_bytes).parts;
}

static fc_status launch_tree_attn(const void* d_q, const void* d_k_cache, const void* d_v_cache, int kv_cap,
                                  const int32_t* d_kv_len, const void* d_k_tree, const void* d_v_tree,
                                  const uint64_t* d_mask, const int32_t* d_n_nodes, int batch, int n_pad, int H,
                                  int Hkv, int D, float scale, void* d_out, void* d_ws, size_t ws_bytes,
                                  const int32_t* d_pos, float rope_base, fc_stream stream) {
  if (batch < 0 || H < 1 || Hkv < 1 || kv_cap < 1) return FC_ERR_INVALID_ARG;
  if (D != HD || (n_pad != 64 && n_pad != 128) || H % Hkv != 0 || H / Hkv > 16) return FC_ERR_UNSUPPORTED;
  if (!(scale > 0.f)) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_q || !d_k_cache || !d_v_cache || !d_kv_len || !d_k_tree || !d_v_tree || !d_mask || !d_n_nodes || !d_out)
    return FC_ERR_INVALID_ARG;
  const uintptr_t al = reinterpret_cast<uintptr_t>(d_q) | reinterpret_cast<uintptr_t>(d_k_cache) |
                       reinterpret_cast<uintptr_t>(d_v_cache) | reinterpret_cast<uintptr_t>(d_k_tree) |
                       reinterpret_cast<uintptr_t>(d_v_tree) | reinterpret_cast<uintptr_t>(d_out) |
                       reinterpret_cast<uintptr_t>(d_ws);
  if (al % 16 || reinterpret_cast<uintptr_t>(d_mask) % 8) return FC_ERR_INVALID_ARG;
  const uint64_t groups = (uint64_t)batch * Hkv;
  const int G = H / Hkv;
  const int ctas = (G * n_pad + TILES * BM - 1) / (TILES * BM);
  const uint64_t units = attn_units(batch, n_pad, H, Hkv);
  const bool streamed = use_stream(units, G, n_pad, kv_cap, d_pos != nullptr);
  const SplitPlan sp = streamed ? SplitPlan{units, 1} : choose_split(units, kv_cap, d_ws ? ws_bytes : 0);
  const uint64_t n_split = units - sp.u_split;
  const uint64_t grid = streamed ? (uint64_t)sm_count() : sp.u_split + n_split * sp.parts;
  if (grid > 0x7FFFFFFFull) return FC_ERR_UNSUPPORTED;
  CUtensorMap mkc, mvc, mkt, mvt;
  if (!make_map(&mkc, d_k_cache, (uint64_t)kv_cap, groups, BN) || !make_map(&mvc, d_v_cache, (uint64_t)kv_cap, groups, BN) ||
      !make_map(&mkt, d_k_tree, (uint64_t)n_pad, groups, BN) || !make_map(&mvt, d_v_tree, (uint64_t)n_pad, groups, BN))
    return FC_ERR_CUDA;
  // the streaming kernel keeps three K/V stages when a group's rows fit 64
  const bool three = streamed && G * n_pad <= 64;
  auto kern = streamed ? (three ? k_tree_attn_stream<3> : k_tree_attn_stream<2>)
                       : (d_pos ? k_tree_attn<true> : k_tree_attn<false>);
  const uint32_t smem_bytes = streamed ? (three ? StreamLayout<3>::SMEM : StreamLayout<2>::SMEM) : SMEM_BYTES;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_bytes) != cudaSuccess)
    return FC_ERR_CUDA;
  {  // the register split needs the whole launch allocation (see REGS_LAUNCH)
    cudaFuncAttributes fa;
    if (cudaFuncGetAttributes(&fa, kern) != cudaSuccess) return FC_ERR_CUDA;
    if (fa.numRegs < REGS_LAUNCH) return FC_ERR_INTERNAL;
  }
  AttnArgs a;
  a.q = static_cast<const __nv_bfloat16*>(d_q);
  a.kv_len = d_kv_len;
  a.mask = d_mask;
  a.n_nodes = d_n_nodes;
  a.out = static_cast<__nv_bfloat16*>(d_out);
  a.B = batch;
  a.n_pad = n_pad;
  a.H = H;
  a.Hkv = Hkv;
  a.G = G;
  a.kv_cap = kv_cap;
  a.ctas = ctas;
  a.u_split = (int)sp.u_split;
  a.parts = sp.parts;
  a.scale_log2 = scale * 1.4426950408889634f;
  a.ws_cnt = nullptr;
  a.ws_ml = nullptr;
  a.ws_o = nullptr;
  a.err = fc_error_slot();
  a.pos = d_pos;
  a.rope_nl2f = d_pos ? -2.0 * std::log2((double)rope_base) / HD : 0.0;
  if (sp.parts > 1) {
    const WsLayout w = ws_layout(n_split, sp.parts);
    unsigned char* base = static_cast<unsigned char*>(d_ws);
    a.ws_cnt = reinterpret_cast<int*>(base + w.cnt);
    a.ws_ml = reinterpret_cast<float2*>(base + w.ml);
    a.ws_o = reinterpret_cast<float*>(base + w.o);
    if (cudaMemsetAsync(a.ws_cnt, 0, n_split * 2 * sizeof(int), static_cast<cudaStream_t>(stream)) != cudaSuccess)
      return FC_ERR_CUDA;
  }
  kern<<<(unsigned)grid, TA_THREADS, smem_bytes, static_cast<cudaStream_t>(stream)>>>(mkc, mvc, mkt, mvt, a);
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_tree_attn(const void* d_q, const void* d_k_cache, const void* d_v_cache, int kv_cap,
                                  const int32_t* d_kv_len, const void* d_k_tree, const void* d_v_tree,
                                  const uint64_t* d_mask, const int32_t* d_n_nodes, int batch, int n_pad, int H, int Hkv,
                                  int D, float scale, void* d_out, void* d_ws, size_t ws_bytes, fc_stream stream) {
  FC_NVTX_RANGE();
  return launch_tree_attn(d_q, d_k_cache, d_v_cache, kv_cap, d_kv_len, d_k_tree, d_v_tree, d_mask, d_n_nodes, batch,
                          n_pad, H, Hkv, D, scale, d_out, d_ws, ws_bytes, nullptr, 0.f, stream);
}

extern "C" fc_status fc_tree_attn_rope(const void* d_q, const void* d_k_cache, const void* d_v_cache, int kv_cap,
                                       const int32_t* d_kv_len, const void* d_k_tree, const void* d_v_tree,
                                       const uint64_t* d_mask, const int32_t* d_n_nodes, int batch, int n_pad, int H,
                                       int Hkv, int D, float scale, const int32_t* d_pos, float rope_base,
                                       void* d_out, void* d_ws, size_t ws_bytes, fc_stream stream) {
  FC_NVTX_RANGE();
  if (!(rope_base > 0.f) || !std::isfinite(rope_base)) return FC_ERR_INVALID_ARG;
  if (batch > 0 && !d_pos) return FC_ERR_INVALID_ARG;
  return launch_tree_attn(d_q, d_k_cache, d_v_cache, kv_cap, d_kv_len, d_k_tree, d_v_tree, d_mask, d_n_nodes, batch,
                          n_pad, H, Hkv, D, scale, d_out, d_ws, ws_bytes, d_pos, rope_base, stream);
}

extern "C" fc_status fc_rope(const void* d_in, void* d_out, int batch, int n_pad, int heads, int D, int layout,
                             const int32_t* d_pos, float base, fc_stream stream) {
  FC_NVTX_RANGE();
  if (batch < 0 || n_pad < 1 || heads < 1 || D < 16 || D > 1024 || D % 16 || (layout != 0 && layout != 1))
    return FC_ERR_INVALID_ARG;
  if (!(base > 0.f) || !std::isfinite(base)) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_in || !d_out || !d_pos) return FC_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(d_in) | reinterpret_cast<uintptr_t>(d_out)) % 16) return FC_ERR_INVALID_ARG;
  const size_t items = (size_t)batch * n_pad * heads * (D / 16);
  const unsigned blocks = (unsigned)std::min<size_t>((items + 255) / 256, 152 * 16);
  k_rope<<<blocks, 256, 0, static_cast<cudaStream_t>(stream)>>>(static_cast<const uint4*>(d_in),
                                                                static_cast<uint4*>(d_out), batch, n_pad, heads, D,
                                                                layout, d_pos, -2.0 * std::log2((double)base) / D);
  return FC_CHECK_LAUNCH();
}
