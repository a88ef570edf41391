// fc_tree_attn: tree-masked verification attention (Section IV-D, Eq. 4).
// Every draft-tree node attends to the whole KV cache of its sequence and to
// its tree ancestors (and itself), so one forward verifies every draft.
//
// GB300 design (one CTA = 128 query rows of one (sequence, kv head) group):
//   * GQA packing: the rows of a CTA are (query head in group, tree node)
//     pairs over the group's H/Hkv heads and the sequence's n_nodes nodes,
//     packed densely, so small trees do not waste tensor-core rows and every
//     K/V tile loaded serves all heads that share it.
//   * K/V tiles of 128 keys x 128 dims stream from HBM with TMA (128-byte
//     swizzle, two stages); the tree's own K/V form one last tile.
//   * S = Q K^T and O += P V run on the 5th-generation tensor cores
//     (tcgen05.mma, bf16 in, fp32 accumulate) with S (double-buffered) and O
//     in tensor memory; one thread issues the MMAs.
//   * a 128-thread softmax warpgroup owns one row per thread: it reads S
//     from tensor memory, applies the tree mask bits (and the ragged cache
//     tail) in registers, runs the online softmax in base 2, rescales O in
//     tensor memory, and writes P (bf16) to shared memory for the PV MMA.
//   * QK of block j+1 and PV of block j-1 overlap the softmax of block j.
//   * every mbarrier wait is bounded; a wait that runs out raises
//     FC_ERR_TIMEOUT, the CTA drains its in-flight copies and MMAs (bounded
//     again), frees its tensor memory and returns.
#include <algorithm>
#include <mutex>

#include "fc_common.cuh"

FC_DEFINE_ERROR_WORD(attn)

namespace {

constexpr int TA_THREADS = 256;
constexpr int BM = 128;  // query rows per CTA
constexpr int BN = 128;  // keys per block
constexpr int HD = 128;  // head dim
constexpr uint32_t HALF_BYTES = BN * 64 * 2;  // one 64-dim half of a 128-row tile
constexpr uint32_t TILE_BYTES = 2 * HALF_BYTES;
constexpr uint32_t OFF_Q = 0;
constexpr uint32_t OFF_K = OFF_Q + TILE_BYTES;
constexpr uint32_t OFF_V = OFF_K + 2 * TILE_BYTES;
constexpr uint32_t OFF_P = OFF_V + 2 * TILE_BYTES;
constexpr uint32_t OFF_BAR = OFF_P + TILE_BYTES;
constexpr uint32_t SMEM_BYTES = OFF_BAR + 256 + 1024;  // + alignment slack
constexpr uint32_t TMEM_COLS = 512;
constexpr uint64_t WAIT_NS = 4000000000ull;   // ~2 s of SM clock cycles
constexpr uint64_t DRAIN_NS = 400000000ull;   // ~0.2 s
// Lazy rescaling: O and l are rescaled only when a row's running maximum
// (base-2 logits) grows by more than this; until then probabilities may reach
// 2^RESCALE_THRESHOLD, harmless in bf16/fp32.
constexpr float RESCALE_THRESHOLD = 8.f;

// barrier slots (8 bytes each) after OFF_BAR
enum { B_KFULL = 0, B_VFULL = 2, B_EMPTY = 4, B_SFULL = 6, B_PFULL = 8, B_ODONE = 9, N_BARS = 10 };

struct AttnArgs {
  const __nv_bfloat16* q;
  const int32_t* kv_len;
  const uint64_t* mask;
  const int32_t* n_nodes;
  __nv_bfloat16* out;
  int B, n_pad, H, Hkv, G, kv_cap, tiles;
  float scale_log2;
};

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__global__ void __launch_bounds__(TA_THREADS, 1)
    k_tree_attn(const __grid_constant__ CUtensorMap tm_kc, const __grid_constant__ CUtensorMap tm_vc,
                const __grid_constant__ CUtensorMap tm_kt, const __grid_constant__ CUtensorMap tm_vt, AttnArgs a) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int bg = blockIdx.x / a.tiles, t = blockIdx.x - bg * a.tiles;
  const int b = bg / a.Hkv, g = bg - b * a.Hkv;
  const int nn_raw = a.n_nodes[b], kvl = a.kv_len[b];
  const bool bad = nn_raw < 1 || nn_raw > a.n_pad || kvl < 0 || kvl > a.kv_cap;
  const int nn = bad ? 0 : nn_raw;
  if (bad && t == 0 && tid == 0) fc_flag(&g_fc_err, FC_EBIT_INVALID);

  // Zero the padding rows (nodes >= n_nodes) of this group; tiles share the work.
  {
    const int pad_rows = a.G * (a.n_pad - nn);
    for (int e = t * TA_THREADS + tid; e < pad_rows * (HD / 8); e += a.tiles * TA_THREADS) {
      int r = e / (HD / 8), ch = e - r * (HD / 8);
      int hh = r / (a.n_pad - nn), i = nn + (r - hh * (a.n_pad - nn));
      uint4* dst = reinterpret_cast<uint4*>(a.out + (((size_t)b * a.n_pad + i) * a.H + g * a.G + hh) * HD) + ch;
      *dst = make_uint4(0, 0, 0, 0);
    }
  }
  const int rows_total = a.G * nn;
  const int row0 = t * BM;
  if (row0 >= rows_total) return;

  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase + OFF_Q, sK = sbase + OFF_K, sV = sbase + OFF_V, sP = sbase + OFF_P;
  const uint32_t bar0 = sbase + OFF_BAR;
  auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };

  const int nblk_c = (kvl + BN - 1) / BN;
  const int nblk = nblk_c + 1;  // + the tree block

  if (tid == 0) {
    s_abort = 0;
    for (int i = 0; i < N_BARS; ++i) mbar_init(bar(i), i == B_PFULL ? 128u : 1u);
    fence_mbar_init();
    prefetch_tmap(&tm_kc);
    prefetch_tmap(&tm_vc);
    prefetch_tmap(&tm_kt);
    prefetch_tmap(&tm_vt);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), TMEM_COLS);
    tmem_relinquish();
  }
  // Q tile: rows (head in group, node) packed densely, 128-byte swizzled, K-major.
  for (int c = tid; c < BM * 16; c += TA_THREADS) {
    const int r = c >> 4, ch = c & 15, half = ch >> 3, gran = ch & 7;
    const int rg = row0 + r;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (rg < rows_total) {
      const int hh = rg / nn, i = rg - hh * nn;
      v = *(reinterpret_cast<const uint4*>(a.q + (((size_t)b * a.n_pad + i) * a.H + g * a.G + hh) * HD) + ch);
    }
    *reinterpret_cast<uint4*>(smem + OFF_Q + half * HALF_BYTES + r * 128 + ((gran ^ (r & 7)) << 4)) = v;
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  const uint32_t tS0 = tmem, tO = tmem + 256;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      int issued = 0;
      for (int j = 0; j < nblk; ++j) {
        const int st = j & 1;
        if (j >= 2 && !mbar_wait_bounded(bar(B_EMPTY + st), ((j >> 1) - 1) & 1, &s_abort, WAIT_NS)) break;
        const uint32_t dK = sK + st * TILE_BYTES, dV = sV + st * TILE_BYTES;
        if (j < nblk_c) {
          mbar_expect_tx(bar(B_KFULL + st), TILE_BYTES);
          tma_load_3d(dK, &tm_kc, 0, j * BN, bg, bar(B_KFULL + st));
          tma_load_3d(dK + HALF_BYTES, &tm_kc, 64, j * BN, bg, bar(B_KFULL + st));
          mbar_expect_tx(bar(B_VFULL + st), TILE_BYTES);
          tma_load_3d(dV, &tm_vc, 0, j * BN, bg, bar(B_VFULL + st));
          tma_load_3d(dV + HALF_BYTES, &tm_vc, 64, j * BN, bg, bar(B_VFULL + st));
        } else {
          const uint32_t bytes = (uint32_t)a.n_pad * 64 * 2 * 2;
          mbar_expect_tx(bar(B_KFULL + st), bytes);
          tma_load_3d(dK, &tm_kt, 0, 0, bg, bar(B_KFULL + st));
          tma_load_3d(dK + HALF_BYTES, &tm_kt, 64, 0, bg, bar(B_KFULL + st));
          mbar_expect_tx(bar(B_VFULL + st), bytes);
          tma_load_3d(dV, &tm_vt, 0, 0, bg, bar(B_VFULL + st));
          tma_load_3d(dV + HALF_BYTES, &tm_vt, 64, 0, bg, bar(B_VFULL + st));
        }
        issued = j + 1;
      }
      if (s_abort) {  // let the copies already issued land before the CTA exits
        volatile int dummy = 0;
        for (int j = max(0, issued - 2); j < issued; ++j) {
          mbar_wait_bounded(bar(B_KFULL + (j & 1)), (j >> 1) & 1, &dummy, DRAIN_NS);
          mbar_wait_bounded(bar(B_VFULL + (j & 1)), (j >> 1) & 1, &dummy, DRAIN_NS);
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer (+ ragged V rows zeroed by the warp) -------
    constexpr uint32_t IDESC_QK = idesc_bf16_f32(BM, BN, 0);
    constexpr uint32_t IDESC_PV = idesc_bf16_f32(BM, HD, 1);
    int last_qk = -1, last_pv = -1;
    for (int j = 0; j <= nblk; ++j) {
      if (j < nblk) {
        const int st = j & 1;
        if (!__all_sync(0xFFFFFFFFu, mbar_wait_bounded(bar(B_KFULL + st), (j >> 1) & 1, &s_abort, WAIT_NS))) break;
        if (lane == 0) {
          tc_fence_after();
          const uint32_t kb = sK + st * TILE_BYTES;
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk) {
            const uint32_t off = (kk >> 2) * HALF_BYTES + (kk & 3) * 32;
            tc_mma_f16(tS0 + st * 128, smem_desc_sw128(sQ + off, 16, 1024), smem_desc_sw128(kb + off, 16, 1024),
                       IDESC_QK, kk > 0);
          }
          tc_commit(bar(B_SFULL + st));
        }
        last_qk = j;
        __syncwarp();
      }
      if (j >= 1) {
        const int jj = j - 1, st = jj & 1;
        if (!__all_sync(0xFFFFFFFFu, mbar_wait_bounded(bar(B_PFULL), jj & 1, &s_abort, WAIT_NS))) break;
        if (!__all_sync(0xFFFFFFFFu, mbar_wait_bounded(bar(B_VFULL + st), (jj >> 1) & 1, &s_abort, WAIT_NS))) break;
        const int nv = (jj < nblk_c) ? min(BN, kvl - jj * BN) : nn;
        unsigned char* vt = smem + OFF_V + st * TILE_BYTES;
        if (nv < BN) {  // never let garbage (possibly NaN) rows meet a zero probability
          for (int e = lane; e < (BN - nv) * 16; e += 32) {
            const int r = nv + (e >> 4), ch = e & 15;
            *reinterpret_cast<uint4*>(vt + (ch >> 3) * HALF_BYTES + r * 128 + (ch & 7) * 16) = make_uint4(0, 0, 0, 0);
          }
          fence_proxy_async_smem();
        }
        __syncwarp();
        if (lane == 0) {
          tc_fence_after();
          const uint32_t vb = sV + st * TILE_BYTES;
#pragma unroll
          for (int kk = 0; kk < BN / 16; ++kk) {
            const uint32_t aoff = (kk >> 2) * HALF_BYTES + (kk & 3) * 32;
            tc_mma_f16(tO, smem_desc_sw128(sP + aoff, 16, 1024), smem_desc_sw128(vb + kk * 2048, HALF_BYTES, 1024),
                       IDESC_PV, (jj > 0 || kk > 0));
          }
          tc_commit(bar(B_ODONE));
          tc_commit(bar(B_EMPTY + st));
        }
        last_pv = jj;
        __syncwarp();
      }
    }
    if (s_abort) {  // let issued MMAs retire before the tensor memory is freed
      volatile int dummy = 0;
      if (last_qk >= 0) mbar_wait_bounded(bar(B_SFULL + (last_qk & 1)), (last_qk >> 1) & 1, &dummy, DRAIN_NS);
      if (last_pv >= 0) mbar_wait_bounded(bar(B_ODONE), last_pv & 1, &dummy, DRAIN_NS);
    }
  } else if (warp >= 4) {
    // ---------------- softmax warpgroup: thread = row ----------------
    const int q4 = warp - 4;
    const int r = q4 * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const int rg = row0 + r;
    const bool row_ok = rg < rows_total;
    const int hh = row_ok ? rg / nn : 0, i = row_ok ? rg - hh * nn : 0;
    const int nw = a.n_pad / 64;
    const uint64_t* mrow = a.mask + ((size_t)b * a.n_pad + i) * nw;
    const uint64_t m0 = mrow[0], m1 = (nw > 1) ? mrow[1] : 0ull;
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    uint32_t sreg[BN];
    for (int j = 0; j < nblk && ok; ++j) {
      const int st = j & 1;
      if (!__all_sync(0xFFFFFFFFu, mbar_wait_bounded(bar(B_SFULL + st), (j >> 1) & 1, &s_abort, WAIT_NS))) {
        ok = false;
        break;
      }
      tc_fence_after();
#pragma unroll
      for (int c = 0; c < BN / 32; ++c)
        tmem_ld32(tS0 + st * 128 + c * 32 + lane_off, *reinterpret_cast<uint32_t(*)[32]>(&sreg[c * 32]));
      tc_wait_ld();
      const bool tree = (j == nblk - 1);
      const int nv = tree ? BN : min(BN, kvl - j * BN);
      if (tree || nv < BN) {  // block-uniform: only the ragged tail and the tree block are masked
#pragma unroll
        for (int c = 0; c < BN; ++c) {
          const bool keep = tree ? (((c < 64 ? m0 >> c : m1 >> (c - 64)) & 1ull) != 0) : (c < nv);
          if (!keep) sreg[c] = __float_as_uint(-INFINITY);
        }
      }
      // raw row maximum with independent partial maxima (scale > 0 commutes with max)
      float pm[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) pm[u] = -INFINITY;
#pragma unroll
      for (int c = 0; c < BN; ++c) pm[c & 7] = fmaxf(pm[c & 7], __uint_as_float(sreg[c]));
      const float mx = fmaxf(fmaxf(fmaxf(pm[0], pm[1]), fmaxf(pm[2], pm[3])),
                             fmaxf(fmaxf(pm[4], pm[5]), fmaxf(pm[6], pm[7]))) * a.scale_log2;
      // lazy rescale: keep the old reference unless the maximum grew a lot
      const float m_new = (mx > m_run + RESCALE_THRESHOLD) ? mx : m_run;
      const float m_use = (m_new == -INFINITY) ? 0.f : m_new;
      const float alpha = fast_exp2(m_run - m_use);
      float ps[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) ps[u] = 0.f;
#pragma unroll
      for (int c = 0; c < BN; ++c) {
        const float p = fast_exp2(fmaf(__uint_as_float(sreg[c]), a.scale_log2, -m_use));
        sreg[c] = __float_as_uint(p);
        ps[c & 7] += p;
      }
      const float sum = ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
      l_run = l_run * alpha + sum;
      m_run = m_new;
      if (j >= 1) {  // PV(j-1) must be done before O is rescaled and P overwritten
        if (!__all_sync(0xFFFFFFFFu, mbar_wait_bounded(bar(B_ODONE), (j - 1) & 1, &s_abort, WAIT_NS))) {
          ok = false;
          break;
        }
        tc_fence_after();
        // tcgen05.ld/st are warp-collective: the branch must be warp-uniform.
        if (__any_sync(0xFFFFFFFFu, alpha != 1.f)) {
#pragma unroll
          for (int c = 0; c < HD / 32; ++c) {
            uint32_t o[32];
            tmem_ld32(tO + c * 32 + lane_off, o);
            tc_wait_ld();
#pragma unroll
            for (int x = 0; x < 32; ++x) o[x] = __float_as_uint(__uint_as_float(o[x]) * alpha);
            tmem_st32(tO + c * 32 + lane_off, o);
          }
          tc_wait_st();
        }
      }
      // P row -> shared memory (bf16, 128-byte swizzle, K-major A operand)
#pragma unroll
      for (int ch = 0; ch < 16; ++ch) {
        uint4 v;
        v.x = pack_bf16x2(__uint_as_float(sreg[ch * 8 + 0]), __uint_as_float(sreg[ch * 8 + 1]));
        v.y = pack_bf16x2(__uint_as_float(sreg[ch * 8 + 2]), __uint_as_float(sreg[ch * 8 + 3]));
        v.z = pack_bf16x2(__uint_as_float(sreg[ch * 8 + 4]), __uint_as_float(sreg[ch * 8 + 5]));
        v.w = pack_bf16x2(__uint_as_float(sreg[ch * 8 + 6]), __uint_as_float(sreg[ch * 8 + 7]));
        *reinterpret_cast<uint4*>(smem + OFF_P + (ch >> 3) * HALF_BYTES + r * 128 + (((ch & 7) ^ (r & 7)) << 4)) = v;
      }
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(bar(B_PFULL));
    }
    if (ok && __all_sync(0xFFFFFFFFu, mbar_wait_bounded(bar(B_ODONE), (nblk - 1) & 1, &s_abort, WAIT_NS))) {
      tc_fence_after();
      const float inv = 1.f / l_run;
      __nv_bfloat16* dst = a.out + (((size_t)b * a.n_pad + i) * a.H + g * a.G + hh) * HD;
#pragma unroll
      for (int c = 0; c < HD / 32; ++c) {
        uint32_t o[32];
        tmem_ld32(tO + c * 32 + lane_off, o);
        tc_wait_ld();
        if (row_ok) {
#pragma unroll
          for (int x = 0; x < 32; x += 8) {
            uint4 v;
            v.x = pack_bf16x2(__uint_as_float(o[x + 0]) * inv, __uint_as_float(o[x + 1]) * inv);
            v.y = pack_bf16x2(__uint_as_float(o[x + 2]) * inv, __uint_as_float(o[x + 3]) * inv);
            v.z = pack_bf16x2(__uint_as_float(o[x + 4]) * inv, __uint_as_float(o[x + 5]) * inv);
            v.w = pack_bf16x2(__uint_as_float(o[x + 6]) * inv, __uint_as_float(o[x + 7]) * inv);
            *reinterpret_cast<uint4*>(dst + c * 32 + x) = v;
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (tid == 0 && s_abort) fc_flag(&g_fc_err, FC_EBIT_TIMEOUT);
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

}  // namespace

extern "C" fc_status fc_tree_attn(const void* d_q, const void* d_k_cache, const void* d_v_cache, int kv_cap,
                                  const int32_t* d_kv_len, const void* d_k_tree, const void* d_v_tree,
                                  const uint64_t* d_mask, const int32_t* d_n_nodes, int batch, int n_pad, int H, int Hkv,
                                  int D, float scale, void* d_out, fc_stream stream) {
  if (batch < 0 || H < 1 || Hkv < 1 || kv_cap < 1) return FC_ERR_INVALID_ARG;
  if (D != HD || (n_pad != 64 && n_pad != 128) || H % Hkv != 0 || H / Hkv > 16) return FC_ERR_UNSUPPORTED;
  if (!(scale > 0.f)) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_q || !d_k_cache || !d_v_cache || !d_kv_len || !d_k_tree || !d_v_tree || !d_mask || !d_n_nodes || !d_out)
    return FC_ERR_INVALID_ARG;
  const uintptr_t al = reinterpret_cast<uintptr_t>(d_q) | reinterpret_cast<uintptr_t>(d_k_cache) |
                       reinterpret_cast<uintptr_t>(d_v_cache) | reinterpret_cast<uintptr_t>(d_k_tree) |
                       reinterpret_cast<uintptr_t>(d_v_tree) | reinterpret_cast<uintptr_t>(d_out);
  if (al % 16 || reinterpret_cast<uintptr_t>(d_mask) % 8) return FC_ERR_INVALID_ARG;
  const uint64_t groups = (uint64_t)batch * Hkv;
  const int G = H / Hkv;
  const int tiles = (G * n_pad + BM - 1) / BM;
  if (groups * tiles > 0x7FFFFFFFull) return FC_ERR_UNSUPPORTED;
  CUtensorMap mkc, mvc, mkt, mvt;
  if (!make_map(&mkc, d_k_cache, (uint64_t)kv_cap, groups, BN) || !make_map(&mvc, d_v_cache, (uint64_t)kv_cap, groups, BN) ||
      !make_map(&mkt, d_k_tree, (uint64_t)n_pad, groups, (uint32_t)n_pad) ||
      !make_map(&mvt, d_v_tree, (uint64_t)n_pad, groups, (uint32_t)n_pad))
    return FC_ERR_CUDA;
  if (cudaFuncSetAttribute(k_tree_attn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES) != cudaSuccess)
    return FC_ERR_CUDA;
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
  a.tiles = tiles;
  a.scale_log2 = scale * 1.4426950408889634f;
  k_tree_attn<<<(unsigned)(groups * tiles), TA_THREADS, SMEM_BYTES, static_cast<cudaStream_t>(stream)>>>(mkc, mvc, mkt,
                                                                                                        mvt, a);
  return FC_CHECK_LAUNCH();
}
