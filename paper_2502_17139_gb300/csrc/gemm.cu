// fc_gemm_bf16: C[M][N] = A[M][K] B[K][N] for the decoder forward that
// verifies every draft in one pass (Section IV-D).  Row-major bf16 operands,
// fp32 accumulation in tensor memory, bf16 output.
//
// GB300 design (a persistent, warp-specialised tcgen05 kernel, one CTA per SM):
//   * output tiles of 128 x 256; the CTAs walk the tile list with a stride of
//     the grid, M fastest, so the CTAs of a wave share the weight columns they
//     read (and the activations, a few MB, stay in L2);
//   * warp 0 streams 64-deep K slices of A (128 x 64, K-major) and B (64 x 256,
//     N-major: the weights as stored) into a 4-stage ring with TMA (128-byte
//     swizzle; rows and columns past the matrix edge arrive as zeros, so ragged
//     M, N and K need no special case in the main loop);
//   * warp 1 issues tcgen05.mma kind::f16 (M 128, N 256, K 16; four per slice)
//     into one of two tensor-memory accumulators of 256 fp32 columns, and
//     releases each ring stage with a commit when its MMAs are done;
//   * warps 2-5 drain the other accumulator meanwhile (tcgen05.ld, one row per
//     thread), round to bf16 and store the rows; so a tile's epilogue overlaps
//     the next tile's main loop;
//   * every wait is bounded: a wait that runs out raises FC_ERR_TIMEOUT, and
//     the CTA lets its in-flight copies and MMAs land before it frees tensor
//     memory and exits.
//
// Two epilogues fold the decoder's next step into the GEMM, so its output
// never makes a round trip through HBM in bf16:
//   * K/V heads (fc_gemm_kv_heads): the fused K/V projection's 256-column
//     tile holds two whole heads (D = 128); the epilogue rotates the key
//     heads by each row's node position (RoPE, rotate-half pairing: columns
//     d and d + 64 of a head, both in the tile) from the fp32 accumulators and
//     writes both kinds head-major, as the tree attention and the cache
//     append read them;
//   * SiLU * up (fc_gemm_silu_mul): with the gate and up weights interleaved
//     in 128-column blocks (fc_interleave_gate_up), a tile holds gate block t
//     and up block t, and the epilogue writes act[:, 128t .. 128t + 128) =
//     silu(gate) * up.
#include <algorithm>
#include <cmath>
#include <mutex>

#include "fc_common.cuh"

FC_DEFINE_ERROR_WORD(gemm)

namespace {

constexpr int GM_THREADS = 192;  // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr uint32_t A_BYTES = BM * BK * 2;                // 16 KB
constexpr uint32_t B_CHUNK = BK * 64 * 2;                // 8 KB: 64 K rows x 64 N columns
constexpr uint32_t B_BYTES = (BN / 64) * B_CHUNK;        // 32 KB
constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;      // 48 KB
constexpr uint32_t OFF_BAR = STAGES * STAGE_BYTES;
constexpr uint32_t SMEM_BYTES = OFF_BAR + 256 + 1024;    // + alignment slack
constexpr uint32_t TMEM_COLS = 2 * BN;                   // two accumulators
constexpr uint64_t WAIT_CYCLES = 4000000000ull;          // ~2 s
constexpr uint64_t DRAIN_CYCLES = 400000000ull;          // ~0.2 s

enum { B_FULL = 0, B_EMPTY = STAGES, B_ACC_FULL = 2 * STAGES, B_ACC_EMPTY = 2 * STAGES + 2,
       B_DRAIN = 2 * STAGES + 4, N_BARS = 2 * STAGES + 5 };

enum { EPI_STORE = 0, EPI_KV_HEADS = 1, EPI_SILU_MUL = 2 };

struct GemmArgs {
  __nv_bfloat16* c;  // EPI_STORE: C [M][N]; EPI_SILU_MUL: act [M][N / 2]
  int M, N, K;
  int tiles_m, tiles;
  // EPI_KV_HEADS: rows are (sequence, node) = b * n_pad + i; columns are Hkv key
  // heads then Hkv value heads of 128
  __nv_bfloat16* k_out;  // [B][Hkv][n_pad][128], rotated
  __nv_bfloat16* v_out;  // [B][Hkv][n_pad][128]
  const int32_t* pos;    // [B][n_pad]; a negative position leaves its row unrotated
  int n_pad, hkv;
  double rope_nl2f;      // -2 log2(base) / 128
  unsigned int* err;     // the launch's error word (NULL: this file's own)
};

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], "
      "[%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

__device__ __forceinline__ bool wait_warp(uint32_t bar, uint32_t parity, volatile int* abort) {
  return __all_sync(0xFFFFFFFFu, mbar_wait_bounded(bar, parity, abort, WAIT_CYCLES));
}

__device__ __forceinline__ uint4 pack8_bits(const uint32_t* v) {
  uint4 o;
  o.x = pack_bf16x2(__uint_as_float(v[0]), __uint_as_float(v[1]));
  o.y = pack_bf16x2(__uint_as_float(v[2]), __uint_as_float(v[3]));
  o.z = pack_bf16x2(__uint_as_float(v[4]), __uint_as_float(v[5]));
  o.w = pack_bf16x2(__uint_as_float(v[6]), __uint_as_float(v[7]));
  return o;
}

__device__ __forceinline__ uint4 pack8(const float* v) {
  uint4 o;
  o.x = pack_bf16x2(v[0], v[1]);
  o.y = pack_bf16x2(v[2], v[3]);
  o.z = pack_bf16x2(v[4], v[5]);
  o.w = pack_bf16x2(v[6], v[7]);
  return o;
}

template <int EPI>
__global__ void __launch_bounds__(GM_THREADS, 1)
    k_gemm(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b, GemmArgs g) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  __shared__ float2 s_rope[64];
  if constexpr (EPI == EPI_KV_HEADS) fc_rope_table(s_rope, 64, g.rope_nl2f);  // read after the barrier below
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + OFF_BAR;
  auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };
  const int nk = (g.K + BK - 1) / BK;

  if (tid == 0) {
    s_abort = 0;
    for (int i = 0; i < STAGES; ++i) {
      mbar_init(bar(B_FULL + i), 1);
      mbar_init(bar(B_EMPTY + i), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(B_ACC_FULL + i), 1);
      mbar_init(bar(B_ACC_EMPTY + i), 4);  // one arrival per epilogue warp
    }
    mbar_init(bar(B_DRAIN), 1);
    fence_mbar_init();
    prefetch_tmap(&tm_a);
    prefetch_tmap(&tm_b);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      uint32_t issued = 0;
      for (int t = blockIdx.x; t < g.tiles && !s_abort; t += gridDim.x) {
        const int m0 = (t % g.tiles_m) * BM, n0 = (t / g.tiles_m) * BN;
        for (int kb = 0; kb < nk; ++kb) {
          const uint32_t s = issued % STAGES, ph = (issued / STAGES) & 1;
          if (!mbar_wait_bounded(bar(B_EMPTY + s), ph ^ 1, &s_abort, WAIT_CYCLES)) break;
          const uint32_t st = sbase + s * STAGE_BYTES;
          mbar_expect_tx(bar(B_FULL + s), STAGE_BYTES);
          tma_load_2d(st, &tm_a, kb * BK, m0, bar(B_FULL + s));
#pragma unroll
          for (int c = 0; c < BN / 64; ++c) tma_load_2d(st + A_BYTES + c * B_CHUNK, &tm_b, n0 + 64 * c, kb * BK, bar(B_FULL + s));
          ++issued;
        }
      }
      if (s_abort) {  // let the copies in flight land before the CTA exits
        volatile int dummy = 0;
        for (uint32_t i = issued > STAGES ? issued - STAGES : 0; i < issued; ++i)
          mbar_wait_bounded(bar(B_FULL + i % STAGES), (i / STAGES) & 1, &dummy, DRAIN_CYCLES);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer (the whole warp, one lane elected per MMA) -----
    constexpr uint32_t IDESC = idesc_bf16_f32(BM, BN, 1);  // A K-major, B N-major
    uint32_t consumed = 0, acc_i = 0;
    bool ok = true;
    for (int t = blockIdx.x; ok && t < g.tiles; t += gridDim.x, ++acc_i) {
      const uint32_t buf = acc_i & 1, acc_ph = (acc_i >> 1) & 1;
      if (!(ok = wait_warp(bar(B_ACC_EMPTY + buf), acc_ph ^ 1, &s_abort))) break;
      tc_fence_after();
      const uint32_t d = tmem + buf * BN;
      for (int kb = 0; kb < nk; ++kb, ++consumed) {
        const uint32_t s = consumed % STAGES, ph = (consumed / STAGES) & 1;
        if (!(ok = wait_warp(bar(B_FULL + s), ph, &s_abort))) break;
        tc_fence_after();
        const uint32_t sa = sbase + s * STAGE_BYTES, sb = sa + A_BYTES;
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk)
          tc_mma_f16(d, smem_desc_sw128(sa + kk * 32, 16, 1024), smem_desc_sw128(sb + kk * 2048, B_CHUNK, 1024),
                     IDESC, (kb > 0 || kk > 0) ? 1u : 0u);
        tc_commit(bar(B_EMPTY + s));
      }
      if (!ok) break;
      tc_commit(bar(B_ACC_FULL + buf));
    }
    if (__any_sync(0xFFFFFFFFu, s_abort)) {  // let issued MMAs retire before tensor memory is freed
      tc_commit(bar(B_DRAIN));
      volatile int dummy = 0;
      mbar_wait_bounded(bar(B_DRAIN), 0, &dummy, DRAIN_CYCLES);
    }
  } else {
    // ---------------- epilogue: thread = output row of the tile ----------------
    const int q4 = warp & 3;  // the tensor-memory lane quarter this warp may read
    const int r = q4 * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    uint32_t acc_i = 0;
    for (int t = blockIdx.x; t < g.tiles; t += gridDim.x, ++acc_i) {
      const uint32_t buf = acc_i & 1, acc_ph = (acc_i >> 1) & 1;
      if (!wait_warp(bar(B_ACC_FULL + buf), acc_ph, &s_abort)) break;
      tc_fence_after();
      const int m0 = (t % g.tiles_m) * BM, n0 = (t / g.tiles_m) * BN;
      const int row = m0 + r;
      const uint32_t tacc = tmem + buf * BN + lane_off;
      if constexpr (EPI == EPI_STORE) {
        __nv_bfloat16* crow = g.c + (size_t)row * g.N;
#pragma unroll 1
        for (int cc = 0; cc < BN / 32; ++cc) {
          uint32_t v[32];
          tmem_ld32(tacc + cc * 32, v);
          tc_wait_ld();
          const int col = n0 + cc * 32;
          if (row < g.M && col < g.N) {
#pragma unroll
            for (int u = 0; u < 4; ++u)
              if (col + 8 * u + 8 <= g.N)
                *reinterpret_cast<uint4*>(crow + col + 8 * u) = pack8_bits(v + 8 * u);
          }
        }
      } else if constexpr (EPI == EPI_SILU_MUL) {
        // gate columns [0, 128) and up columns [128, 256) of the tile -> act block n0 / 2
        __nv_bfloat16* arow = g.c + (size_t)row * (g.N / 2) + n0 / 2;
#pragma unroll 1
        for (int cc = 0; cc < 4; ++cc) {
          uint32_t gv[32], uv[32];
          tmem_ld32(tacc + cc * 32, gv);
          tmem_ld32(tacc + 128 + cc * 32, uv);
          tc_wait_ld();
          if (row < g.M) {
            float a[32];
#pragma unroll
            for (int u = 0; u < 32; ++u) {
              const float x = __uint_as_float(gv[u]);
              // the fast divide: an IEEE division takes a slow path for a zero dividend,
              // which doubled this epilogue's time on padding rows (all zeros)
              a[u] = __fdividef(x, 1.f + __expf(-x)) * __uint_as_float(uv[u]);
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
              *reinterpret_cast<uint4*>(arow + cc * 32 + 8 * u) = pack8(a + 8 * u);
          }
        }
      } else {
        // two heads of 128 columns; head hh < hkv is a key head (rotated)
        const int b = row / g.n_pad, i = row - b * g.n_pad;
        const int p = row < g.M ? g.pos[row] : -1;
#pragma unroll 1
        for (int j = 0; j < 2; ++j) {
          const int hh = n0 / 128 + j;
          const bool key = hh < g.hkv;
          const int head = key ? hh : hh - g.hkv;
          __nv_bfloat16* dst = (key ? g.k_out : g.v_out) + (((size_t)b * g.hkv + head) * g.n_pad + i) * 128;
#pragma unroll 1
          for (int q = 0; q < 2; ++q) {  // dims 32q .. 32q + 31 and their partners 64 + 32q ..
            uint32_t lv[32], hv[32];
            tmem_ld32(tacc + j * 128 + q * 32, lv);
            tmem_ld32(tacc + j * 128 + 64 + q * 32, hv);
            tc_wait_ld();
            if (row < g.M) {
              float lo[32], hi[32];
#pragma unroll
              for (int u = 0; u < 32; ++u) {
                lo[u] = __uint_as_float(lv[u]);
                hi[u] = __uint_as_float(hv[u]);
              }
              if (key && p >= 0) {
#pragma unroll
                for (int u = 0; u < 32; ++u) {
                  float sn, cs;
                  fc_rope_sincos((float)p, s_rope[q * 32 + u], sn, cs);
                  const float x0 = lo[u], x1 = hi[u];
                  lo[u] = x0 * cs - x1 * sn;
                  hi[u] = x1 * cs + x0 * sn;
                }
              }
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                *reinterpret_cast<uint4*>(dst + q * 32 + 8 * u) = pack8(lo + 8 * u);
                *reinterpret_cast<uint4*>(dst + 64 + q * 32 + 8 * u) = pack8(hi + 8 * u);
              }
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(B_ACC_EMPTY + buf));
    }
  }
  tc_fence_before();
  __syncthreads();
  if (tid == 0 && s_abort) fc_flag(FC_ERR_WORD(g.err), FC_EBIT_TIMEOUT);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

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

// Row-major bf16 matrix [rows][cols] as a 2-D map with a (64, box_rows) box,
// 128-byte swizzle; reads past the edges return zeros.
bool make_map_2d(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t es[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 0;
  return n;
}

bool aligned16(const void* p) { return reinterpret_cast<uintptr_t>(p) % 16 == 0; }

template <int EPI>
fc_status launch_gemm(const void* d_a, const void* d_b, int M, int N, int K, GemmArgs g, cudaStream_t stream) {
  CUtensorMap ma, mb;
  if (!make_map_2d(&ma, d_a, (uint64_t)M, (uint64_t)K, BM) || !make_map_2d(&mb, d_b, (uint64_t)K, (uint64_t)N, BK))
    return FC_ERR_CUDA;
  g.M = M;
  g.N = N;
  g.K = K;
  g.tiles_m = (M + BM - 1) / BM;
  g.err = fc_error_slot();
  const int64_t tiles = (int64_t)g.tiles_m * ((N + BN - 1) / BN);
  if (tiles > 0x7FFFFFFF) return FC_ERR_UNSUPPORTED;
  g.tiles = (int)tiles;
  const int sms = sm_count();
  if (sms <= 0) return FC_ERR_CUDA;
  if (cudaFuncSetAttribute(k_gemm<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES) != cudaSuccess)
    return FC_ERR_CUDA;
  const int grid = (int)std::min<int64_t>(tiles, sms);
  k_gemm<EPI><<<grid, GM_THREADS, SMEM_BYTES, stream>>>(ma, mb, g);
  return FC_CHECK_LAUNCH();
}

// gate/up weights [K][2 * inter] (gate columns, then up columns) -> 128-column
// blocks interleaved: out[:, 256 t + c] = gate[:, 128 t + c] and
// out[:, 256 t + 128 + c] = up[:, 128 t + c], c < 128.  16-byte chunks.
__global__ void k_interleave_gate_up(const uint4* __restrict__ in, uint4* __restrict__ out, int K, int inter) {
  const int cw = inter / 8;  // chunks per half row
  const size_t items = (size_t)K * 2 * cw;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < items; e += (size_t)gridDim.x * blockDim.x) {
    const size_t k = e / (2 * cw);
    const int c = (int)(e - k * 2 * cw);       // output chunk in the row
    const int blk = c / 32, within = c % 32;   // 256-column block, chunk inside it
    const int half = within / 16, cc = within % 16;
    const int src = half * cw + blk * 16 + cc;  // gate or up chunk
    out[e] = in[k * 2 * cw + src];
  }
}

}  // namespace

extern "C" size_t fc_gemm_workspace(void) { return 0; }

extern "C" fc_status fc_gemm_bf16(const void* d_a, const void* d_b, void* d_c, int M, int N, int K, void* d_ws,
                                  size_t ws_bytes, fc_stream stream) {
  FC_NVTX_RANGE();
  (void)d_ws;
  (void)ws_bytes;
  if (M < 0 || N < 1 || K < 1) return FC_ERR_INVALID_ARG;
  if (M == 0) return FC_OK;
  if (!d_a || !d_b || !d_c) return FC_ERR_INVALID_ARG;
  if (!aligned16(d_a) || !aligned16(d_b) || !aligned16(d_c)) return FC_ERR_INVALID_ARG;
  if (N % 8 || K % 8) return FC_ERR_UNSUPPORTED;
  GemmArgs g{};
  g.c = static_cast<__nv_bfloat16*>(d_c);
  return launch_gemm<EPI_STORE>(d_a, d_b, M, N, K, g, static_cast<cudaStream_t>(stream));
}

extern "C" fc_status fc_gemm_kv_heads(const void* d_a, const void* d_wkv, int M, int K, int Hkv, int D, int batch,
                                      int n_pad, const int32_t* d_pos, float rope_base, void* d_k_rot,
                                      void* d_v_heads, fc_stream stream) {
  FC_NVTX_RANGE();
  if (M < 0 || K < 1 || Hkv < 1 || batch < 0 || n_pad < 1 || M != batch * n_pad) return FC_ERR_INVALID_ARG;
  if (D != 128 || K % 8) return FC_ERR_UNSUPPORTED;
  if (!(rope_base > 0.f) || !std::isfinite(rope_base)) return FC_ERR_INVALID_ARG;
  if (M == 0) return FC_OK;
  if (!d_a || !d_wkv || !d_pos || !d_k_rot || !d_v_heads) return FC_ERR_INVALID_ARG;
  if (!aligned16(d_a) || !aligned16(d_wkv) || !aligned16(d_k_rot) || !aligned16(d_v_heads)) return FC_ERR_INVALID_ARG;
  GemmArgs g{};
  g.k_out = static_cast<__nv_bfloat16*>(d_k_rot);
  g.v_out = static_cast<__nv_bfloat16*>(d_v_heads);
  g.pos = d_pos;
  g.n_pad = n_pad;
  g.hkv = Hkv;
  g.rope_nl2f = -2.0 * std::log2((double)rope_base) / 128.0;
  return launch_gemm<EPI_KV_HEADS>(d_a, d_wkv, M, 2 * Hkv * 128, K, g, static_cast<cudaStream_t>(stream));
}

extern "C" fc_status fc_gemm_silu_mul(const void* d_a, const void* d_wgu, int M, int K, int inter, void* d_act,
                                      fc_stream stream) {
  FC_NVTX_RANGE();
  if (M < 0 || K < 1 || inter < 1) return FC_ERR_INVALID_ARG;
  if (inter % 128 || K % 8) return FC_ERR_UNSUPPORTED;
  if (M == 0) return FC_OK;
  if (!d_a || !d_wgu || !d_act || !aligned16(d_a) || !aligned16(d_wgu) || !aligned16(d_act)) return FC_ERR_INVALID_ARG;
  GemmArgs g{};
  g.c = static_cast<__nv_bfloat16*>(d_act);
  return launch_gemm<EPI_SILU_MUL>(d_a, d_wgu, M, 2 * inter, K, g, static_cast<cudaStream_t>(stream));
}

extern "C" fc_status fc_interleave_gate_up(const void* d_wgu, void* d_out, int K, int inter, fc_stream stream) {
  FC_NVTX_RANGE();
  if (K < 1 || inter < 1) return FC_ERR_INVALID_ARG;
  if (inter % 128) return FC_ERR_UNSUPPORTED;
  if (!d_wgu || !d_out || d_wgu == d_out || !aligned16(d_wgu) || !aligned16(d_out)) return FC_ERR_INVALID_ARG;
  const size_t items = (size_t)K * (2 * inter / 8);
  const unsigned blocks = (unsigned)std::min<size_t>((items + 255) / 256, 152 * 16);
  k_interleave_gate_up<<<blocks, 256, 0, static_cast<cudaStream_t>(stream)>>>(
      static_cast<const uint4*>(d_wgu), static_cast<uint4*>(d_out), K, inter);
  return FC_CHECK_LAUNCH();
}
