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
#include <algorithm>
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

struct GemmArgs {
  __nv_bfloat16* c;
  int M, N, K;
  int tiles_m, tiles;
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

__global__ void __launch_bounds__(GM_THREADS, 1)
    k_gemm(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b, GemmArgs g) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
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
      __nv_bfloat16* crow = g.c + (size_t)row * g.N;
#pragma unroll 1
      for (int cc = 0; cc < BN / 32; ++cc) {
        uint32_t v[32];
        tmem_ld32(tmem + buf * BN + cc * 32 + lane_off, v);
        tc_wait_ld();
        const int col = n0 + cc * 32;
        if (row < g.M && col < g.N) {
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            if (col + 8 * u + 8 <= g.N) {
              uint4 o;
              o.x = pack_bf16x2(__uint_as_float(v[8 * u + 0]), __uint_as_float(v[8 * u + 1]));
              o.y = pack_bf16x2(__uint_as_float(v[8 * u + 2]), __uint_as_float(v[8 * u + 3]));
              o.z = pack_bf16x2(__uint_as_float(v[8 * u + 4]), __uint_as_float(v[8 * u + 5]));
              o.w = pack_bf16x2(__uint_as_float(v[8 * u + 6]), __uint_as_float(v[8 * u + 7]));
              *reinterpret_cast<uint4*>(crow + col + 8 * u) = o;
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
  if (tid == 0 && s_abort) fc_flag(&g_fc_err, FC_EBIT_TIMEOUT);
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
  CUtensorMap ma, mb;
  if (!make_map_2d(&ma, d_a, (uint64_t)M, (uint64_t)K, BM) || !make_map_2d(&mb, d_b, (uint64_t)K, (uint64_t)N, BK))
    return FC_ERR_CUDA;
  GemmArgs g;
  g.c = static_cast<__nv_bfloat16*>(d_c);
  g.M = M;
  g.N = N;
  g.K = K;
  g.tiles_m = (M + BM - 1) / BM;
  const int64_t tiles = (int64_t)g.tiles_m * ((N + BN - 1) / BN);
  if (tiles > 0x7FFFFFFF) return FC_ERR_UNSUPPORTED;
  g.tiles = (int)tiles;
  const int sms = sm_count();
  if (sms <= 0) return FC_ERR_CUDA;
  if (cudaFuncSetAttribute(k_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES) != cudaSuccess)
    return FC_ERR_CUDA;
  const int grid = (int)std::min<int64_t>(tiles, sms);
  k_gemm<<<grid, GM_THREADS, SMEM_BYTES, static_cast<cudaStream_t>(stream)>>>(ma, mb, g);
  return FC_CHECK_LAUNCH();
}
