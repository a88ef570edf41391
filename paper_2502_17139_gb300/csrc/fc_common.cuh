// Shared device/host helpers for the fastcoder CUDA library (sm_103a).
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include <nvtx3/nvToolsExt.h>

#include "../../include/fastcoder.h"

// One NVTX range per C-ABI call, named after the call: a profiler's timeline
// then shows which entry point enqueued which kernels.  With no tool
// attached the push and pop are calls into empty functions.
struct FcNvtxRange {
  explicit FcNvtxRange(const char* name) { nvtxRangePushA(name); }
  ~FcNvtxRange() { nvtxRangePop(); }
  FcNvtxRange(const FcNvtxRange&) = delete;
  FcNvtxRange& operator=(const FcNvtxRange&) = delete;
};
#define FC_NVTX_RANGE() FcNvtxRange fc_nvtx_range_(__func__)

// ---------------------------------------------------------------------------
// Device error word.  Kernels OR one of these bits in; fc_get_error() reads
// and clears it.  Every translation unit owns one word (the library is built
// without relocatable device code), and fc_get_error() collects them all.
// ---------------------------------------------------------------------------
#define FC_EBIT_INVALID 1u
#define FC_EBIT_CAPACITY 2u
#define FC_EBIT_TIMEOUT 4u
#define FC_EBIT_INTERNAL 8u

#define FC_DEFINE_ERROR_WORD(NAME)                                              \
  static __device__ unsigned int g_fc_err;                                      \
  extern "C" unsigned int fc_take_error_##NAME(cudaStream_t s) {                \
    unsigned int h = 0, z = 0;                                                  \
    if (cudaMemcpyFromSymbolAsync(&h, g_fc_err, sizeof h, 0,                    \
                                  cudaMemcpyDeviceToHost, s) != cudaSuccess)    \
      return FC_EBIT_INTERNAL;                                                  \
    cudaMemcpyToSymbolAsync(g_fc_err, &z, sizeof z, 0, cudaMemcpyHostToDevice, s); \
    cudaStreamSynchronize(s);                                                   \
    return h;                                                                   \
  }

__device__ __forceinline__ void fc_flag(unsigned int* word, unsigned int bit) { atomicOr(word, bit); }

// Kernels take the error word of their launch as an argument: NULL means
// their translation unit's own word (collected by fc_get_error), a device
// pointer a word of the caller's (fc_pipeline gives every sub-batch its own,
// so an error is reported for the sub-batch that raised it).
#define FC_ERR_WORD(err) ((err) ? (err) : &g_fc_err)

// Host: the error word that launches made by the calling thread pass to their
// kernels (NULL unless an FcErrorScope is active on this thread).
unsigned int* fc_error_slot();
// Host: routes the calling thread's launches to `word` while in scope.
struct FcErrorScope {
  unsigned int* prev;
  explicit FcErrorScope(unsigned int* word);
  ~FcErrorScope();
  FcErrorScope(const FcErrorScope&) = delete;
  FcErrorScope& operator=(const FcErrorScope&) = delete;
};

// Debug builds (compiled with -DFC_DEBUG into libfastcoder_debug.so) check
// the indexes that gathers take from data, such as suffix-array entries,
// before using them: an index out of range sets FC_ERR_INTERNAL in the
// translation unit's error word and the access is skipped.  Release builds
// trust the datastores and trees they are given (this library builds both).
__device__ __forceinline__ bool fc_debug_ok(bool ok, unsigned int* word) {
  if (!ok) fc_flag(word, FC_EBIT_INTERNAL);
  return ok;
}
#ifdef FC_DEBUG
#define FC_DEBUG_CHECK(ok) fc_debug_ok((ok), &g_fc_err)
#else
#define FC_DEBUG_CHECK(ok) true
#endif

// Host: the status of a set of error bits, the most severe first.
static inline fc_status fc_status_of_bits(unsigned int e) {
  if (e & FC_EBIT_INTERNAL) return FC_ERR_INTERNAL;
  if (e & FC_EBIT_TIMEOUT) return FC_ERR_TIMEOUT;
  if (e & FC_EBIT_CAPACITY) return FC_ERR_CAPACITY;
  if (e & FC_EBIT_INVALID) return FC_ERR_INVALID_ARG;
  return FC_OK;
}

// Host: runs set_up(device) once per device (kernel attributes are per
// device); `done` holds a bit per device already set up (devices past 63 are
// set up on every call).
template <typename F>
fc_status fc_once_per_device(std::atomic<unsigned long long>& done, F&& set_up) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return FC_ERR_CUDA;
  const unsigned long long bit = dev < 64 ? 1ull << dev : 0ull;
  if (bit && (done.load(std::memory_order_acquire) & bit)) return FC_OK;
  const fc_status st = set_up(dev);
  if (st == FC_OK && bit) done.fetch_or(bit, std::memory_order_acq_rel);
  return st;
}

// Host: map a CUDA launch result to a status.
static inline fc_status fc_cuda_status(cudaError_t e) { return e == cudaSuccess ? FC_OK : FC_ERR_CUDA; }

#define FC_CHECK_LAUNCH() fc_cuda_status(cudaGetLastError())

// Host: the limits every retrieval-shaped call accepts.
static inline bool fc_retrieve_params_ok(const fc_retrieve_params& p) {
  return p.n_max >= 1 && p.n_max <= FC_MAX_NMAX && p.n_min >= 1 && p.n_min <= p.n_max && p.top_k >= 1 &&
         p.top_k <= FC_MAX_TOPK && p.draft_len >= 1 && p.draft_len <= FC_MAX_DRAFT_LEN && p.max_occ >= 1 &&
         p.max_occ <= FC_MAX_OCC;
}

// ---------------------------------------------------------------------------
// Small PTX wrappers (sm_100 family).  Shared-memory addresses are 32-bit
// CTA-window addresses.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}" ::"r"(bar),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// try_wait with a suspend-time hint: the thread sleeps in hardware until the
// phase completes or about hint_ns pass, instead of spinning (a spinning
// waiter steals issue slots and the shared-memory pipe from the warps doing
// the work).
__device__ __forceinline__ bool mbar_try_wait_sleep(uint32_t bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\tselp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}

// Bounded wait: returns false (and raises *abort) when the barrier phase has
// not completed within limit_cycles SM clock cycles, or when another thread
// of the CTA already gave up.  Each poll may sleep up to ~0.5 ms.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity, volatile int* abort,
                                                  uint64_t limit_cycles) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  for (;;) {
    if (mbar_try_wait_sleep(bar, parity, 500000u)) return true;
    if (*abort) return false;
    if ((uint64_t)(clock64() - t0) > limit_cycles) {
      *abort = 1;
      return false;
    }
  }
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// 3-D tiled TMA load into shared memory, completion counted on an mbarrier.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int x, int y, int z,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void prefetch_tmap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ---- tcgen05 (5th-generation tensor cores, accumulators in tensor memory) --
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// tcgen05.mma and tcgen05.commit are issued by one thread, but these wrappers
// are called by the whole warp with warp-uniform operands: elect.sync picks
// the issuing lane inside the instruction sequence, so the compiler keeps the
// control flow uniform and the operands in uniform registers.  Issuing from a
// divergent `if (lane == 0)` branch instead costs tens of cycles per MMA in
// operand moves and starves the tensor pipe.

// D[tmem] (+)= A[smem desc] * B[smem desc], kind::f16 (bf16 inputs, fp32 accumulate).
__device__ __forceinline__ void tc_mma_f16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p, e;\n\tsetp.ne.b32 p, %4, 0;\n\telect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem desc]: A (M x K, bf16 pairs packed per 32-bit
// column, one row per lane) is read from tensor memory.
__device__ __forceinline__ void tc_mma_f16_tmem_a(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                                  uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p, e;\n\tsetp.ne.b32 p, %4, 0;\n\telect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on an mbarrier once every tcgen05 op issued so far by the warp's
// issuing lane is done (warp-collective like the MMA wrappers).
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile(
      "{\n\t.reg .pred e;\n\telect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n\t}" ::"r"(bar)
      : "memory");
}

__device__ __forceinline__ void tc_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tc_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// 32 lanes x 32 consecutive 32-bit columns: thread t of the warp receives
// lane (quarter*32 + t), columns [col, col + 32).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
          taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
      "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
      "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

// Shared-memory matrix descriptor for tcgen05 (sm_100 layout):
//   [0,14) start address >> 4, [16,30) leading byte offset >> 4,
//   [32,46) stride byte offset >> 4, [46,48) version = 1,
//   [49,52) base offset = 0, [52] lbo mode = 0, [61,64) swizzle mode
//   (2 = 128-byte swizzle).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr, uint32_t lbo_bytes, uint32_t sbo_bytes) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)((lbo_bytes >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo_bytes >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1u << 46;
  d |= (uint64_t)2u << 61;
  return d;
}

// Instruction descriptor for tcgen05.mma kind::f16 with bf16 A/B and fp32 D:
//   [4,6) D format (1 = f32), [7,10) A format (1 = bf16), [10,13) B format
//   (1 = bf16), [15] A major (0 = K), [16] B major (0 = K, 1 = MN),
//   [17,23) N >> 3, [24,29) M >> 4.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(uint32_t M, uint32_t N, uint32_t b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (b_mn_major << 16) | ((N >> 3) << 17) | ((M >> 4) << 24);
}

// ---- rotary position embedding (Su et al., RoFormer), rotate-half pairing:
// dimension i pairs with i + D/2 and turns by pos * f_i, f_i = base^(-2i/D).
// f_i is held as two floats (hi + lo, from fp64), so that pos * f_i comes out
// as hi * pos, its exact rounding error (an fma) and lo * pos: the angle is
// good to ~1e-7 rad at any position below 2^24, where a plain fp32 product
// would be off by pos * f_i * 2^-24.  The angle is reduced modulo 2 pi with a
// two-constant Cody-Waite split (2 pi rounded to fp32, then the rest) before
// the MUFU sine and cosine, which are accurate on [-pi, pi].
constexpr int FC_ROPE_MAX_HALF = 512;  // D / 2 for D up to 1024

// tab[i] = (hi, lo) of f_i for i < half, filled by the calling block's
// threads; the caller synchronises before use.
__device__ __forceinline__ void fc_rope_table(float2* tab, int half, double nl2f) {
  for (int i = threadIdx.x; i < half; i += blockDim.x) {
    const double f = exp2((double)i * nl2f);
    const float hi = (float)f;
    tab[i] = make_float2(hi, (float)(f - (double)hi));
  }
}

__device__ __forceinline__ void fc_rope_sincos(float pos, float2 f, float& sn, float& cs) {
  const float a_hi = pos * f.x;
  const float a_lo = fmaf(pos, f.y, fmaf(pos, f.x, -a_hi));
  const float k = rintf(a_hi * 0.15915493667125702f);  // a / (2 pi), rounded
  float r = fmaf(-k, 6.2831854820251465f, a_hi);        // 2 pi rounded to fp32
  r = fmaf(-k, -1.7484555314695172e-07f, r) + a_lo;     // 2 pi minus that
  __sincosf(r, &sn, &cs);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
