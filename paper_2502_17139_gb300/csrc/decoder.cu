// The pieces of a decoder forward around the tree attention (Section IV-D:
// the target model verifies every draft in one forward), for a LLaMA-family
// model like the paper's: token embedding, residual add + RMSNorm, the
// SiLU-gated MLP's activation and the head-major layout of the tree's keys
// (rotated) and values.  The GEMMs are gemm.cu's tcgen05 kernel.
//
//   * k_embed: one row per warp; ids >= vocab (tree padding) embed as zeros.
//   * k_add_rmsnorm: one CTA per row; x += r is rounded to bf16 (the
//     residual stream), then out = x / sqrt(mean(x^2) + eps) * w in fp32.
//   * k_silu_mul: out = silu(gate) * up, fp32 math.
//   * k_rope_heads: node-major projection rows -> head-major [B][heads][n][D],
//     rotated by position (the rotation of tree_attn.cu) or copied.
#include <algorithm>
#include <cmath>


#include "fc_common.cuh"

FC_DEFINE_ERROR_WORD(dec)

namespace {

constexpr int ROWS_PER_BLOCK = 8;  // one warp per row

__global__ void k_embed(const uint32_t* __restrict__ tok, int n, const uint4* __restrict__ table, int vocab,
                        int hidden, uint4* __restrict__ out) {
  const int row = blockIdx.x * ROWS_PER_BLOCK + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= n) return;
  const uint32_t t = tok[row];
  const int w = hidden / 8;
  uint4* o = out + (size_t)row * w;
  if (t >= (uint32_t)vocab) {
    for (int c = lane; c < w; c += 32) o[c] = make_uint4(0, 0, 0, 0);
    return;
  }
  const uint4* src = table + (size_t)t * w;
  for (int c = lane; c < w; c += 32) o[c] = src[c];
}

__device__ __forceinline__ float2 bf2f(uint32_t v) {
  return __bfloat1622float2(*reinterpret_cast<__nv_bfloat162*>(&v));
}
__device__ __forceinline__ uint32_t f2bf(float a, float b) {
  __nv_bfloat162 r = __float22bfloat162_rn(make_float2(a, b));
  return *reinterpret_cast<uint32_t*>(&r);
}

// One CTA of NORM_THREADS per row; a thread holds up to NORM_CHUNKS 16-byte
// chunks of the row in registers between the sum of squares and the scaling,
// so the row is read once.  Rows wider than NORM_THREADS * NORM_CHUNKS chunks
// reread the rest.
constexpr int NORM_THREADS = 256, NORM_CHUNKS = 2;

__global__ void __launch_bounds__(NORM_THREADS) k_add_rmsnorm(uint4* __restrict__ x, const uint4* __restrict__ r,
                                                              const uint4* __restrict__ w, uint4* __restrict__ out,
                                                              int rows, int dim, float eps) {
  __shared__ float s_part[NORM_THREADS / 32];
  const int row = blockIdx.x, tid = threadIdx.x, lane = tid & 31, wp = tid >> 5;
  if (row >= rows) return;
  const int cw = dim / 8;
  uint4* xr = x + (size_t)row * cw;
  const uint4* rr = r ? r + (size_t)row * cw : nullptr;
  uint4 keep[NORM_CHUNKS];
  float ss = 0.f;
  // x (+ r): rounded to bf16 and written back when r is given; sum of squares
  auto load = [&](int c) {
    uint4 v = xr[c];
    if (rr) {  // the residual stream in bf16: x + r, rounded
      const uint4 a = rr[c];
      uint32_t* vv = &v.x;
      const uint32_t* aa = &a.x;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 xv = bf2f(vv[q]), av = bf2f(aa[q]);
        vv[q] = f2bf(xv.x + av.x, xv.y + av.y);
      }
      xr[c] = v;
    }
    const uint32_t* vv = &v.x;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 f = bf2f(vv[q]);
      ss = fmaf(f.x, f.x, fmaf(f.y, f.y, ss));
    }
    return v;
  };
#pragma unroll
  for (int k = 0; k < NORM_CHUNKS; ++k) {
    const int c = tid + k * NORM_THREADS;
    if (c < cw) keep[k] = load(c);
  }
  for (int c = tid + NORM_CHUNKS * NORM_THREADS; c < cw; c += NORM_THREADS) load(c);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
  if (lane == 0) s_part[wp] = ss;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int i = 0; i < NORM_THREADS / 32; ++i) tot += s_part[i];
  const float inv = rsqrtf(tot / (float)dim + eps);
  uint4* orow = out + (size_t)row * cw;
  auto store = [&](int c, const uint4& v) {
    const uint4 g = w[c];
    const uint32_t* vv = &v.x;
    const uint32_t* gg = &g.x;
    uint4 res;
    uint32_t* rv = &res.x;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 f = bf2f(vv[q]), gw = bf2f(gg[q]);
      rv[q] = f2bf(f.x * inv * gw.x, f.y * inv * gw.y);
    }
    orow[c] = res;
  };
#pragma unroll
  for (int k = 0; k < NORM_CHUNKS; ++k) {
    const int c = tid + k * NORM_THREADS;
    if (c < cw) store(c, keep[k]);
  }
  for (int c = tid + NORM_CHUNKS * NORM_THREADS; c < cw; c += NORM_THREADS) store(c, xr[c]);
}

__global__ void k_silu_mul(const uint4* __restrict__ gu, uint4* __restrict__ out, int rows, int inter) {
  const int cw = inter / 8;
  const size_t items = (size_t)rows * cw;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < items; e += (size_t)gridDim.x * blockDim.x) {
    const size_t row = e / cw;
    const int c = (int)(e - row * cw);
    const uint4 g = gu[row * 2 * cw + c], u = gu[row * 2 * cw + cw + c];
    const uint32_t* gg = &g.x;
    const uint32_t* uu = &u.x;
    uint4 res;
    uint32_t* rv = &res.x;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 a = bf2f(gg[q]), b = bf2f(uu[q]);
      rv[q] = f2bf(__fdividef(a.x, 1.f + __expf(-a.x)) * b.x, __fdividef(a.y, 1.f + __expf(-a.y)) * b.y);
    }
    out[e] = res;
  }
}

// node-major rows in[(b * n_pad + i) * stride + h * D + d] -> head-major
// out[((b * heads + h) * n_pad + i) * D + d], rotated by pos[b][i] when
// rotate != 0 (a negative position is copied unrotated).  One thread per pair
// of partner 16-byte chunks (dimensions 8c..8c+7 and D/2 + 8c..).
__global__ void k_rope_heads(const __nv_bfloat16* __restrict__ in, int stride, __nv_bfloat16* __restrict__ out,
                             int B, int n_pad, int heads, int D, const int32_t* __restrict__ pos, int rotate,
                             double nl2f) {
  __shared__ float2 tab[FC_ROPE_MAX_HALF];
  if (rotate) {
    for (int i = threadIdx.x; i < D / 2; i += blockDim.x) {
      const double f = exp2((double)i * nl2f);
      const float hi = (float)f;
      tab[i] = make_float2(hi, (float)(f - (double)hi));
    }
  }
  __syncthreads();
  const int ch = D / 16;
  const size_t items = (size_t)B * n_pad * heads * ch;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < items; e += (size_t)gridDim.x * blockDim.x) {
    const int c = (int)(e % ch);
    size_t t = e / ch;
    const int h = (int)(t % heads);
    t /= heads;
    const int i = (int)(t % n_pad);
    const int b = (int)(t / n_pad);
    const uint4* src = reinterpret_cast<const uint4*>(in + ((size_t)b * n_pad + i) * stride + (size_t)h * D);
    uint4 lo = src[c], hi = src[c + ch];
    const int p = rotate ? pos[(size_t)b * n_pad + i] : -1;
    if (p >= 0) {
      uint32_t* l = &lo.x;
      uint32_t* hh = &hi.x;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 xl = bf2f(l[q]), xh = bf2f(hh[q]);
        float s0, c0, s1, c1;
        fc_rope_sincos((float)p, tab[8 * c + 2 * q], s0, c0);
        fc_rope_sincos((float)p, tab[8 * c + 2 * q + 1], s1, c1);
        l[q] = f2bf(xl.x * c0 - xh.x * s0, xl.y * c1 - xh.y * s1);
        hh[q] = f2bf(xh.x * c0 + xl.x * s0, xh.y * c1 + xl.y * s1);
      }
    }
    uint4* dst = reinterpret_cast<uint4*>(out + (((size_t)b * heads + h) * n_pad + i) * D);
    dst[c] = lo;
    dst[c + ch] = hi;
  }
}

bool aligned16(const void* p) { return reinterpret_cast<uintptr_t>(p) % 16 == 0; }

}  // namespace

extern "C" fc_status fc_embed(const uint32_t* d_tok, int n, const void* d_table, int vocab, int hidden, void* d_out,
                              fc_stream stream) {
  FC_NVTX_RANGE();
  if (n < 0 || vocab < 1 || hidden < 8 || hidden % 8) return FC_ERR_INVALID_ARG;
  if (n == 0) return FC_OK;
  if (!d_tok || !d_table || !d_out || !aligned16(d_table) || !aligned16(d_out)) return FC_ERR_INVALID_ARG;
  k_embed<<<(n + ROWS_PER_BLOCK - 1) / ROWS_PER_BLOCK, ROWS_PER_BLOCK * 32, 0, static_cast<cudaStream_t>(stream)>>>(
      d_tok, n, static_cast<const uint4*>(d_table), vocab, hidden, static_cast<uint4*>(d_out));
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_add_rmsnorm(void* d_x, const void* d_r, const void* d_w, void* d_out, int rows, int dim,
                                    float eps, fc_stream stream) {
  FC_NVTX_RANGE();
  if (rows < 0 || dim < 8 || dim % 8 || !(eps >= 0.f)) return FC_ERR_INVALID_ARG;
  if (rows == 0) return FC_OK;
  if (!d_x || !d_w || !d_out || !aligned16(d_x) || !aligned16(d_w) || !aligned16(d_out) || (d_r && !aligned16(d_r)))
    return FC_ERR_INVALID_ARG;
  k_add_rmsnorm<<<rows, NORM_THREADS, 0, static_cast<cudaStream_t>(stream)>>>(
      static_cast<uint4*>(d_x), static_cast<const uint4*>(d_r), static_cast<const uint4*>(d_w),
      static_cast<uint4*>(d_out), rows, dim, eps);
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_silu_mul(const void* d_gu, void* d_out, int rows, int inter, fc_stream stream) {
  FC_NVTX_RANGE();
  if (rows < 0 || inter < 8 || inter % 8) return FC_ERR_INVALID_ARG;
  if (rows == 0) return FC_OK;
  if (!d_gu || !d_out || !aligned16(d_gu) || !aligned16(d_out)) return FC_ERR_INVALID_ARG;
  const size_t items = (size_t)rows * (inter / 8);
  const unsigned blocks = (unsigned)std::min<size_t>((items + 255) / 256, 152 * 32);
  k_silu_mul<<<blocks, 256, 0, static_cast<cudaStream_t>(stream)>>>(static_cast<const uint4*>(d_gu),
                                                                    static_cast<uint4*>(d_out), rows, inter);
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_rope_heads(const void* d_in, int in_stride, void* d_out, int batch, int n_pad, int heads, int D,
                                   const int32_t* d_pos, float base, fc_stream stream) {
  FC_NVTX_RANGE();
  if (batch < 0 || n_pad < 1 || heads < 1 || D < 16 || D > 1024 || D % 16 || in_stride < heads * D ||
      in_stride % 8)
    return FC_ERR_INVALID_ARG;
  const bool rotate = base > 0.f;
  if (rotate && !std::isfinite(base)) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_in || !d_out || (rotate && !d_pos) || !aligned16(d_in) || !aligned16(d_out)) return FC_ERR_INVALID_ARG;
  const size_t items = (size_t)batch * n_pad * heads * (D / 16);
  const unsigned blocks = (unsigned)std::min<size_t>((items + 255) / 256, 152 * 16);
  k_rope_heads<<<blocks, 256, 0, static_cast<cudaStream_t>(stream)>>>(
      static_cast<const __nv_bfloat16*>(d_in), in_stride, static_cast<__nv_bfloat16*>(d_out), batch, n_pad, heads, D,
      d_pos, rotate ? 1 : 0, rotate ? -2.0 * std::log2((double)base) / D : 0.0);
  return FC_CHECK_LAUNCH();
}
