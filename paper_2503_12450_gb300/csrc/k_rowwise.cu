// Row-wise and elementwise kernels of the decoding step:
//   - embedding of the input tokens (Eq. 6): class embedding / zero fake
//     conditional tokens on the buffer positions, latent projection or mask
//     embedding on the image positions, plus the position embedding;
//   - LayerNorm of fp32 residual rows into the GEMM operand dtype, optionally
//     gathering rows (the step's switch from all tokens to I_compute) and
//     keeping an fp32 copy of the gathered rows as the compact residual stream;
//   - the final LayerNorm that scatters the recomputed rows into the output
//     cache (Eq. 9: outputs of I_cache tokens stay as cached);
//   - classifier-free guidance with the condition cache (Eq. 7, Eq. 10) on
//     16-byte vectors.
// All of these are bound by HBM bandwidth; one warp per row (LayerNorm) or
// grid-stride 16-byte vectors (CFG) keeps loads coalesced.
#include <cuda_fp8.h>

#include "lazymar_internal.cuh"

namespace lm {

// ---------------------------------------------------------------------------
// Embedding
// ---------------------------------------------------------------------------
// One thread per (token, 4 consecutive columns), grid-stride; the 16-float
// latent of a decoded token is read by all threads of that token (L1 hits).
template <typename TW>
__device__ __forceinline__ float4 load4(const TW* p) {
  if constexpr (sizeof(TW) == 2) {
    const uint2 u = *reinterpret_cast<const uint2*>(p);
    const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
    const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
    return make_float4(a.x, a.y, b.x, b.y);
  } else {
    return *reinterpret_cast<const float4*>(p);
  }
}

template <typename TW, int TD>
__global__ void __launch_bounds__(256) embed_kernel(const float* __restrict__ lat, const uint8_t* __restrict__ mask,
                                                    const int* __restrict__ labels, const TW* __restrict__ pos,
                                                    const TW* __restrict__ cls, const TW* __restrict__ memb,
                                                    const TW* __restrict__ ew, const TW* __restrict__ eb,
                                                    float* __restrict__ H, int n4, int B, int T, int nb, int n_img,
                                                    int D, int tdim, int n_classes, unsigned* err) {
  const int D4 = D / 4;
  pdl_wait();
  pdl_trigger();
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += gridDim.x * blockDim.x) {
    const int tok = i / D4;  // r * T + t
    const int d = (i - tok * D4) * 4;
    const int r = tok / T, t = tok - r * T;
    const bool cond = r < B;
    const int pair = cond ? r : r - B;
    float4 v = load4(pos + (size_t)t * D + d);
    if (t < nb) {
      if (cond) {
        int y = labels[pair];
        if (y < 0 || y >= n_classes) {
          if (d == 0) atomicOr(err, ERR_LABEL);
          y = 0;
        }
        const float4 c = load4(cls + (size_t)y * D + d);
        v.x += c.x; v.y += c.y; v.z += c.z; v.w += c.w;
      }
    } else {
      const int img = t - nb;
      if (mask[(size_t)pair * n_img + img]) {
        const float4 m = load4(memb + d);
        v.x += m.x; v.y += m.y; v.z += m.z; v.w += m.w;
      } else {
        const float* lr = lat + ((size_t)pair * n_img + img) * tdim;
        const float4 bb = load4(eb + d);
        float acc[4] = {bb.x, bb.y, bb.z, bb.w};
        if constexpr (TD > 0) {
          // latent width known at compile time: vector loads of the latent
          // and of each of the 4 weight rows (TD contiguous values)
          float l[TD > 0 ? TD : 4];
#pragma unroll
          for (int j = 0; j < TD; j += 4) {
            const float4 q = *reinterpret_cast<const float4*>(lr + j);
            l[j] = q.x; l[j + 1] = q.y; l[j + 2] = q.z; l[j + 3] = q.w;
          }
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const TW* w = ew + (size_t)(d + k) * TD;
#pragma unroll
            for (int j = 0; j < TD; j += 4) {
              const float4 wq = load4(w + j);
              acc[k] = fmaf(wq.x, l[j], acc[k]);
              acc[k] = fmaf(wq.y, l[j + 1], acc[k]);
              acc[k] = fmaf(wq.z, l[j + 2], acc[k]);
              acc[k] = fmaf(wq.w, l[j + 3], acc[k]);
            }
          }
        } else {
          for (int j = 0; j < tdim; ++j) {
            const float lj = lr[j];
#pragma unroll
            for (int k = 0; k < 4; ++k) acc[k] = fmaf(to_f(ew[(size_t)(d + k) * tdim + j]), lj, acc[k]);
          }
        }
        v.x += acc[0]; v.y += acc[1]; v.z += acc[2]; v.w += acc[3];
      }
    }
    *reinterpret_cast<float4*>(H + (size_t)tok * D + d) = v;
  }
}

cudaError_t launch_embed(const Ctx& c, int dtype, const float* lat, const uint8_t* mask, const int* labels,
                         const void* pos, const void* cls, const void* memb, const void* ew, const void* eb, float* H,
                         int rows, int B, int T, int nb, int n_img, int D, int tdim, int n_classes) {
  if (rows == 0) return cudaSuccess;
  const long long n4l = (long long)rows * T * (D / 4);
  if (n4l >= (1ll << 31)) return cudaErrorInvalidValue;
  const int n4 = (int)n4l;
  long long blocks = (n4l + 255) / 256;
  const long long cap = (long long)c.num_sms * 16;
  if (blocks > cap) blocks = cap;
#define LM_EMBED(TW, TD)                                                                                    \
  launch_pdl(embed_kernel<TW, TD>, dim3((unsigned)blocks), dim3(256), 0, c.stream, lat, mask, labels,        \
             (const TW*)pos, (const TW*)cls, (const TW*)memb, (const TW*)ew, (const TW*)eb, H, n4, B, T, nb, \
             n_img, D, tdim, n_classes, c.err)
  if (dtype == LAZYMAR_BF16) return tdim == 16 ? LM_EMBED(bf16, 16) : LM_EMBED(bf16, 0);
  return tdim == 16 ? LM_EMBED(float, 16) : LM_EMBED(float, 0);
#undef LM_EMBED
}

// ---------------------------------------------------------------------------
// LayerNorm (one warp per row, NV float4 per lane: D = 128 * NV)
// ---------------------------------------------------------------------------
template <int NV>
__device__ __forceinline__ void ln_stats(const float4 (&v)[NV], int D, float eps, float& mean, float& rstd) {
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < NV; ++i) s += (v[i].x + v[i].y) + (v[i].z + v[i].w);
  mean = warp_sum(s) / (float)D;
  float q = 0.f;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const float a = v[i].x - mean, b = v[i].y - mean, cc = v[i].z - mean, d = v[i].w - mean;
    q += (a * a + b * b) + (cc * cc + d * d);
  }
  rstd = rsqrtf(warp_sum(q) / (float)D + eps);
}

// Four gain or shift values as loaded (packed bf16 or fp32). They are weights,
// which no kernel writes, so the row kernels load them before waiting for the
// predecessor grid.
template <typename TO> struct Param4;
template <> struct Param4<bf16> {
  uint2 u;
  __device__ __forceinline__ void load(const bf16* p) { u = *reinterpret_cast<const uint2*>(p); }
  __device__ __forceinline__ float4 get() const {
    const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
    const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
    return make_float4(a.x, a.y, b.x, b.y);
  }
};
template <> struct Param4<float> {
  float4 u;
  __device__ __forceinline__ void load(const float* p) { u = *reinterpret_cast<const float4*>(p); }
  __device__ __forceinline__ float4 get() const { return u; }
};

template <typename TO>
__device__ __forceinline__ void ln_write4(TO* y, const Param4<TO>& gp, const Param4<TO>& bp, int col, float4 x,
                                          float mean, float rstd) {
  float o[4] = {x.x, x.y, x.z, x.w};
  const float4 g4 = gp.get(), b4 = bp.get();
  const float gv[4] = {g4.x, g4.y, g4.z, g4.w}, bv[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) o[k] = (o[k] - mean) * rstd * gv[k] + bv[k];
  if constexpr (sizeof(TO) == 2) {
    __nv_bfloat162 h0 = __floats2bfloat162_rn(o[0], o[1]), h1 = __floats2bfloat162_rn(o[2], o[3]);
    uint2 u;
    u.x = *reinterpret_cast<uint32_t*>(&h0);
    u.y = *reinterpret_cast<uint32_t*>(&h1);
    *reinterpret_cast<uint2*>(y + col) = u;
  } else {
    *reinterpret_cast<float4*>(y + col) = make_float4(o[0], o[1], o[2], o[3]);
  }
}

template <typename TO, int NV>
__global__ void __launch_bounds__(256) layernorm_kernel(const float* __restrict__ x, const int* __restrict__ row_map,
                                                        const TO* __restrict__ g, const TO* __restrict__ b,
                                                        TO* __restrict__ y, float* __restrict__ x_copy, int M, int D,
                                                        float eps) {
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  Param4<TO> gp[NV], bp[NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    gp[i].load(g + 4 * (lane + 32 * i));
    bp[i].load(b + 4 * (lane + 32 * i));
  }
  pdl_wait();
  pdl_trigger();
  if (row >= M) return;
  const int src = row_map ? row_map[row] : row;
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)src * D);
  float4 v[NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) v[i] = xr[lane + 32 * i];
  if (x_copy) {
    float4* cr = reinterpret_cast<float4*>(x_copy + (size_t)row * D);
#pragma unroll
    for (int i = 0; i < NV; ++i) cr[lane + 32 * i] = v[i];
  }
  float mean, rstd;
  ln_stats<NV>(v, D, eps, mean, rstd);
  TO* yr = y + (size_t)row * D;
#pragma unroll
  for (int i = 0; i < NV; ++i) ln_write4<TO>(yr, gp[i], bp[i], 4 * (lane + 32 * i), v[i], mean, rstd);
}

// Four values to four E4M3 bytes (round to nearest even, saturating at the
// largest finite value 448), the A operand of an 8-bit GEMM.
__device__ __forceinline__ uint32_t pack_e4m3x4(float a, float b, float c, float d) {
  const uint32_t lo = __nv_cvt_float2_to_fp8x2(make_float2(a, b), __NV_SATFINITE, __NV_E4M3);
  const uint32_t hi = __nv_cvt_float2_to_fp8x2(make_float2(c, d), __NV_SATFINITE, __NV_E4M3);
  return lo | (hi << 16);
}

// layernorm_kernel with an E4M3 output (gain and shift in TG): the A operand
// of the E4M3 Q/K/V projection.
template <typename TG, int NV>
__global__ void __launch_bounds__(256) layernorm_e4m3_kernel(const float* __restrict__ x,
                                                             const int* __restrict__ row_map,
                                                             const TG* __restrict__ g, const TG* __restrict__ b,
                                                             uint8_t* __restrict__ y, float* __restrict__ x_copy,
                                                             int M, int D, float eps) {
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  Param4<TG> gp[NV], bp[NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    gp[i].load(g + 4 * (lane + 32 * i));
    bp[i].load(b + 4 * (lane + 32 * i));
  }
  pdl_wait();
  pdl_trigger();
  if (row >= M) return;
  const int src = row_map ? row_map[row] : row;
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)src * D);
  float4 v[NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) v[i] = xr[lane + 32 * i];
  if (x_copy) {
    float4* cr = reinterpret_cast<float4*>(x_copy + (size_t)row * D);
#pragma unroll
    for (int i = 0; i < NV; ++i) cr[lane + 32 * i] = v[i];
  }
  float mean, rstd;
  ln_stats<NV>(v, D, eps, mean, rstd);
  uint8_t* yr = y + (size_t)row * D;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const int col = 4 * (lane + 32 * i);
    const float4 gg = gp[i].get(), bb = bp[i].get();
    *reinterpret_cast<uint32_t*>(yr + col) =
        pack_e4m3x4((v[i].x - mean) * rstd * gg.x + bb.x, (v[i].y - mean) * rstd * gg.y + bb.y,
                    (v[i].z - mean) * rstd * gg.z + bb.z, (v[i].w - mean) * rstd * gg.w + bb.w);
  }
}

// E4M3 weights with one scale per row (output channel): scale = max|w| / 448
// (1 for an all-zero row), q = e4m3(w / scale). One warp per row.
__global__ void __launch_bounds__(256) quantize_rows_e4m3_kernel(const bf16* __restrict__ w, int rows, int cols,
                                                                 uint8_t* __restrict__ q, float* __restrict__ scale) {
  pdl_wait();
  pdl_trigger();
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= rows) return;
  const bf16* wr = w + (size_t)row * cols;
  float amax = 0.f;
  for (int k = lane * 8; k < cols; k += 256) {
    float f[8];
    Vec<bf16, 8>::load(wr + k, f);
#pragma unroll
    for (int i = 0; i < 8; ++i) amax = fmaxf(amax, fabsf(f[i]));
  }
  amax = warp_max(amax);
  const float s = amax > 0.f ? amax / 448.f : 1.f;
  if (lane == 0) scale[row] = s;
  uint8_t* qr = q + (size_t)row * cols;
  for (int k = lane * 8; k < cols; k += 256) {
    float f[8];
    Vec<bf16, 8>::load(wr + k, f);
    uint2 u;
    u.x = pack_e4m3x4(f[0] / s, f[1] / s, f[2] / s, f[3] / s);
    u.y = pack_e4m3x4(f[4] / s, f[5] / s, f[6] / s, f[7] / s);
    *reinterpret_cast<uint2*>(qr + k) = u;
  }
}

cudaError_t launch_quantize_e4m3(const Ctx& c, const void* w, int rows, int cols, void* q, float* scale) {
  if (rows == 0) return cudaSuccess;
  if (cols % 8 != 0) return cudaErrorInvalidValue;
  return launch_pdl(quantize_rows_e4m3_kernel, dim3((unsigned)((rows + 7) / 8)), dim3(256), 0, c.stream,
                    static_cast<const bf16*>(w), rows, cols, static_cast<uint8_t*>(q), scale);
}

template <typename TO, int NV>
__global__ void __launch_bounds__(256) final_ln_kernel(const float* __restrict__ x, const int* __restrict__ row_map,
                                                       int T, int nb, int n_img, const TO* __restrict__ g,
                                                       const TO* __restrict__ b, TO* __restrict__ z, int M, int D,
                                                       float eps) {
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  Param4<TO> gp[NV], bp[NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    gp[i].load(g + 4 * (lane + 32 * i));
    bp[i].load(b + 4 * (lane + 32 * i));
  }
  pdl_wait();
  pdl_trigger();
  if (row >= M) return;
  const int tok = row_map ? row_map[row] : row;
  const int r = tok / T, t = tok - r * T;
  if (t < nb) return;
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)row * D);
  float4 v[NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) v[i] = xr[lane + 32 * i];
  float mean, rstd;
  ln_stats<NV>(v, D, eps, mean, rstd);
  TO* zr = z + ((size_t)r * n_img + (t - nb)) * D;
#pragma unroll
  for (int i = 0; i < NV; ++i) ln_write4<TO>(zr, gp[i], bp[i], 4 * (lane + 32 * i), v[i], mean, rstd);
}

#define LM_LN_DISPATCH(KERNEL, TO, ...)                                                          \
  switch (D / 128) {                                                                             \
    case 1: return launch_pdl(KERNEL<TO, 1>, dim3(grid), dim3(256), 0, c.stream, __VA_ARGS__);   \
    case 2: return launch_pdl(KERNEL<TO, 2>, dim3(grid), dim3(256), 0, c.stream, __VA_ARGS__);   \
    case 4: return launch_pdl(KERNEL<TO, 4>, dim3(grid), dim3(256), 0, c.stream, __VA_ARGS__);   \
    case 6: return launch_pdl(KERNEL<TO, 6>, dim3(grid), dim3(256), 0, c.stream, __VA_ARGS__);   \
    case 8: return launch_pdl(KERNEL<TO, 8>, dim3(grid), dim3(256), 0, c.stream, __VA_ARGS__);   \
    case 10: return launch_pdl(KERNEL<TO, 10>, dim3(grid), dim3(256), 0, c.stream, __VA_ARGS__); \
    case 12: return launch_pdl(KERNEL<TO, 12>, dim3(grid), dim3(256), 0, c.stream, __VA_ARGS__); \
    case 16: return launch_pdl(KERNEL<TO, 16>, dim3(grid), dim3(256), 0, c.stream, __VA_ARGS__); \
    default: return cudaErrorInvalidValue;                                                       \
  }

bool layernorm_width_ok(int D) {
  const int k = D / 128;
  return D % 128 == 0 && (k == 1 || k == 2 || k == 4 || k == 6 || k == 8 || k == 10 || k == 12 || k == 16);
}

cudaError_t launch_layernorm(const Ctx& c, int dtype, const float* x, const int* row_map, const void* g,
                             const void* b, void* y, float* x_copy, int M, int D, float eps) {
  if (M == 0) return cudaSuccess;
  const unsigned grid = (unsigned)((M + 7) / 8);
  if (dtype == LAZYMAR_E4M3) {
    // bf16 gain and shift, E4M3 output
    LM_LN_DISPATCH(layernorm_e4m3_kernel, bf16, x, row_map, (const bf16*)g, (const bf16*)b, (uint8_t*)y, x_copy, M,
                   D, eps)
  } else if (dtype == LAZYMAR_BF16) {
    LM_LN_DISPATCH(layernorm_kernel, bf16, x, row_map, (const bf16*)g, (const bf16*)b, (bf16*)y, x_copy, M, D, eps)
  } else {
    LM_LN_DISPATCH(layernorm_kernel, float, x, row_map, (const float*)g, (const float*)b, (float*)y, x_copy, M, D,
                   eps)
  }
  return cudaGetLastError();
}

cudaError_t launch_final_ln(const Ctx& c, int dtype, const float* x, const int* row_map, int T, int nb, int n_img,
                            const void* g, const void* b, void* z, int M, int D, float eps) {
  if (M == 0) return cudaSuccess;
  const unsigned grid = (unsigned)((M + 7) / 8);
  if (dtype == LAZYMAR_BF16) {
    LM_LN_DISPATCH(final_ln_kernel, bf16, x, row_map, T, nb, n_img, (const bf16*)g, (const bf16*)b, (bf16*)z, M, D,
                   eps)
  } else {
    LM_LN_DISPATCH(final_ln_kernel, float, x, row_map, T, nb, n_img, (const float*)g, (const float*)b, (float*)z, M,
                   D, eps)
  }
  return cudaGetLastError();
}

// fp32 -> dtype copy (the block output features used as the selection
// criterion when criterion == FEATURE).
template <typename TO>
__global__ void cast_kernel(const float* __restrict__ x, TO* __restrict__ y, size_t n) {
  pdl_wait();
  pdl_trigger();
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x)
    y[i] = from_f<TO>(x[i]);
}
cudaError_t launch_cast(const Ctx& c, int dtype, const float* x, void* y, size_t n) {
  if (n == 0) return cudaSuccess;
  const unsigned grid = (unsigned)((n + 255) / 256 < (size_t)c.num_sms * 8 ? (n + 255) / 256 : (size_t)c.num_sms * 8);
  if (dtype == LAZYMAR_BF16) return launch_pdl(cast_kernel<bf16>, dim3(grid), dim3(256), 0, c.stream, x, (bf16*)y, n);
  return launch_pdl(cast_kernel<float>, dim3(grid), dim3(256), 0, c.stream, x, (float*)y, n);
}

// Gathers the selected tokens' query rows and residual rows into compact
// buffers: row i of qc / xc is row row_map[i] of q / x. One CTA per row pair,
// 16-byte vectors; q rows are D elements of TQ, x rows D fp32 values.
template <typename TQ>
__global__ void __launch_bounds__(128) gather_rows_kernel(const TQ* __restrict__ q, const float* __restrict__ x,
                                                          const int* __restrict__ row_map, TQ* __restrict__ qc,
                                                          float* __restrict__ xc, int D) {
  pdl_wait();
  pdl_trigger();
  const size_t dst = blockIdx.x, src = (size_t)row_map[blockIdx.x];
  const int nq = D * (int)sizeof(TQ) / 16, nx = D / 4;
  const uint4* qs = reinterpret_cast<const uint4*>(q + src * D);
  uint4* qd = reinterpret_cast<uint4*>(qc + dst * D);
  const uint4* xs = reinterpret_cast<const uint4*>(x + src * D);
  uint4* xd = reinterpret_cast<uint4*>(xc + dst * D);
  for (int i = threadIdx.x; i < nq + nx; i += blockDim.x) {
    if (i < nq) qd[i] = qs[i];
    else xd[i - nq] = xs[i - nq];
  }
}
cudaError_t launch_gather_rows(const Ctx& c, int dtype, const void* q, const float* x, const int* row_map, void* qc,
                               float* xc, int M, int D) {
  if (M == 0) return cudaSuccess;
  if (dtype == LAZYMAR_BF16)
    return launch_pdl(gather_rows_kernel<bf16>, dim3((unsigned)M), dim3(128), 0, c.stream, (const bf16*)q, x, row_map,
                      (bf16*)qc, xc, D);
  return launch_pdl(gather_rows_kernel<float>, dim3((unsigned)M), dim3(128), 0, c.stream, (const float*)q, x, row_map,
                    (float*)qc, xc, D);
}

// ---------------------------------------------------------------------------
// Classifier-free guidance with the condition cache
// ---------------------------------------------------------------------------
template <typename T>
__device__ __forceinline__ void cfg_elems(int mode, float gamma, const float* c, const float* u_in, float* d, float* u,
                                          float* g, int n) {
  for (int i = 0; i < n; ++i) {
    float uu;
    if (mode == LAZYMAR_CFG_REUSE) {
      uu = c[i] - d[i];
    } else {
      uu = u_in[i];
      if (mode == LAZYMAR_CFG_REFRESH) d[i] = c[i] - uu;
    }
    u[i] = uu;
    g[i] = uu + gamma * (c[i] - uu);
  }
}

template <typename T>
__global__ void __launch_bounds__(256) cfg_kernel(int mode, const T* __restrict__ zc, const T* __restrict__ zu,
                                                  T* __restrict__ delta, float gamma, size_t n, T* __restrict__ zu_out,
                                                  T* __restrict__ g_out) {
  constexpr int V = 16 / sizeof(T);
  pdl_wait();
  pdl_trigger();
  const size_t nv = n / V;
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < nv; i += stride) {
    const size_t o = i * V;
    float c[V], u[V], d[V], uo[V], g[V];
    Vec<T, V>::load(zc + o, c);
    if (mode == LAZYMAR_CFG_REUSE) Vec<T, V>::load(delta + o, d);
    else Vec<T, V>::load(zu + o, u);
    cfg_elems<T>(mode, gamma, c, u, d, uo, g, V);
    if (mode == LAZYMAR_CFG_REFRESH) Vec<T, V>::store(delta + o, d);
    if (mode == LAZYMAR_CFG_REUSE && zu_out) Vec<T, V>::store(zu_out + o, uo);
    if (g_out) Vec<T, V>::store(g_out + o, g);
  }
  // scalar tail
  const size_t tail0 = nv * V;
  const size_t gt = blockIdx.x * (size_t)blockDim.x + threadIdx.x;
  if (gt < n - tail0) {
    const size_t o = tail0 + gt;
    float c = to_f(zc[o]), u = 0.f, d = 0.f, uo, g;
    if (mode == LAZYMAR_CFG_REUSE) d = to_f(delta[o]);
    else u = to_f(zu[o]);
    cfg_elems<T>(mode, gamma, &c, &u, &d, &uo, &g, 1);
    if (mode == LAZYMAR_CFG_REFRESH) delta[o] = from_f<T>(d);
    if (mode == LAZYMAR_CFG_REUSE && zu_out) zu_out[o] = from_f<T>(uo);
    if (g_out) g_out[o] = from_f<T>(g);
  }
}

// Copies every segment of L, block-strided over 16-byte vectors where both
// ends are 16-byte aligned, byte by byte for the rest.
__global__ void __launch_bounds__(256) copy_list_kernel(const CopyList L) {
  pdl_wait();
  pdl_trigger();
  const size_t t = blockIdx.x * (size_t)blockDim.x + threadIdx.x, stride = (size_t)gridDim.x * blockDim.x;
  for (int s = 0; s < L.n; ++s) {
    const uint8_t* src = static_cast<const uint8_t*>(L.src[s]);
    uint8_t* dst = static_cast<uint8_t*>(L.dst[s]);
    const size_t n = L.bytes[s];
    size_t done = 0;
    if (((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15u) == 0) {
      const size_t nv = n / 16;
      for (size_t i = t; i < nv; i += stride)
        reinterpret_cast<uint4*>(dst)[i] = reinterpret_cast<const uint4*>(src)[i];
      done = nv * 16;
    }
    for (size_t i = done + t; i < n; i += stride) dst[i] = src[i];
  }
}

cudaError_t launch_copy_list(const Ctx& c, const CopyList& L) {
  if (L.n <= 0) return cudaSuccess;
  if (L.n > kMaxCopySegs) return cudaErrorInvalidValue;
  size_t total = 0;
  for (int s = 0; s < L.n; ++s) total += L.bytes[s];
  size_t blocks = (total / 16 + 1023) / 1024;  // about four vectors per thread
  const size_t cap = (size_t)c.num_sms * 2;
  if (blocks > cap) blocks = cap;
  if (blocks == 0) blocks = 1;
  return launch_pdl(copy_list_kernel, dim3((unsigned)blocks), dim3(256), 0, c.stream, L);
}

cudaError_t launch_cfg(const Ctx& c, int dtype, int mode, const void* zc, const void* zu, void* delta, float gamma,
                       size_t n, void* zu_out, void* g_out) {
  if (n == 0) return cudaSuccess;
  const size_t V = dtype == LAZYMAR_BF16 ? 8 : 4;
  size_t blocks = (n / V + 255) / 256;
  const size_t cap = (size_t)c.num_sms * 8;
  if (blocks > cap) blocks = cap;
  if (blocks == 0) blocks = 1;
  if (dtype == LAZYMAR_BF16)
    return launch_pdl(cfg_kernel<bf16>, dim3((unsigned)blocks), dim3(256), 0, c.stream, mode, (const bf16*)zc,
                      (const bf16*)zu, (bf16*)delta, gamma, n, (bf16*)zu_out, (bf16*)g_out);
  return launch_pdl(cfg_kernel<float>, dim3((unsigned)blocks), dim3(256), 0, c.stream, mode, (const float*)zc,
                    (const float*)zu, (float*)delta, gamma, n, (float*)zu_out, (float*)g_out);
}

}  // namespace lm
