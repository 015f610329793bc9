// Diffusion head (Sec. 4.1): the per-token denoiser that draws the continuous
// latent of every token decoded at a decoding step, run for the standard
// ancestral sampler over 100 kept steps of a cosine noise schedule, with
// classifier-free guidance on its noise prediction.
//
// One sampling call runs, for the R = 2M rows (M tokens x {cond, uncond}):
//   gather z rows -> W_c z + b_c (tcgen05 GEMM)                      once
//   per chunk of kept steps (they depend on the embeddings only):
//     SiLU(t_emb[j] + c_emb) for every step j of the chunk  (row-wise)
//     all blocks' and the final modulations of those steps  (one tcgen05 GEMM)
//   per kept step j = n_steps-1 .. 0:
//     block 0: input projection + LN + modulation           (row-wise; inside
//              a chunk done by the previous step's final kernel)
//     per block: fc1 + SiLU (GEMM), fc2 gated into the fp32 residual (GEMM),
//                next LN + modulation                        (row-wise)
//     final LN + modulation, output projection, guidance, the sampler
//     update of x, and the next step's block-0 rows          (one CTA per token)
// The loop runs eagerly on the first call with a given (z buffer, B, n_img,
// n_new), is captured into a CUDA graph on the second and replayed after that.
// The guidance scale and temperature are read from device memory, so they may
// change between calls. The time embeddings of the kept steps depend on the
// weights only and are computed once at create.
#include <cmath>
#include <cstring>
#include <map>
#include <tuple>
#include <string>
#include <vector>

#include "lazymar_internal.cuh"

namespace lm {
namespace hd {

// Four packed bf16 values as floats.
__device__ __forceinline__ void unpack4_bf16(uint2 u, float* v) {
  const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
  const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
  v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y;
}
// Four consecutive bf16 values (8-byte aligned) as floats.
__device__ __forceinline__ void load4_bf16(const bf16* p, float* v) {
  unpack4_bf16(*reinterpret_cast<const uint2*>(p), v);
}

// Sinusoidal features of the kept training steps: [cos(t f_i), sin(t f_i)],
// f_i = 10000^(-i / half), in double precision (t f_i reaches ~1000 rad).
__global__ void sinusoid_kernel(const int* __restrict__ t, bf16* __restrict__ out, int n, int half) {
  const int j = blockIdx.x;
  if (j >= n) return;
  for (int i = threadIdx.x; i < half; i += blockDim.x) {
    const double f = exp(-log(10000.0) * (double)i / (double)half);
    const double a = (double)t[j] * f;
    out[(size_t)j * 2 * half + i] = __float2bfloat16_rn((float)cos(a));
    out[(size_t)j * 2 * half + half + i] = __float2bfloat16_rn((float)sin(a));
  }
}

// Rows of z for the decoded tokens: row m < M is pair b = m / n_new's
// conditional row at position pos[m], row M + m its unconditional row.
template <typename TZ>
__global__ void __launch_bounds__(256) gather_z_kernel(const TZ* __restrict__ z, const int* __restrict__ pos, int B,
                                                       int n_img, int D, int M, int n_new, bf16* __restrict__ out,
                                                       unsigned* err) {
  pdl_wait();
  pdl_trigger();
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (r >= 2 * M) return;
  const int m = r < M ? r : r - M;
  const int b = m / n_new;
  int p = pos[m];
  if (p < 0 || p >= n_img) {
    if (lane == 0) atomicOr(err, ERR_INDEX);
    p = 0;
  }
  const size_t src = ((size_t)(r < M ? b : B + b) * n_img + p) * D;
  for (int c = lane; c < D; c += 32) out[(size_t)r * D + c] = __float2bfloat16_rn(to_f(z[src + c]));
}

// For cnt kept steps j0, j0 - 1, ..: sy[k R + r] = SiLU(t_emb[j0 - k] +
// c_emb[r]), 8 bf16 per thread.
__global__ void __launch_bounds__(256) cond_silu_kernel(const bf16* __restrict__ temb, int j0, int cnt,
                                                        const bf16* __restrict__ cemb, bf16* __restrict__ sy, int R,
                                                        int w) {
  pdl_wait();
  pdl_trigger();
  const int w8 = w / 8;
  const int per = R * w8;
  const int n = cnt * per;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
    const int k = i / per, rem = i - k * per;
    const int c8 = rem % w8;
    float a[8], b[8];
    Vec<bf16, 8>::load(temb + (size_t)(j0 - k) * w + c8 * 8, a);
    Vec<bf16, 8>::load(cemb + (size_t)rem * 8, b);
#pragma unroll
    for (int k = 0; k < 8; ++k) a[k] = silu(a[k] + b[k]);
    Vec<bf16, 8>::store(sy + (size_t)i * 8, a);
  }
}

// One row by one warp, VPL float4 per lane (w = 128 VPL): the row's
// LayerNorm without gain or shift, modulated by (1 + scale) and shift from
// the modulation row mr, to bf16 at hr. With INPROJ the row is first computed
// as W_in x + b_in from the token's latent xm (W_in stored transposed,
// [td, w]) and stored to xr; otherwise it is read from xr.
template <int VPL, bool INPROJ>
__device__ __forceinline__ void ln_mod_row(float* __restrict__ xr, const float* __restrict__ xm,
                                           const bf16* __restrict__ win_t, const bf16* __restrict__ bin,
                                           const bf16* __restrict__ mr, int shift_off, int scale_off,
                                           bf16* __restrict__ hr, int td, float eps, int lane) {
  constexpr int w = 128 * VPL;
  float4 v[VPL];
  // the modulation does not depend on the row: its loads go out first
  uint2 shp[VPL], scp[VPL];
#pragma unroll
  for (int i = 0; i < VPL; ++i) {
    const int c = 4 * (lane + 32 * i);
    shp[i] = *reinterpret_cast<const uint2*>(mr + shift_off + c);
    scp[i] = *reinterpret_cast<const uint2*>(mr + scale_off + c);
  }
  if (INPROJ) {
    // latent index k outermost: each k issues VPL independent weight loads
#pragma unroll
    for (int i = 0; i < VPL; ++i) {
      float a[4];
      load4_bf16(bin + 4 * (lane + 32 * i), a);
      v[i] = make_float4(a[0], a[1], a[2], a[3]);
    }
#pragma unroll 4
    for (int k = 0; k < td; ++k) {
      const float xk = xm[k];
      const bf16* wrow = win_t + (size_t)k * w;
#pragma unroll
      for (int i = 0; i < VPL; ++i) {
        float wk[4];
        load4_bf16(wrow + 4 * (lane + 32 * i), wk);
        v[i].x = fmaf(xk, wk[0], v[i].x);
        v[i].y = fmaf(xk, wk[1], v[i].y);
        v[i].z = fmaf(xk, wk[2], v[i].z);
        v[i].w = fmaf(xk, wk[3], v[i].w);
      }
    }
#pragma unroll
    for (int i = 0; i < VPL; ++i) reinterpret_cast<float4*>(xr)[lane + 32 * i] = v[i];
  } else {
#pragma unroll
    for (int i = 0; i < VPL; ++i) v[i] = reinterpret_cast<const float4*>(xr)[lane + 32 * i];
  }
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < VPL; ++i) s += (v[i].x + v[i].y) + (v[i].z + v[i].w);
  const float mean = warp_sum(s) * (1.f / w);
  float q = 0.f;
#pragma unroll
  for (int i = 0; i < VPL; ++i) {
    const float a = v[i].x - mean, b = v[i].y - mean, c = v[i].z - mean, d = v[i].w - mean;
    q += (a * a + b * b) + (c * c + d * d);
  }
  const float rstd = rsqrtf(warp_sum(q) * (1.f / w) + eps);
#pragma unroll
  for (int i = 0; i < VPL; ++i) {
    const int c = 4 * (lane + 32 * i);
    float sh[4], sc[4];
    unpack4_bf16(shp[i], sh);
    unpack4_bf16(scp[i], sc);
    const float o0 = fmaf((v[i].x - mean) * rstd, 1.f + sc[0], sh[0]);
    const float o1 = fmaf((v[i].y - mean) * rstd, 1.f + sc[1], sh[1]);
    const float o2 = fmaf((v[i].z - mean) * rstd, 1.f + sc[2], sh[2]);
    const float o3 = fmaf((v[i].w - mean) * rstd, 1.f + sc[3], sh[3]);
    uint2 u;
    u.x = pack_bf16(o0, o1);
    u.y = pack_bf16(o2, o3);
    *reinterpret_cast<uint2*>(hr + c) = u;
  }
}

// One warp per row r of R (ln_mod_row; with INPROJ from the latent of
// token r mod M).
template <int VPL, bool INPROJ>
__global__ void __launch_bounds__(256) ln_mod_kernel(float* __restrict__ xh, const float* __restrict__ x,
                                                     const bf16* __restrict__ win_t, const bf16* __restrict__ bin,
                                                     const bf16* __restrict__ mod, int ldm, int shift_off,
                                                     int scale_off, bf16* __restrict__ hb, int R, int M, int td,
                                                     float eps) {
  pdl_wait();
  pdl_trigger();
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (r >= R) return;
  constexpr int w = 128 * VPL;
  ln_mod_row<VPL, INPROJ>(xh + (size_t)r * w, x + (size_t)(r < M ? r : r - M) * td, win_t, bin,
                          mod + (size_t)r * ldm, shift_off, scale_off, hb + (size_t)r * w, td, eps, lane);
}

// Schedule constants of one kept step: mean = a_x x - a_eps eps; the log
// variance interpolates between log_beta (v = 1) and log_post (v = -1).
struct StepConst {
  float a_x, a_eps, log_beta, log_post;
  int last;  // j == 0: no noise
};

// One CTA per token m: final LayerNorm + modulation of rows m (cond) and
// M + m (uncond), the output projection [eps, v] of both, guidance and the
// sampler update of x[m]. With `eval_out` the raw outputs of both rows are
// written there instead and x is left alone. With next_mod the CTA then runs
// the next kept step's block-0 input projection, LayerNorm and modulation of
// both rows from the updated x (ln_mod_row with that step's modulations), so
// the next network evaluation starts at its first GEMM: xh and hb rows of
// the token hold what ln_mod_kernel would write. xh_next is xh itself, so
// neither is restrict: the CTA reads its two rows before the barrier that
// precedes their rewrite.
constexpr int FIN_THREADS = 256;
template <int VPL>
__global__ void __launch_bounds__(FIN_THREADS, 2) final_kernel(const float* xh, const bf16* __restrict__ mod,
                                                            int ldm, int shift_off, int scale_off,
                                                            const bf16* __restrict__ wout, const float* __restrict__ bout,
                                                            int M, int w, int td, float eps, StepConst sc,
                                                            const float* __restrict__ params, float* __restrict__ x,
                                                            const float* __restrict__ noise, float* __restrict__ x_done,
                                                            float* __restrict__ eval_out, const bf16* __restrict__ next_mod,
                                                            const bf16* __restrict__ win_t, const bf16* __restrict__ bin,
                                                            float* xh_next, bf16* __restrict__ hb) {
  extern __shared__ float sm[];
  float* h = sm;                        // [2][w] modulated rows
  float* o = sm + 2 * w;                // [2][2 td] outputs
  float* red = o + 4 * td;              // [2][FIN_THREADS / 32] partial sums
  float* xs = red + 2 * (FIN_THREADS / 32);  // [td] the updated latent
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int NWARP = FIN_THREADS / 32;
  // The output weights (no kernel writes them) of this warp's output columns
  // oc = warp + 8 i go to L1 while the predecessor grid finishes.
  for (int oc = warp; oc < 2 * td; oc += NWARP)
    for (int c = 8 * lane; c < w; c += 256)
      asm volatile("prefetch.global.L1 [%0];" ::"l"(wout + (size_t)oc * w + c));
  pdl_wait();
  pdl_trigger();
  const int m = blockIdx.x;
  if (m >= M) return;
  // both rows at once: threads 0-127 normalise row m (conditional), threads
  // 128-255 row M + m (unconditional); each thread holds w / 128 <= 16
  // columns t + 128 i, and the modulation loads go out with the row's
  {
    static_assert(FIN_THREADS == 256, "two rows of 128 threads");
    const int g = tid >> 7, t = tid & 127;
    const int r = g == 0 ? m : M + m;
    const int n = w >> 7;
    const float* xr = xh + (size_t)r * w;
    const bf16* mr = mod + (size_t)r * ldm;
    float v[16], sh[16], scl[16];
    float sum = 0.f;
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if (i < n) {
        const int c = t + 128 * i;
        sh[i] = to_f(mr[shift_off + c]);
        scl[i] = to_f(mr[scale_off + c]);
        v[i] = xr[c];
        sum += v[i];
      }
    sum = warp_sum(sum);
    if (lane == 0) red[warp] = sum;
    __syncthreads();
    const float mean = ((red[4 * g] + red[4 * g + 1]) + (red[4 * g + 2] + red[4 * g + 3])) / (float)w;
    float q = 0.f;
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if (i < n) {
        const float d = v[i] - mean;
        q = fmaf(d, d, q);
      }
    q = warp_sum(q);
    if (lane == 0) red[NWARP + warp] = q;
    __syncthreads();
    const float qt = (red[NWARP + 4 * g] + red[NWARP + 4 * g + 1]) + (red[NWARP + 4 * g + 2] + red[NWARP + 4 * g + 3]);
    const float rstd = rsqrtf(qt / (float)w + eps);
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if (i < n) h[g * w + t + 128 * i] = fmaf((v[i] - mean) * rstd, 1.f + scl[i], sh[i]);
    __syncthreads();
  }
  // 2 rows x 2 td outputs: warp w takes output columns oc = w + 8 i, two at a
  // time, each for both rows (one weight load serves two rows); each lane
  // takes 8 consecutive columns per 256 (one 16-byte weight load, w % 128 == 0)
  for (int oa = warp; oa < 2 * td; oa += 2 * NWARP) {
    const int ob = oa + NWARP;
    const bool two = ob < 2 * td;
    const bf16* wa = wout + (size_t)oa * w;
    const bf16* wb = wout + (size_t)(two ? ob : oa) * w;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};  // (oa, row 0), (oa, row 1), (ob, row 0), (ob, row 1)
    for (int c = 8 * lane; c < w; c += 256) {
      float va[8], vb[8];
      Vec<bf16, 8>::load(wa + c, va);
      Vec<bf16, 8>::load(wb + c, vb);
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const float4 h0 = *reinterpret_cast<const float4*>(h + r * w + c);
        const float4 h1 = *reinterpret_cast<const float4*>(h + r * w + c + 4);
        const float hv[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          acc[r] = fmaf(hv[e], va[e], acc[r]);
          acc[2 + r] = fmaf(hv[e], vb[e], acc[2 + r]);
        }
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[i] = warp_sum(acc[i]);
    if (lane == 0) {
      o[oa] = acc[0] + bout[oa];
      o[2 * td + oa] = acc[1] + bout[oa];
      if (two) {
        o[ob] = acc[2] + bout[ob];
        o[2 * td + ob] = acc[3] + bout[ob];
      }
    }
  }
  __syncthreads();
  if (eval_out) {
    for (int k = tid; k < 4 * td; k += FIN_THREADS) {
      const int s = k / (2 * td), oc = k - s * 2 * td;
      eval_out[(size_t)(s == 0 ? m : M + m) * 2 * td + oc] = o[k];
    }
    return;
  }
  const float gamma = params[0], temperature = params[1];
  for (int k = tid; k < td; k += FIN_THREADS) {
    const float ec = o[k], vc = o[td + k], eu = o[2 * td + k];
    const float e = fmaf(gamma, ec - eu, eu);
    const float xv = x[(size_t)m * td + k];
    float nx = fmaf(sc.a_x, xv, -sc.a_eps * e);
    if (!sc.last) {
      const float frac = 0.5f * (vc + 1.f);
      const float log_var = fmaf(frac, sc.log_beta - sc.log_post, sc.log_post);
      nx = fmaf(expf(0.5f * log_var) * temperature, noise[(size_t)m * td + k], nx);
    }
    x[(size_t)m * td + k] = nx;
    if (x_done) x_done[(size_t)m * td + k] = nx;
    xs[k] = nx;
  }
  if (next_mod) {
    __syncthreads();
    if (warp < 2) {
      const int r = warp == 0 ? m : M + m;
      ln_mod_row<VPL, true>(xh_next + (size_t)r * w, xs, win_t, bin, next_mod + (size_t)r * ldm, 0, w,
                            hb + (size_t)r * w, td, eps, lane);
    }
  }
}

}  // namespace hd
}  // namespace lm

// ---------------------------------------------------------------------------
// Handle and C ABI
// ---------------------------------------------------------------------------
using namespace lm;

namespace {

lazymar_status head_fail(lazymar_status s, const std::string& msg) { return report_error(s, msg.c_str()); }
lazymar_status head_cuda(cudaError_t e, const char* what) {
  return head_fail(LAZYMAR_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}
#define HD_CUDA(expr)                                     \
  do {                                                    \
    cudaError_t e_ = (expr);                              \
    if (e_ != cudaSuccess) return head_cuda(e_, #expr);   \
  } while (0)
#define HD_TRY(expr)                 \
  do {                               \
    lazymar_status s_ = (expr);      \
    if (s_ != LAZYMAR_OK) return s_; \
  } while (0)

uint16_t to_bf16_bits(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7fffffffu) > 0x7f800000u) return 0x7fc0;
  u += 0x7fffu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

bool width_ok(int w) {
  const int k = w / 128;
  return w % 128 == 0 && k >= 1 && k <= 16;
}

}  // namespace

struct lazymar_head {
  lazymar_head_config cfg{};
  int dev = 0, num_sms = 0, w = 0, td = 0, nmod = 0;
  int chunk = 1;  // kept steps whose modulations are computed by one GEMM
  uint8_t* arena = nullptr;
  // weights (bf16 unless noted)
  bf16 *t_w1 = nullptr, *t_b1 = nullptr, *t_w2 = nullptr, *t_b2 = nullptr, *c_w = nullptr, *c_b = nullptr;
  bf16 *in_wt = nullptr, *in_b = nullptr, *ada_w = nullptr, *ada_b = nullptr, *out_w = nullptr;
  float* out_b = nullptr;  // fp32
  std::vector<bf16*> w1, b1, w2, b2;
  bf16* temb = nullptr;  // [n_steps, w]
  std::vector<hd::StepConst> sched;
  // per call
  int* pos = nullptr;
  float *noise = nullptr, *x = nullptr, *xh = nullptr, *eval = nullptr, *params = nullptr, *x_done = nullptr;
  bf16 *zg = nullptr, *cemb = nullptr, *sy = nullptr, *mod = nullptr, *hb = nullptr, *u = nullptr;
  unsigned* err = nullptr;
  float host_params[2] = {0.f, 0.f};
  // counters
  long long launches = 0;
  double flops = 0.0;
  struct Graph {
    cudaGraphExec_t exec = nullptr;
    int eager_runs = 0;
    long long launches = 0;
    double flops = 0.0;
  };
  // by (z, B, n_img, n_new): a graph bakes in the z buffer and the shape
  std::map<std::tuple<const void*, int, int, int>, Graph> graphs;
  cudaStream_t gstream = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
};

namespace {

template <class F>
lazymar_status hlaunch(lazymar_head* h, double flops, const char* what, F&& f) {
  NvtxRange range(what);
  cudaError_t e = f();
  if (e != cudaSuccess) return head_cuda(e, what);
  h->launches += 1;
  h->flops += flops;
  return LAZYMAR_OK;
}

lazymar_status hgemm(lazymar_head* h, const Ctx& c, const void* A, const void* W, int M, int N, int K,
                     const GemmEpi& e) {
  if (M == 0) return LAZYMAR_OK;
  return hlaunch(h, 2.0 * M * N * K, "head gemm", [&] { return launch_gemm(c, LAZYMAR_BF16, A, W, M, N, K, e, 0); });
}

template <int VPL>
cudaError_t launch_ln_mod_t(const Ctx& c, lazymar_head* h, const bf16* mod, bool inproj, int R, int M, int shift_off,
                            int scale_off) {
  const unsigned grid = (unsigned)((R + 7) / 8);
  if (inproj)
    return launch_pdl(hd::ln_mod_kernel<VPL, true>, dim3(grid), dim3(256), 0, c.stream, h->xh, (const float*)h->x,
                      (const bf16*)h->in_wt, (const bf16*)h->in_b, mod, h->nmod, shift_off, scale_off, h->hb, R, M,
                      h->td, h->cfg.ln_eps);
  return launch_pdl(hd::ln_mod_kernel<VPL, false>, dim3(grid), dim3(256), 0, c.stream, h->xh, (const float*)h->x,
                    (const bf16*)h->in_wt, (const bf16*)h->in_b, mod, h->nmod, shift_off, scale_off, h->hb, R, M,
                    h->td, h->cfg.ln_eps);
}

cudaError_t launch_ln_mod(const Ctx& c, lazymar_head* h, const bf16* mod, bool inproj, int R, int M, int shift_off,
                          int scale_off) {
  switch (h->w / 128) {
    case 1: return launch_ln_mod_t<1>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 2: return launch_ln_mod_t<2>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 3: return launch_ln_mod_t<3>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 4: return launch_ln_mod_t<4>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 5: return launch_ln_mod_t<5>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 6: return launch_ln_mod_t<6>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 7: return launch_ln_mod_t<7>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 8: return launch_ln_mod_t<8>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 9: return launch_ln_mod_t<9>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 10: return launch_ln_mod_t<10>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 11: return launch_ln_mod_t<11>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 12: return launch_ln_mod_t<12>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 13: return launch_ln_mod_t<13>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 14: return launch_ln_mod_t<14>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 15: return launch_ln_mod_t<15>(c, h, mod, inproj, R, M, shift_off, scale_off);
    case 16: return launch_ln_mod_t<16>(c, h, mod, inproj, R, M, shift_off, scale_off);
    default: return cudaErrorInvalidValue;
  }
}

template <int VPL>
cudaError_t launch_final_t(const Ctx& c, lazymar_head* h, size_t smem, const bf16* mod, int fshift, int fscale, int M,
                           const hd::StepConst& sc, const float* noise, float* x_done, float* eval_out,
                           const bf16* next_mod) {
  return launch_pdl(hd::final_kernel<VPL>, dim3(M), dim3(hd::FIN_THREADS), smem, c.stream, (const float*)h->xh, mod,
                    h->nmod, fshift, fscale, (const bf16*)h->out_w, (const float*)h->out_b, M, h->w, h->td,
                    h->cfg.ln_eps, sc, (const float*)h->params, h->x, noise, x_done, eval_out, next_mod,
                    (const bf16*)h->in_wt, (const bf16*)h->in_b, h->xh, h->hb);
}

cudaError_t launch_final(const Ctx& c, lazymar_head* h, size_t smem, const bf16* mod, int fshift, int fscale, int M,
                         const hd::StepConst& sc, const float* noise, float* x_done, float* eval_out,
                         const bf16* next_mod) {
  switch (h->w / 128) {
#define LM_FIN(V) \
  case V: return launch_final_t<V>(c, h, smem, mod, fshift, fscale, M, sc, noise, x_done, eval_out, next_mod);
    LM_FIN(1) LM_FIN(2) LM_FIN(3) LM_FIN(4) LM_FIN(5) LM_FIN(6) LM_FIN(7) LM_FIN(8)
    LM_FIN(9) LM_FIN(10) LM_FIN(11) LM_FIN(12) LM_FIN(13) LM_FIN(14) LM_FIN(15) LM_FIN(16)
#undef LM_FIN
    default: return cudaErrorInvalidValue;
  }
}

// Gathers the z rows and embeds them (W_c z + b_c), once per call.
lazymar_status prologue(lazymar_head* h, const Ctx& c, const void* z, int B, int n_img, int n_new, int M) {
  const int R = 2 * M, cd = h->cfg.cond_dim;
  HD_TRY(hlaunch(h, 0.0, "head gather", [&] {
    const unsigned grid = (unsigned)((R + 7) / 8);
    if (h->cfg.z_dtype == LAZYMAR_BF16)
      return launch_pdl(hd::gather_z_kernel<bf16>, dim3(grid), dim3(256), 0, c.stream, (const bf16*)z,
                        (const int*)h->pos, B, n_img, cd, M, n_new, h->zg, h->err);
    return launch_pdl(hd::gather_z_kernel<float>, dim3(grid), dim3(256), 0, c.stream, (const float*)z,
                      (const int*)h->pos, B, n_img, cd, M, n_new, h->zg, h->err);
  }));
  return hgemm(h, c, h->zg, h->c_w, R, h->w, cd,
               GemmEpi{LAZYMAR_EPI_BIAS, h->c_b, h->cemb, h->w, nullptr, nullptr, nullptr, 0});
}

// The modulations (all blocks' shift, scale, gate and the final shift,
// scale) of cnt kept steps j0, j0 - 1, .. for the R rows, in one GEMM:
// step j0 - k's rows start at h->mod + k R nmod. They depend on t_emb and
// c_emb only, not on x.
lazymar_status modulations(lazymar_head* h, const Ctx& c, int M, int j0, int cnt) {
  const int R = 2 * M, w = h->w;
  HD_TRY(hlaunch(h, 0.0, "head condition", [&] {
    const long long n = (long long)cnt * R * (w / 8);
    long long blocks = (n + 255) / 256;
    if (blocks > 8LL * h->num_sms) blocks = 8LL * h->num_sms;
    return launch_pdl(hd::cond_silu_kernel, dim3((unsigned)blocks), dim3(256), 0, c.stream, (const bf16*)h->temb, j0,
                      cnt, (const bf16*)h->cemb, h->sy, R, w);
  }));
  return hgemm(h, c, h->sy, h->ada_w, cnt * R, h->nmod, w,
               GemmEpi{LAZYMAR_EPI_BIAS, h->ada_b, h->mod, h->nmod, nullptr, nullptr, nullptr, 0});
}

// One network evaluation at kept step j on rows [x; x] with its modulations
// `mod` (R rows of nmod); ends with the final kernel (sampler update, or raw
// outputs to eval_out).
// With first_done the block-0 rows were already computed by the previous
// step's final kernel; with next_mod this step's final kernel computes them
// for the next kept step (whose modulations are next_mod).
lazymar_status network(lazymar_head* h, const Ctx& c, int M, int j, const bf16* mod, bool done, float* eval_out,
                       bool first_done = false, const bf16* next_mod = nullptr) {
  const int R = 2 * M, w = h->w, depth = h->cfg.depth, td = h->td;
  for (int b = 0; b < depth; ++b) {
    if (b > 0 || !first_done)
      HD_TRY(hlaunch(h, b == 0 ? 2.0 * R * td * w : 0.0, "head layernorm", [&] {
        return launch_ln_mod(c, h, mod, b == 0, R, M, 3 * w * b, 3 * w * b + w);
      }));
    HD_TRY(hgemm(h, c, h->hb, h->w1[b], R, w, w,
                 GemmEpi{LAZYMAR_EPI_SILU, h->b1[b], h->u, w, nullptr, nullptr, nullptr, 0}));
    GemmEpi e2{LAZYMAR_EPI_RESIDUAL, h->b2[b], h->xh, w, nullptr, nullptr, nullptr, 0};
    e2.gate = mod + 3 * w * b + 2 * w;
    e2.ldg = h->nmod;
    HD_TRY(hgemm(h, c, h->u, h->w2[b], R, w, w, e2));
  }
  const hd::StepConst sc = h->sched[j];
  const int fshift = 3 * w * depth, fscale = fshift + w;
  const size_t smem = (size_t)(2 * w + 4 * td + 2 * (hd::FIN_THREADS / 32) + td) * sizeof(float);
  const double flops = 2.0 * R * 2 * td * w + (next_mod ? 2.0 * R * td * w : 0.0);
  return hlaunch(h, flops, "head final", [&] {
    return launch_final(c, h, smem, mod, fshift, fscale, M, sc,
                        (const float*)(h->noise + (size_t)(h->cfg.n_steps - 1 - j + (sc.last ? 0 : 1)) * M * td),
                        done ? h->x_done : nullptr, eval_out, next_mod);
  });
}

// The whole sampling loop: x from noise[0], kept steps n_steps-1 .. 0.
lazymar_status sample_body(lazymar_head* h, const Ctx& c, const void* z, int B, int n_img, int n_new) {
  const int M = B * n_new, td = h->td;
  HD_TRY(prologue(h, c, z, B, n_img, n_new, M));
  HD_CUDA(cudaMemcpyAsync(h->x, h->noise, (size_t)M * td * sizeof(float), cudaMemcpyDeviceToDevice, c.stream));
  for (int j0 = h->cfg.n_steps - 1; j0 >= 0; j0 -= h->chunk) {
    const int cnt = j0 + 1 < h->chunk ? j0 + 1 : h->chunk;
    HD_TRY(modulations(h, c, M, j0, cnt));
    // inside a chunk each final kernel also computes the next step's block-0
    // rows, whose modulations are already there
    for (int k = 0; k < cnt; ++k)
      HD_TRY(network(h, c, M, j0 - k, h->mod + (size_t)k * 2 * M * h->nmod, j0 - k == 0, nullptr, k > 0,
                     k + 1 < cnt ? h->mod + (size_t)(k + 1) * 2 * M * h->nmod : nullptr));
  }
  return LAZYMAR_OK;
}

lazymar_status check_call(lazymar_head* h, const void* z, int B, int n_img, const int32_t* pos, int n_new) {
  if (!h || !z || !pos) return head_fail(LAZYMAR_ERR_INVALID_ARG, "NULL argument");
  if (B < 1 || n_img < 1 || n_new < 1 || (long long)B * n_new > h->cfg.max_tokens)
    return head_fail(LAZYMAR_ERR_INVALID_ARG, "need B >= 1, n_img >= 1, 1 <= B * n_new <= max_tokens");
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, z) != cudaSuccess ||
      (a.type != cudaMemoryTypeDevice && a.type != cudaMemoryTypeManaged)) {
    cudaGetLastError();
    return head_fail(LAZYMAR_ERR_INVALID_ARG, "z must be a device pointer");
  }
  return LAZYMAR_OK;
}

struct HeadGuard {
  int prev = -1;
  explicit HeadGuard(int dev) {
    int cur = 0;
    if (cudaGetDevice(&cur) == cudaSuccess && cur != dev) {
      prev = cur;
      cudaSetDevice(dev);
    }
  }
  ~HeadGuard() {
    if (prev >= 0) cudaSetDevice(prev);
  }
};

lazymar_status upload_bf16(bf16* dst, const float* src, size_t n, bool transpose = false, size_t rows = 0,
                           size_t cols = 0) {
  if (!src) return head_fail(LAZYMAR_ERR_INVALID_ARG, "a head weight pointer is NULL");
  std::vector<float> t(n);
  HD_CUDA(cudaMemcpy(t.data(), src, n * sizeof(float), cudaMemcpyDefault));
  std::vector<uint16_t> b(n);
  if (transpose) {
    for (size_t r = 0; r < rows; ++r)
      for (size_t k = 0; k < cols; ++k) b[k * rows + r] = to_bf16_bits(t[r * cols + k]);
  } else {
    for (size_t i = 0; i < n; ++i) b[i] = to_bf16_bits(t[i]);
  }
  HD_CUDA(cudaMemcpy(dst, b.data(), n * 2, cudaMemcpyHostToDevice));
  return LAZYMAR_OK;
}

lazymar_status upload_f32(float* dst, const float* src, size_t n, bool round_bf16) {
  if (!src) return head_fail(LAZYMAR_ERR_INVALID_ARG, "a head weight pointer is NULL");
  std::vector<float> t(n);
  HD_CUDA(cudaMemcpy(t.data(), src, n * sizeof(float), cudaMemcpyDefault));
  if (round_bf16)
    for (auto& v : t) {
      const uint32_t u = (uint32_t)to_bf16_bits(v) << 16;
      std::memcpy(&v, &u, 4);
    }
  HD_CUDA(cudaMemcpy(dst, t.data(), n * sizeof(float), cudaMemcpyHostToDevice));
  return LAZYMAR_OK;
}

// Cosine schedule (alpha_bar(t) = f(t) / f(0), f(t) = cos^2(((t / T) + s) /
// (1 + s) pi / 2), s = 0.008, betas clipped at 0.999), kept steps
// round-half-even(i (T - 1) / (n - 1)), respaced betas from the kept
// cumulative products; per kept step the constants of the sampler update
// (mean = x / sqrt(1 - beta) - beta / (sqrt(1 - beta) sqrt(1 - alpha_bar)) eps).
void make_schedule(int n_train, int n_steps, std::vector<int>& kept, std::vector<hd::StepConst>& sc) {
  const double s = 0.008, pi = 3.14159265358979323846;
  auto f = [&](double t) {
    const double c = std::cos((t / n_train + s) / (1.0 + s) * pi / 2.0);
    return c * c;
  };
  std::vector<double> ab(n_train);
  double prod = 1.0;
  for (int i = 0; i < n_train; ++i) {
    double beta = 1.0 - f(i + 1) / f(i);
    if (beta > 0.999) beta = 0.999;
    prod *= 1.0 - beta;
    ab[i] = prod;
  }
  kept.resize(n_steps);
  for (int i = 0; i < n_steps; ++i)
    kept[i] = n_steps == 1 ? 0 : (int)std::nearbyint((double)i * (n_train - 1) / (double)(n_steps - 1));
  std::vector<double> beta(n_steps), abk(n_steps), post(n_steps);
  double last = 1.0;
  for (int j = 0; j < n_steps; ++j) {
    abk[j] = ab[kept[j]];
    beta[j] = 1.0 - abk[j] / last;
    post[j] = beta[j] * (1.0 - last) / (1.0 - abk[j]);
    last = abk[j];
  }
  sc.resize(n_steps);
  for (int j = 0; j < n_steps; ++j) {
    const double sa = std::sqrt(1.0 - beta[j]);
    sc[j].a_x = (float)(1.0 / sa);
    sc[j].a_eps = (float)(beta[j] / (sa * std::sqrt(1.0 - abk[j])));
    sc[j].log_beta = (float)std::log(beta[j]);
    sc[j].log_post = (float)std::log(n_steps > 1 && j == 0 ? post[1] : post[j]);
    sc[j].last = j == 0;
  }
}

}  // namespace

extern "C" lazymar_status lazymar_head_create(const lazymar_head_config* cfg, const lazymar_head_weights* w,
                                              lazymar_head** out) {
  if (!cfg || !w || !out || !w->blocks) return head_fail(LAZYMAR_ERR_INVALID_ARG, "NULL argument");
  *out = nullptr;
  const lazymar_head_config& c = *cfg;
  if (c.token_dim < 1 || c.token_dim > 64 || c.depth < 1 || c.max_tokens < 1 || c.n_train < 1 || c.n_steps < 1 ||
      c.n_steps > c.n_train || !(c.ln_eps > 0.f))
    return head_fail(LAZYMAR_ERR_INVALID_ARG, "head config: sizes out of range");
  if (c.z_dtype != LAZYMAR_BF16 && c.z_dtype != LAZYMAR_F32) return head_fail(LAZYMAR_ERR_INVALID_ARG, "head config: z_dtype");
  if (!width_ok(c.width) || c.cond_dim < 64 || c.cond_dim % 64 != 0 || c.freq_dim < 128 || c.freq_dim % 128 != 0)
    return head_fail(LAZYMAR_ERR_UNSUPPORTED,
                     "head config: width = 128 k (k <= 16), cond_dim % 64 == 0, freq_dim % 128 == 0 required");
  if ((long long)2 * c.max_tokens * (3LL * c.width * c.depth + 2 * c.width) >= (1ll << 31))
    return head_fail(LAZYMAR_ERR_UNSUPPORTED, "head config: max_tokens too large");
  auto* h = new lazymar_head();
  h->cfg = c;
  h->w = c.width;
  h->td = c.token_dim;
  h->nmod = 3 * c.width * c.depth + 2 * c.width;
  auto destroy = [&](lazymar_status s) {
    lazymar_head_destroy(h);
    return s;
  };
  cudaError_t e = cudaGetDevice(&h->dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->dev);
  if (e != cudaSuccess) return destroy(head_cuda(e, "device query"));

  const size_t W = c.width, F = c.freq_dim, CD = c.cond_dim, TD = c.token_dim, NM = h->nmod, NS = c.n_steps;
  const size_t R = 2 * (size_t)c.max_tokens, MT = c.max_tokens;
  // modulations of up to `chunk` kept steps at once, within 1 GB and with
  // fewer than 2^31 rows x columns per GEMM
  {
    const double per_step = (double)R * NM;
    long long ch = (long long)(1e9 / (2.0 * per_step));
    const long long cap = (long long)((double)(1ll << 31) / per_step);
    if (ch > cap) ch = cap;
    if (ch > c.n_steps) ch = c.n_steps;
    h->chunk = ch < 1 ? 1 : (int)ch;
  }
  const size_t CH = (size_t)h->chunk;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += (bytes + 255) & ~size_t(255);
    return o;
  };
  const size_t o_tw1 = take(W * F * 2), o_tb1 = take(W * 2), o_tw2 = take(W * W * 2), o_tb2 = take(W * 2),
               o_cw = take(W * CD * 2), o_cb = take(W * 2), o_inw = take(W * TD * 2), o_inb = take(W * 2),
               o_adaw = take(NM * W * 2), o_adab = take(NM * 2), o_outw = take(2 * TD * W * 2), o_outb = take(2 * TD * 4);
  std::vector<size_t> o_w1(c.depth), o_b1(c.depth), o_w2(c.depth), o_b2(c.depth);
  for (int b = 0; b < c.depth; ++b) {
    o_w1[b] = take(W * W * 2); o_b1[b] = take(W * 2); o_w2[b] = take(W * W * 2); o_b2[b] = take(W * 2);
  }
  const size_t o_temb = take(NS * W * 2), o_sin = take(NS * F * 2), o_t1 = take(NS * W * 2), o_kept = take(NS * 4);
  const size_t o_pos = take(MT * 4), o_noise = take(NS * MT * TD * 4), o_x = take(MT * TD * 4), o_xd = take(MT * TD * 4),
               o_xh = take(R * W * 4), o_eval = take(R * 2 * TD * 4), o_par = take(2 * 4), o_zg = take(R * CD * 2),
               o_cemb = take(R * W * 2), o_sy = take(CH * R * W * 2), o_mod = take(CH * R * NM * 2), o_hb = take(R * W * 2),
               o_u = take(R * W * 2), o_err = take(4);
  e = cudaMalloc(&h->arena, off);
  if (e != cudaSuccess) {
    cudaGetLastError();
    h->arena = nullptr;
    return destroy(head_fail(LAZYMAR_ERR_OOM, "head: cudaMalloc failed"));
  }
  e = cudaMemset(h->arena, 0, off);
  if (e != cudaSuccess) return destroy(head_cuda(e, "cudaMemset"));
  uint8_t* a = h->arena;
  auto B16 = [&](size_t o) { return reinterpret_cast<bf16*>(a + o); };
  auto F32 = [&](size_t o) { return reinterpret_cast<float*>(a + o); };
  h->t_w1 = B16(o_tw1); h->t_b1 = B16(o_tb1); h->t_w2 = B16(o_tw2); h->t_b2 = B16(o_tb2);
  h->c_w = B16(o_cw); h->c_b = B16(o_cb); h->in_wt = B16(o_inw); h->in_b = B16(o_inb);
  h->ada_w = B16(o_adaw); h->ada_b = B16(o_adab); h->out_w = B16(o_outw); h->out_b = F32(o_outb);
  for (int b = 0; b < c.depth; ++b) {
    h->w1.push_back(B16(o_w1[b])); h->b1.push_back(B16(o_b1[b]));
    h->w2.push_back(B16(o_w2[b])); h->b2.push_back(B16(o_b2[b]));
  }
  h->temb = B16(o_temb);
  h->pos = reinterpret_cast<int*>(a + o_pos); h->noise = F32(o_noise); h->x = F32(o_x); h->x_done = F32(o_xd);
  h->xh = F32(o_xh); h->eval = F32(o_eval); h->params = F32(o_par);
  h->zg = B16(o_zg); h->cemb = B16(o_cemb); h->sy = B16(o_sy); h->mod = B16(o_mod); h->hb = B16(o_hb); h->u = B16(o_u);
  h->err = reinterpret_cast<unsigned*>(a + o_err);

  lazymar_status st;
  if ((st = upload_bf16(h->t_w1, w->t_w1, W * F)) || (st = upload_bf16(h->t_b1, w->t_b1, W)) ||
      (st = upload_bf16(h->t_w2, w->t_w2, W * W)) || (st = upload_bf16(h->t_b2, w->t_b2, W)) ||
      (st = upload_bf16(h->c_w, w->c_w, W * CD)) || (st = upload_bf16(h->c_b, w->c_b, W)) ||
      (st = upload_bf16(h->in_wt, w->in_w, W * TD, true, W, TD)) || (st = upload_bf16(h->in_b, w->in_b, W)) ||
      (st = upload_bf16(h->out_w, w->out_w, 2 * TD * W)) || (st = upload_f32(h->out_b, w->out_b, 2 * TD, true)))
    return destroy(st);
  for (int b = 0; b < c.depth; ++b) {
    const lazymar_head_block_weights& bw = w->blocks[b];
    if ((st = upload_bf16(h->ada_w + (size_t)3 * W * b * W, bw.ada_w, 3 * W * W)) ||
        (st = upload_bf16(h->ada_b + (size_t)3 * W * b, bw.ada_b, 3 * W)) ||
        (st = upload_bf16(h->w1[b], bw.w1, W * W)) || (st = upload_bf16(h->b1[b], bw.b1, W)) ||
        (st = upload_bf16(h->w2[b], bw.w2, W * W)) || (st = upload_bf16(h->b2[b], bw.b2, W)))
      return destroy(st);
  }
  if ((st = upload_bf16(h->ada_w + (size_t)3 * W * c.depth * W, w->f_ada_w, 2 * W * W)) ||
      (st = upload_bf16(h->ada_b + (size_t)3 * W * c.depth, w->f_ada_b, 2 * W)))
    return destroy(st);

  // schedule and the time embeddings of the kept steps
  std::vector<int> kept;
  make_schedule(c.n_train, c.n_steps, kept, h->sched);
  e = cudaMemcpy(a + o_kept, kept.data(), NS * 4, cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return destroy(head_cuda(e, "cudaMemcpy"));
  if ((e = cudaStreamCreateWithFlags(&h->gstream, cudaStreamNonBlocking)) != cudaSuccess ||
      (e = cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming)) != cudaSuccess ||
      (e = cudaEventCreateWithFlags(&h->ev_join, cudaEventDisableTiming)) != cudaSuccess)
    return destroy(head_cuda(e, "stream/event creation"));
  const Ctx cx{h->gstream, h->err, h->num_sms};
  hd::sinusoid_kernel<<<(unsigned)NS, 128, 0, h->gstream>>>(reinterpret_cast<const int*>(a + o_kept), B16(o_sin),
                                                            (int)NS, (int)F / 2);
  if ((e = cudaGetLastError()) != cudaSuccess) return destroy(head_cuda(e, "sinusoid kernel"));
  if ((st = hgemm(h, cx, B16(o_sin), h->t_w1, (int)NS, (int)W, (int)F,
                  GemmEpi{LAZYMAR_EPI_SILU, h->t_b1, B16(o_t1), (int)W, nullptr, nullptr, nullptr, 0})) ||
      (st = hgemm(h, cx, B16(o_t1), h->t_w2, (int)NS, (int)W, (int)W,
                  GemmEpi{LAZYMAR_EPI_BIAS, h->t_b2, h->temb, (int)W, nullptr, nullptr, nullptr, 0})))
    return destroy(st);
  if ((e = cudaStreamSynchronize(h->gstream)) != cudaSuccess) return destroy(head_cuda(e, "time embedding"));
  h->launches = 0;
  h->flops = 0.0;
  *out = h;
  return LAZYMAR_OK;
}

extern "C" void lazymar_head_destroy(lazymar_head* h) {
  if (!h) return;
  HeadGuard g(h->dev);
  for (auto& kv : h->graphs)
    if (kv.second.exec) cudaGraphExecDestroy(kv.second.exec);
  if (h->ev_fork) cudaEventDestroy(h->ev_fork);
  if (h->ev_join) cudaEventDestroy(h->ev_join);
  if (h->gstream) cudaStreamDestroy(h->gstream);
  if (h->arena) cudaFree(h->arena);
  delete h;
}

namespace {

lazymar_status stage(lazymar_head* h, cudaStream_t st, const int32_t* pos, int M, const float* noise, int n_noise,
                     float gamma, float temperature) {
  HD_CUDA(cudaMemcpyAsync(h->pos, pos, (size_t)M * 4, cudaMemcpyDefault, st));
  if (noise) HD_CUDA(cudaMemcpyAsync(h->noise, noise, (size_t)n_noise * M * h->td * 4, cudaMemcpyDefault, st));
  h->host_params[0] = gamma;
  h->host_params[1] = temperature;
  HD_CUDA(cudaMemcpyAsync(h->params, h->host_params, sizeof h->host_params, cudaMemcpyHostToDevice, st));
  return LAZYMAR_OK;
}

}  // namespace

extern "C" lazymar_status lazymar_head_sample(lazymar_head* h, const void* z, int B, int n_img, const int32_t* pos,
                                              int n_new, const float* noise, float gamma, float temperature,
                                              float* x_out, void* stream) {
  NvtxRange range("lazymar_head_sample");
  HD_TRY(check_call(h, z, B, n_img, pos, n_new));
  if (!noise || !x_out) return head_fail(LAZYMAR_ERR_INVALID_ARG, "NULL noise or x_out");
  HeadGuard g(h->dev);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int M = B * n_new;
  HD_TRY(stage(h, st, pos, M, noise, h->cfg.n_steps, gamma, temperature));
  // the loop runs on the head's stream: eagerly on the first use of a
  // (z, B, n_img, n_new) combination, captured into a CUDA graph on the
  // second and replayed from then on
  auto& ge = h->graphs[std::make_tuple(z, B, n_img, n_new)];
  HD_CUDA(cudaEventRecord(h->ev_fork, st));
  HD_CUDA(cudaStreamWaitEvent(h->gstream, h->ev_fork, 0));
  const Ctx cx{h->gstream, h->err, h->num_sms};
  if (!ge.exec && ge.eager_runs++ == 0) {
    HD_TRY(sample_body(h, cx, z, B, n_img, n_new));
  } else {
    if (!ge.exec) {
      const long long l0 = h->launches;
      const double f0 = h->flops;
      HD_CUDA(cudaStreamBeginCapture(h->gstream, cudaStreamCaptureModeThreadLocal));
      const lazymar_status s = sample_body(h, cx, z, B, n_img, n_new);
      cudaGraph_t gr = nullptr;
      const cudaError_t ec = cudaStreamEndCapture(h->gstream, &gr);
      if (s != LAZYMAR_OK || ec != cudaSuccess) {
        if (gr) cudaGraphDestroy(gr);
        h->launches = l0;
        h->flops = f0;
        return s != LAZYMAR_OK ? s : head_cuda(ec, "cudaStreamEndCapture");
      }
      const cudaError_t ei = cudaGraphInstantiate(&ge.exec, gr, 0);
      cudaGraphDestroy(gr);
      if (ei != cudaSuccess) {
        ge.exec = nullptr;
        h->launches = l0;
        h->flops = f0;
        return head_cuda(ei, "cudaGraphInstantiate");
      }
      ge.launches = h->launches - l0;
      ge.flops = h->flops - f0;
      h->launches = l0;
      h->flops = f0;
    }
    HD_CUDA(cudaGraphLaunch(ge.exec, h->gstream));
    h->launches += ge.launches;
    h->flops += ge.flops;
  }
  HD_CUDA(cudaEventRecord(h->ev_join, h->gstream));
  HD_CUDA(cudaStreamWaitEvent(st, h->ev_join, 0));
  HD_CUDA(cudaMemcpyAsync(x_out, h->x_done, (size_t)M * h->td * 4, cudaMemcpyDefault, st));
  return LAZYMAR_OK;
}

extern "C" lazymar_status lazymar_head_eval(lazymar_head* h, const void* z, int B, int n_img, const int32_t* pos,
                                            int n_new, const float* x, int j, float* out, void* stream) {
  HD_TRY(check_call(h, z, B, n_img, pos, n_new));
  if (!x || !out) return head_fail(LAZYMAR_ERR_INVALID_ARG, "NULL x or out");
  if (j < 0 || j >= h->cfg.n_steps) return head_fail(LAZYMAR_ERR_INVALID_ARG, "j outside 0..n_steps-1");
  HeadGuard g(h->dev);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int M = B * n_new;
  HD_TRY(stage(h, st, pos, M, nullptr, 0, 1.f, 1.f));
  HD_CUDA(cudaMemcpyAsync(h->x, x, (size_t)M * h->td * 4, cudaMemcpyDefault, st));
  const Ctx c{st, h->err, h->num_sms};
  HD_TRY(prologue(h, c, z, B, n_img, n_new, M));
  HD_TRY(modulations(h, c, M, j, 1));
  HD_TRY(network(h, c, M, j, h->mod, false, h->eval));
  HD_CUDA(cudaMemcpyAsync(out, h->eval, (size_t)2 * M * 2 * h->td * 4, cudaMemcpyDefault, st));
  return LAZYMAR_OK;
}

extern "C" lazymar_status lazymar_head_schedule(int n_train, int n_steps, int32_t* kept, float* consts) {
  if (n_train < 1 || n_steps < 1 || n_steps > n_train)
    return head_fail(LAZYMAR_ERR_INVALID_ARG, "need 1 <= n_steps <= n_train");
  std::vector<int> k;
  std::vector<hd::StepConst> sc;
  make_schedule(n_train, n_steps, k, sc);
  for (int j = 0; j < n_steps; ++j) {
    if (kept) kept[j] = k[j];
    if (consts) {
      consts[4 * j] = sc[j].a_x;
      consts[4 * j + 1] = sc[j].a_eps;
      consts[4 * j + 2] = sc[j].log_beta;
      consts[4 * j + 3] = sc[j].log_post;
    }
  }
  return LAZYMAR_OK;
}

extern "C" lazymar_status lazymar_head_counters(lazymar_head* h, long long* launches, double* flops) {
  if (!h) return head_fail(LAZYMAR_ERR_INVALID_ARG, "NULL head");
  if (launches) *launches = h->launches;
  if (flops) *flops = h->flops;
  return LAZYMAR_OK;
}

extern "C" lazymar_status lazymar_head_sync(lazymar_head* h, void* stream) {
  if (!h) return head_fail(LAZYMAR_ERR_INVALID_ARG, "NULL head");
  HeadGuard g(h->dev);
  HD_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
  HD_CUDA(cudaStreamSynchronize(h->gstream));
  unsigned v = 0;
  HD_CUDA(cudaMemcpy(&v, h->err, sizeof v, cudaMemcpyDeviceToHost));
  if (v) HD_CUDA(cudaMemset(h->err, 0, sizeof v));
  if (v & ERR_TIMEOUT) return head_fail(LAZYMAR_ERR_TIMEOUT, "a bounded device wait expired");
  if (v & ERR_INDEX) return head_fail(LAZYMAR_ERR_DEVICE, "a decoded position was out of range");
  return LAZYMAR_OK;
}
