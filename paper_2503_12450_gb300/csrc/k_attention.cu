// Bidirectional multi-head attention of Eq. 3 with a query subset: the queries
// of the recomputed tokens (I_compute) attend over all T keys of their
// sequence, fresh ones for I_compute and cached ones for I_cache (Eq. 9). The
// full-layer form is the same kernel with every token as a query.
//
// bf16: one CTA per (64-query tile, head, row); 4 warps x 16 queries. Q and
// K/V tiles of 64 keys are staged in shared memory by TMA (128B swizzle for
// the first 64 columns of a head, 32B swizzle for the 16-column remainder of
// an 80-wide head), double-buffered on mbarriers. S = Q K^T and O += P V run on
// mma.sync m16n8k16 (bf16 in, fp32 accumulate) with an online softmax in
// registers (exp2 with the 1/sqrt(d) scale folded into log2 e).
//
// f32: one warp per query on CUDA cores (fp32 configuration).
#include <cuda.h>

#include <cfloat>

#include "lazymar_internal.cuh"

namespace lm {

bool make_tmap_bf16(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t pitch_bytes,
                    uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swz);

namespace at {
constexpr int QT = 64;   // queries per CTA
constexpr int KT = 64;   // keys per stage
constexpr int TILE64 = 64 * 128;  // 64 rows x 64 bf16, 128B swizzle
constexpr int TILE16 = 64 * 32;   // 64 rows x 16 bf16, 32B swizzle

// Byte offset of 16-byte chunk `c` (8 head dims) of row `r` inside a tile pair
// (64-column part at `base64`, 16-column remainder at `base16`), following the
// TMA swizzle patterns: 128B swizzle XORs chunk bits [0,3) with row bits [0,3);
// 32B swizzle XORs chunk bit 0 with bit 2 of the row (bit 7 of the address).
__device__ __forceinline__ uint32_t chunk_addr(uint32_t base64, uint32_t base16, int r, int c) {
  return c < 8 ? base64 + (uint32_t)(r * 128) + (uint32_t)(((c ^ (r & 7)) & 7) << 4)
               : base16 + (uint32_t)(r * 32) + (uint32_t)((((c - 8) ^ (r >> 2)) & 1) << 4);
}
}  // namespace at

template <int DH>
__global__ void __launch_bounds__(128) attention_bf16_kernel(const __grid_constant__ CUtensorMap tmQ,
                                                             const __grid_constant__ CUtensorMap tmQ2,
                                                             const __grid_constant__ CUtensorMap tmK,
                                                             const __grid_constant__ CUtensorMap tmK2,
                                                             const __grid_constant__ CUtensorMap tmV,
                                                             const __grid_constant__ CUtensorMap tmV2, bf16* o,
                                                             int n_q, int T, int D, float scale_log2,
                                                             unsigned* err) {
  static_assert(DH == 64 || DH == 80, "head width 64 or 80");
  constexpr bool kTail = DH == 80;
  constexpr int KSTEPS = DH / 16;   // k-steps of Q K^T
  constexpr int NB = DH / 8;        // 8-wide output column blocks
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  // [Q64][K64 x2][V64 x2][Q16][K16 x2][V16 x2][barriers]
  uint8_t* sQ = smem;
  uint8_t* sK = sQ + at::TILE64;
  uint8_t* sV = sK + 2 * at::TILE64;
  uint8_t* sQ2 = sV + 2 * at::TILE64;
  uint8_t* sK2 = sQ2 + at::TILE16;
  uint8_t* sV2 = sK2 + 2 * at::TILE16;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV2 + 2 * at::TILE16);  // [0] Q, [1..2] K/V stages
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 3);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int qt = blockIdx.x, h = blockIdx.y, r = blockIdx.z;
  const int q0 = r * n_q + qt * at::QT;  // first query row (global)
  const int kv0 = r * T;                 // first key row (global)
  const int col = h * DH;
  const int nkt = (T + at::KT - 1) / at::KT;
  constexpr uint32_t kv_bytes = 2u * (at::TILE64 + (kTail ? at::TILE16 : 0));
  constexpr uint32_t q_bytes = at::TILE64 + (kTail ? at::TILE16 : 0);

  if (tid == 0) {
    for (int i = 0; i < 3; ++i) mbar_init(&bars[i], 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  pdl_wait();
  pdl_trigger();
  if (tid == 0) {
    mbar_arrive_expect_tx(&bars[0], q_bytes);
    tma_load_2d(&tmQ, &bars[0], sQ, col, q0);
    if (kTail) tma_load_2d(&tmQ2, &bars[0], sQ2, col + 64, q0);
    for (int j = 0; j < 2 && j < nkt; ++j) {
      mbar_arrive_expect_tx(&bars[1 + j], kv_bytes);
      tma_load_2d(&tmK, &bars[1 + j], sK + j * at::TILE64, col, kv0 + j * at::KT);
      tma_load_2d(&tmV, &bars[1 + j], sV + j * at::TILE64, col, kv0 + j * at::KT);
      if (kTail) {
        tma_load_2d(&tmK2, &bars[1 + j], sK2 + j * at::TILE16, col + 64, kv0 + j * at::KT);
        tma_load_2d(&tmV2, &bars[1 + j], sV2 + j * at::TILE16, col + 64, kv0 + j * at::KT);
      }
    }
  }

  // Q fragments of this warp's 16 queries (A operand, row-major 16 x 16 per k-step).
  bool ok = mbar_wait(&bars[0], 0, abort_flag, err);
  if (__syncthreads_or(!ok)) return;
  uint32_t qf[KSTEPS][4];
  {
    const uint32_t b64 = smem_u32(sQ), b16 = smem_u32(sQ2);
    const int row = warp * 16 + (lane & 15);
#pragma unroll
    for (int kk = 0; kk < KSTEPS; ++kk)
      ldsm_x4(at::chunk_addr(b64, b16, row, 2 * kk + (lane >> 4)), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
  }

  float oacc[NB][4];
#pragma unroll
  for (int i = 0; i < NB; ++i) oacc[i][0] = oacc[i][1] = oacc[i][2] = oacc[i][3] = 0.f;
  float m_run[2] = {-FLT_MAX, -FLT_MAX}, l_run[2] = {0.f, 0.f};
  const int g = lane >> 2, t4 = lane & 3;

  for (int j = 0; j < nkt; ++j) {
    const int st = j & 1;
    ok = mbar_wait(&bars[1 + st], (uint32_t)(j >> 1) & 1u, abort_flag, err);
    if (__syncthreads_or(!ok)) return;
    const uint32_t k64 = smem_u32(sK + st * at::TILE64), k16 = smem_u32(sK2 + st * at::TILE16);
    const uint32_t v64 = smem_u32(sV + st * at::TILE64), v16 = smem_u32(sV2 + st * at::TILE16);

    // S = Q K^T for 16 queries x 64 keys: 8 key blocks of 8.
    float s[8][4];
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) s[nb][0] = s[nb][1] = s[nb][2] = s[nb][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < KSTEPS; ++kk) {
#pragma unroll
      for (int nb = 0; nb < 8; nb += 2) {
        const int key = nb * 8 + ((lane >> 4) << 3) + (lane & 7);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(at::chunk_addr(k64, k16, key, 2 * kk + ((lane >> 3) & 1)), b0, b1, b2, b3);
        mma_bf16_16816(s[nb], qf[kk], b0, b1);
        mma_bf16_16816(s[nb + 1], qf[kk], b2, b3);
      }
    }
    // Scale, mask keys beyond T, online softmax (rows g and g + 8 of the warp).
    float mx[2] = {m_run[0], m_run[1]};
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = j * at::KT + nb * 8 + 2 * t4 + (e & 1);
        s[nb][e] = key < T ? s[nb][e] * scale_log2 : -FLT_MAX;
      }
      mx[0] = fmaxf(mx[0], fmaxf(s[nb][0], s[nb][1]));
      mx[1] = fmaxf(mx[1], fmaxf(s[nb][2], s[nb][3]));
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      mx[i] = fmaxf(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 1));
      mx[i] = fmaxf(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 2));
    }
    float corr[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      corr[i] = exp2f(m_run[i] - mx[i]);
      m_run[i] = mx[i];
      l_run[i] *= corr[i];
    }
#pragma unroll
    for (int i = 0; i < NB; ++i) {
      oacc[i][0] *= corr[0]; oacc[i][1] *= corr[0];
      oacc[i][2] *= corr[1]; oacc[i][3] *= corr[1];
    }
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) {
      s[nb][0] = exp2f(s[nb][0] - mx[0]);
      s[nb][1] = exp2f(s[nb][1] - mx[0]);
      s[nb][2] = exp2f(s[nb][2] - mx[1]);
      s[nb][3] = exp2f(s[nb][3] - mx[1]);
      l_run[0] += s[nb][0] + s[nb][1];
      l_run[1] += s[nb][2] + s[nb][3];
    }
    // O += P V: 4 k-steps of 16 keys; P re-used from the S accumulators.
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * ks][0], s[2 * ks][1]);
      pa[1] = pack_bf16(s[2 * ks][2], s[2 * ks][3]);
      pa[2] = pack_bf16(s[2 * ks + 1][0], s[2 * ks + 1][1]);
      pa[3] = pack_bf16(s[2 * ks + 1][2], s[2 * ks + 1][3]);
      const int key = ks * 16 + (lane & 15);
#pragma unroll
      for (int nb = 0; nb < NB; nb += 2) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(at::chunk_addr(v64, v16, key, nb + (lane >> 4)), b0, b1, b2, b3);
        mma_bf16_16816(oacc[nb], pa, b0, b1);
        mma_bf16_16816(oacc[nb + 1], pa, b2, b3);
      }
    }
    // Every warp has consumed its ldmatrix reads of this stage (the mma that
    // uses them precedes the barrier); the proxy fence then orders those
    // generic-proxy reads before the async-proxy TMA that refills the stage.
    __syncthreads();
    if (tid == 0 && j + 2 < nkt) {
      fence_proxy_async_smem();
      const int jn = j + 2;
      mbar_arrive_expect_tx(&bars[1 + st], kv_bytes);
      tma_load_2d(&tmK, &bars[1 + st], sK + st * at::TILE64, col, kv0 + jn * at::KT);
      tma_load_2d(&tmV, &bars[1 + st], sV + st * at::TILE64, col, kv0 + jn * at::KT);
      if (kTail) {
        tma_load_2d(&tmK2, &bars[1 + st], sK2 + st * at::TILE16, col + 64, kv0 + jn * at::KT);
        tma_load_2d(&tmV2, &bars[1 + st], sV2 + st * at::TILE16, col + 64, kv0 + jn * at::KT);
      }
    }
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    l_run[i] += __shfl_xor_sync(0xffffffffu, l_run[i], 1);
    l_run[i] += __shfl_xor_sync(0xffffffffu, l_run[i], 2);
    l_run[i] = 1.f / l_run[i];
  }
  const int qa = qt * at::QT + warp * 16 + g;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    const int qi = qa + half * 8;
    if (qi >= n_q) continue;
    bf16* dst = o + (size_t)(r * n_q + qi) * D + col + 2 * t4;
#pragma unroll
    for (int nb = 0; nb < NB; ++nb) {
      __nv_bfloat162 v = __floats2bfloat162_rn(oacc[nb][2 * half] * l_run[half], oacc[nb][2 * half + 1] * l_run[half]);
      *reinterpret_cast<__nv_bfloat162*>(dst + nb * 8) = v;
    }
  }
}

// fp32: one warp per query; scores for all T keys staged in shared memory.
__global__ void __launch_bounds__(128) attention_f32_kernel(const float* __restrict__ q, const float* __restrict__ k,
                                                            const float* __restrict__ v, float* __restrict__ o,
                                                            int n_q, int T, int D, int dh, float scale) {
  extern __shared__ float sm[];
  pdl_wait();
  pdl_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* sc = sm + warp * (T + dh);
  float* qv = sc + T;
  const int qi = blockIdx.x * 4 + warp, h = blockIdx.y, r = blockIdx.z;
  if (qi >= n_q) return;
  const float* qrow = q + (size_t)(r * n_q + qi) * D + h * dh;
  for (int d = lane; d < dh; d += 32) qv[d] = qrow[d];
  __syncwarp();
  float mx = -FLT_MAX;
  for (int t = lane; t < T; t += 32) {
    const float* kr = k + (size_t)(r * T + t) * D + h * dh;
    float acc = 0.f;
    for (int d = 0; d < dh; ++d) acc = fmaf(qv[d], kr[d], acc);
    acc *= scale;
    sc[t] = acc;
    mx = fmaxf(mx, acc);
  }
  mx = warp_max(mx);
  float sum = 0.f;
  for (int t = lane; t < T; t += 32) {
    const float p = expf(sc[t] - mx);
    sc[t] = p;
    sum += p;
  }
  sum = warp_sum(sum);
  __syncwarp();
  const float inv = 1.f / sum;
  for (int d = lane; d < dh; d += 32) {
    float acc = 0.f;
    for (int t = 0; t < T; ++t) acc = fmaf(sc[t], v[(size_t)(r * T + t) * D + h * dh + d], acc);
    o[(size_t)(r * n_q + qi) * D + h * dh + d] = acc * inv;
  }
}

bool attention_supported(int dtype, int heads, int dh, const char** why) {
  if (heads <= 0 || dh <= 0) { *why = "heads and head_dim must be positive"; return false; }
  if (dtype == LAZYMAR_BF16) {
    if (dh != 64 && dh != 80) { *why = "bf16 attention supports head_dim 64 or 80"; return false; }
  } else if (dtype == LAZYMAR_F32) {
    if (dh > 128) { *why = "f32 attention supports head_dim <= 128"; return false; }
  } else {
    *why = "unknown dtype";
    return false;
  }
  return true;
}

template <int DH>
static cudaError_t launch_attn_bf16(const Ctx& c, const void* q, const void* k, const void* v, void* o, int rows,
                                    int n_q, int T, int heads) {
  const int D = heads * DH;
  CUtensorMap mq, mq2, mk, mk2, mv, mv2;
  const uint64_t pitch = (uint64_t)D * 2;
  bool ok = make_tmap_bf16(&mq, q, D, (uint64_t)rows * n_q, pitch, 64, at::QT, CU_TENSOR_MAP_SWIZZLE_128B) &&
            make_tmap_bf16(&mk, k, D, (uint64_t)rows * T, pitch, 64, at::KT, CU_TENSOR_MAP_SWIZZLE_128B) &&
            make_tmap_bf16(&mv, v, D, (uint64_t)rows * T, pitch, 64, at::KT, CU_TENSOR_MAP_SWIZZLE_128B);
  if (DH == 80) {
    ok = ok && make_tmap_bf16(&mq2, q, D, (uint64_t)rows * n_q, pitch, 16, at::QT, CU_TENSOR_MAP_SWIZZLE_32B) &&
         make_tmap_bf16(&mk2, k, D, (uint64_t)rows * T, pitch, 16, at::KT, CU_TENSOR_MAP_SWIZZLE_32B) &&
         make_tmap_bf16(&mv2, v, D, (uint64_t)rows * T, pitch, 16, at::KT, CU_TENSOR_MAP_SWIZZLE_32B);
  } else {
    mq2 = mq; mk2 = mk; mv2 = mv;
  }
  if (!ok) return cudaErrorInvalidValue;
  constexpr size_t smem = 1024 + 5 * at::TILE64 + 5 * at::TILE16 + 64;
  static int attr_set[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(attention_bf16_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    attr_set[dev] = 1;
  }
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)DH);
  dim3 grid((n_q + at::QT - 1) / at::QT, heads, rows);
  return launch_pdl(attention_bf16_kernel<DH>, grid, dim3(128), smem, c.stream, mq, mq2, mk, mk2, mv, mv2,
                    static_cast<bf16*>(o), n_q, T, D, scale_log2, c.err);
}

cudaError_t launch_attention(const Ctx& c, int dtype, const void* q, const void* k, const void* v, void* o,
                             int rows, int n_q, int T, int heads, int dh) {
  if (rows == 0 || n_q == 0) return cudaSuccess;
  if (dtype == LAZYMAR_F32) {
    const size_t smem = (size_t)4 * (T + dh) * sizeof(float);
    if (smem > 48 * 1024) {
      cudaError_t e = cudaFuncSetAttribute(attention_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem);
      if (e != cudaSuccess) return e;
    }
    dim3 grid((n_q + 3) / 4, heads, rows);
    return launch_pdl(attention_f32_kernel, grid, dim3(128), smem, c.stream, static_cast<const float*>(q),
                      static_cast<const float*>(k), static_cast<const float*>(v), static_cast<float*>(o), n_q, T,
                      heads * dh, dh, 1.0f / sqrtf((float)dh));
  }
  if (dh == 64) return launch_attn_bf16<64>(c, q, k, v, o, rows, n_q, T, heads);
  return launch_attn_bf16<80>(c, q, k, v, o, rows, n_q, T, heads);
}

}  // namespace lm
