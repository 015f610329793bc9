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

// ---------------------------------------------------------------------------
// bf16, head width 64: tcgen05 tensor cores, accumulators in tensor memory
// ---------------------------------------------------------------------------
// One CTA per (128-query tile, head, row). Warps 0-3 run the softmax (thread t
// owns query row t = tensor-memory lane t) and issue the TMA loads; lane 0 of
// warp 4 issues the MMAs. Keys stream in 64-key chunks c:
//   S(c)  = Q K(c)^T      (tcgen05.mma 128 x 64 x 64, K-major operands) into
//                         tensor-memory columns [0, 64);
//   P(c)  = exp2(S(c) * log2(e)/sqrt(d) - m), written as bf16 to shared memory;
//   O    += P(c) V(c)     (A = P K-major, B = the V tile as loaded, MN-major)
//                         into columns [64, 128), accumulated across chunks.
// The MMA warp issues S(c+1) as soon as the softmax warps have read S(c), so
// the tensor core works while the softmax runs. The running max m is raised
// only when a row's chunk max exceeds it by more than 8 (log2 units): the
// final O / l is the same for any m that is at least every key's score - 8 and
// P stays below 2^8, while O in tensor memory is rescaled only on those
// (rare) raises. K and V have separate two-stage rings: K(c+2) refills as soon
// as S(c) has completed, V(c+1) as soon as O has absorbed P(c-1) V(c-1).
namespace at2 {
constexpr int QT = 128;   // queries per CTA (MMA M)
constexpr int KC = 64;    // keys per chunk
constexpr int THREADS = 160;
constexpr int Q_BYTES = QT * 128;    // 128 rows x 64 bf16, 128B swizzle
constexpr int KV_BYTES = KC * 128;   // 64 rows x 64 bf16
constexpr int P_BYTES = QT * 128;    // 128 rows x 64 keys
constexpr int SMEM = 1024 + Q_BYTES + 4 * KV_BYTES + P_BYTES + 256;
constexpr uint32_t TMEM_COLS = 128;  // S [0, 64), O [64, 128)
constexpr float RESCALE_THRESHOLD = 8.0f;
// kind::f16, D fp32, A/B bf16, N = 64, M = 128; bit 16 marks B as MN-major.
constexpr uint32_t IDESC_S = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(64 >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
constexpr uint32_t IDESC_PV = IDESC_S | (1u << 16);
// Shared-memory descriptors, 128B swizzle. K-major operand (Q, K, P): the
// stride between 8-row groups (SBO) is 1024 B, the leading offset unused (1).
// MN-major V tile (rows = keys = the K dimension, 64 head dims = one 128-byte
// swizzle atom along N): 8-key groups are 1024 B apart; N is a single atom, so
// the N-direction offset never applies and is given the same 1024 B.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
__device__ __forceinline__ uint64_t sw128_mn_desc(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)(1024 >> 4) << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
// byte offset of 16-byte chunk c of row r in a 128-byte-row, 128B-swizzled tile
__device__ __forceinline__ uint32_t sw(int r, int c) { return (uint32_t)(r * 128 + (((c ^ r) & 7) << 4)); }
enum { B_Q = 0, B_K = 1, B_V = 3, B_S_FULL = 5, B_S_FREE = 6, B_P_FULL = 7, B_O_DONE = 8, N_BARS = 9 };
}  // namespace at2

__global__ void __launch_bounds__(at2::THREADS, 3) attention_tc_kernel(const __grid_constant__ CUtensorMap tmQ,
                                                                       const __grid_constant__ CUtensorMap tmK,
                                                                       const __grid_constant__ CUtensorMap tmV,
                                                                       bf16* o, int n_q, int T, int D,
                                                                       float scale_log2, unsigned* err) {
  using namespace at2;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;                    // 16 KB
  uint8_t* sK = sQ + Q_BYTES;            // 2 x 8 KB
  uint8_t* sV = sK + 2 * KV_BYTES;       // 2 x 8 KB
  uint8_t* sP = sV + 2 * KV_BYTES;       // 16 KB (also the output staging tile)
  uint64_t* bars = reinterpret_cast<uint64_t*>(sP + P_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + N_BARS);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int qt = blockIdx.x, h = blockIdx.y, r = blockIdx.z;
  const int q0 = r * n_q + qt * QT, kv0 = r * T, col = h * 64;
  const int nck = (T + KC - 1) / KC;
  // Softmax warps whose 32 query rows all lie beyond n_q sit out: their rows of
  // S, P and O are never read back (matrix rows are independent).
  const int n_valid = min(QT, n_q - qt * QT);
  const int n_act = (n_valid + 31) / 32;

  if (tid == 0) {
    for (int i = 0; i < N_BARS; ++i) mbar_init(&bars[i], (i == B_S_FREE || i == B_P_FULL) ? (uint32_t)n_act : 1u);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 4) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  pdl_trigger();

  auto load_k = [&](int c) {
    uint64_t* bar = &bars[B_K + (c & 1)];
    mbar_arrive_expect_tx(bar, KV_BYTES);
    tma_load_2d(&tmK, bar, sK + (c & 1) * KV_BYTES, col, kv0 + c * KC);
  };
  auto load_v = [&](int c) {
    uint64_t* bar = &bars[B_V + (c & 1)];
    mbar_arrive_expect_tx(bar, KV_BYTES);
    tma_load_2d(&tmV, bar, sV + (c & 1) * KV_BYTES, col, kv0 + c * KC);
  };

  if (warp == 4) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint64_t qd = sw128_desc(smem_u32(sQ)), pd = sw128_desc(smem_u32(sP));
      auto issue_s = [&](int c) {
        const uint64_t kd = sw128_desc(smem_u32(sK + (c & 1) * KV_BYTES));
#pragma unroll
        for (int k = 0; k < 4; ++k) umma_bf16(tmem, qd + 2 * k, kd + 2 * k, IDESC_S, k != 0 ? 1u : 0u);
        umma_commit(&bars[B_S_FULL]);
      };
      bool ok = mbar_wait(&bars[B_Q], 0, abort_flag, err) && mbar_wait(&bars[B_K], 0, abort_flag, err);
      if (ok) {
        tc_fence_after();
        issue_s(0);
      }
      for (int c = 0; c < nck && ok; ++c) {
        if (c + 1 < nck) {
          ok = mbar_wait(&bars[B_K + ((c + 1) & 1)], (uint32_t)((c + 1) >> 1) & 1u, abort_flag, err) &&
               mbar_wait(&bars[B_S_FREE], (uint32_t)c & 1u, abort_flag, err);
          if (!ok) break;
          tc_fence_after();
          issue_s(c + 1);
        }
        ok = mbar_wait(&bars[B_P_FULL], (uint32_t)c & 1u, abort_flag, err) &&
             mbar_wait(&bars[B_V + (c & 1)], (uint32_t)(c >> 1) & 1u, abort_flag, err);
        if (!ok) break;
        tc_fence_after();
        // 16 keys per MMA: 16 rows of the MN-major V tile = 2048 bytes.
        const uint64_t vd = sw128_mn_desc(smem_u32(sV + (c & 1) * KV_BYTES));
#pragma unroll
        for (int k = 0; k < 4; ++k)
          umma_bf16(tmem + 64, pd + 2 * k, vd + 128 * k, IDESC_PV, (c > 0 || k > 0) ? 1u : 0u);
        umma_commit(&bars[B_O_DONE]);
      }
    }
    __syncwarp();
  } else if (warp < n_act) {
    // ---------------- softmax warps (thread = query row) ----------------
    const uint32_t t_lane = (uint32_t)(warp * 32) << 16;
    if (tid == 0) {
      mbar_arrive_expect_tx(&bars[B_Q], Q_BYTES);
      tma_load_2d(&tmQ, &bars[B_Q], sQ, col, q0);
      load_k(0);
      if (nck > 1) load_k(1);
      load_v(0);
      if (nck > 1) load_v(1);
    }
    float m_run = -FLT_MAX, l_run = 0.f;
    bool ok = true;
    for (int c = 0; c < nck; ++c) {
      ok = __all_sync(0xffffffffu, mbar_wait(&bars[B_S_FULL], (uint32_t)c & 1u, abort_flag, err));
      if (!ok) break;
      tc_fence_after();
      if (tid == 0 && c + 2 < nck) load_k(c + 2);  // S(c) has read K stage c & 1
      float sv[64];
      {
        uint32_t ra[32], rb[32];
        tmem_ld32(tmem + t_lane, ra);
        tmem_ld32(tmem + t_lane + 32, rb);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          sv[i] = __uint_as_float(ra[i]);
          sv[32 + i] = __uint_as_float(rb[i]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars[B_S_FREE]);
      // row max of the raw scores; keys beyond T (the last chunk only) drop out
      float mloc = -FLT_MAX;
      if (c * KC + KC <= T) {
#pragma unroll
        for (int i = 0; i < 64; i += 2) mloc = fmax3(mloc, sv[i], sv[i + 1]);
      } else {
#pragma unroll
        for (int i = 0; i < 64; ++i) {
          sv[i] = (c * KC + i < T) ? sv[i] : -FLT_MAX;
          mloc = fmaxf(mloc, sv[i]);
        }
      }
      mloc *= scale_log2;  // log2 units (scale_log2 > 0 keeps the maximum)
      float alpha = 1.f;
      bool raise = false;
      if (c == 0) {
        m_run = mloc;
      } else if (mloc > m_run + RESCALE_THRESHOLD) {
        raise = true;
        alpha = exp2_approx(m_run - mloc);
        m_run = mloc;
      }
      // exponent arguments and the row sum two keys per instruction (the
      // softmax is bound by instruction issue)
      const unsigned long long sc2 = f32x2_pack(scale_log2, scale_log2), nm2 = f32x2_pack(-m_run, -m_run);
      unsigned long long ps2 = f32x2_pack(0.f, 0.f);
      uint32_t pk[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        float x0, x1;
        f32x2_unpack(f32x2_fma(f32x2_pack(sv[2 * i], sv[2 * i + 1]), sc2, nm2), x0, x1);
        const float p0 = exp2_approx(x0), p1 = exp2_approx(x1);
        ps2 = f32x2_add(ps2, f32x2_pack(p0, p1));
        pk[i] = pack_bf16(p0, p1);
      }
      float ps0, ps1;
      f32x2_unpack(ps2, ps0, ps1);
      const float psum = ps0 + ps1;
      // PV(c-1) must be complete before O is rescaled or P is overwritten.
      if (c > 0) {
        ok = __all_sync(0xffffffffu, mbar_wait(&bars[B_O_DONE], (uint32_t)(c - 1) & 1u, abort_flag, err));
        if (!ok) break;
        tc_fence_after();
        if (tid == 0 && c + 1 < nck) load_v(c + 1);  // V stage (c + 1) & 1 held V(c - 1)
        if (__any_sync(0xffffffffu, raise)) {
#pragma unroll 1
          for (int half = 0; half < 2; ++half) {
            uint32_t ra[32];
            tmem_ld32(tmem + t_lane + 64 + 32 * half, ra);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) ra[i] = __float_as_uint(__uint_as_float(ra[i]) * alpha);
            tmem_st32(tmem + t_lane + 64 + 32 * half, ra);
          }
          tmem_wait_st();
        }
      }
#pragma unroll
      for (int j = 0; j < 8; ++j)
        *reinterpret_cast<uint4*>(sP + sw(tid, j)) = make_uint4(pk[4 * j], pk[4 * j + 1], pk[4 * j + 2], pk[4 * j + 3]);
      l_run = l_run * alpha + psum;
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars[B_P_FULL]);
    }
    // epilogue: O / l for this row, staged through the P tile for whole-row stores
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&bars[B_O_DONE], (uint32_t)(nck - 1) & 1u, abort_flag, err));
    if (ok) {
      tc_fence_after();
      const float inv = 1.f / l_run;
      uint32_t ra[32], rb[32];
      tmem_ld32(tmem + t_lane + 64, ra);
      tmem_ld32(tmem + t_lane + 96, rb);
      tmem_wait_ld();
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        uint4 w0, w1;
        w0.x = pack_bf16(__uint_as_float(ra[8 * j + 0]) * inv, __uint_as_float(ra[8 * j + 1]) * inv);
        w0.y = pack_bf16(__uint_as_float(ra[8 * j + 2]) * inv, __uint_as_float(ra[8 * j + 3]) * inv);
        w0.z = pack_bf16(__uint_as_float(ra[8 * j + 4]) * inv, __uint_as_float(ra[8 * j + 5]) * inv);
        w0.w = pack_bf16(__uint_as_float(ra[8 * j + 6]) * inv, __uint_as_float(ra[8 * j + 7]) * inv);
        w1.x = pack_bf16(__uint_as_float(rb[8 * j + 0]) * inv, __uint_as_float(rb[8 * j + 1]) * inv);
        w1.y = pack_bf16(__uint_as_float(rb[8 * j + 2]) * inv, __uint_as_float(rb[8 * j + 3]) * inv);
        w1.z = pack_bf16(__uint_as_float(rb[8 * j + 4]) * inv, __uint_as_float(rb[8 * j + 5]) * inv);
        w1.w = pack_bf16(__uint_as_float(rb[8 * j + 6]) * inv, __uint_as_float(rb[8 * j + 7]) * inv);
        *reinterpret_cast<uint4*>(sP + sw(tid, j)) = w0;
        *reinterpret_cast<uint4*>(sP + sw(tid, 4 + j)) = w1;
      }
      __syncwarp();
      // the warp's 32 rows: 4 rows x 8 chunks of 16 bytes per instruction
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int row = warp * 32 + i * 4 + (lane >> 3), ch = lane & 7;
        const int qi = qt * QT + row;
        if (qi < n_q) {
          const uint4 val = *reinterpret_cast<const uint4*>(sP + sw(row, ch));
          *reinterpret_cast<uint4*>(o + (size_t)(r * n_q + qi) * D + col + 8 * ch) = val;
        }
      }
    }
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 4) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
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

static cudaError_t launch_attn_tc(const Ctx& c, const void* q, const void* k, const void* v, void* o, int rows,
                                  int n_q, int T, int heads) {
  if (T < 1) return cudaErrorInvalidValue;  // the kernel's final wait needs at least one key chunk
  const int D = heads * 64;
  const uint64_t pitch = (uint64_t)D * 2;
  CUtensorMap mq, mk, mv;
  if (!make_tmap_bf16(&mq, q, D, (uint64_t)rows * n_q, pitch, 64, at2::QT, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_tmap_bf16(&mk, k, D, (uint64_t)rows * T, pitch, 64, at2::KC, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_tmap_bf16(&mv, v, D, (uint64_t)rows * T, pitch, 64, at2::KC, CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  static int attr_set[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    cudaError_t e =
        cudaFuncSetAttribute(attention_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, at2::SMEM);
    if (e != cudaSuccess) return e;
    attr_set[dev] = 1;
  }
  const float scale_log2 = 1.4426950408889634f / 8.0f;  // log2(e) / sqrt(64)
  dim3 grid((n_q + at2::QT - 1) / at2::QT, heads, rows);
  return launch_pdl(attention_tc_kernel, grid, dim3(at2::THREADS), (size_t)at2::SMEM, c.stream, mq, mk, mv,
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
  if (dh == 64) return launch_attn_tc(c, q, k, v, o, rows, n_q, T, heads);
  return launch_attn_bf16<80>(c, q, k, v, o, rows, n_q, T, heads);
}

}  // namespace lm
