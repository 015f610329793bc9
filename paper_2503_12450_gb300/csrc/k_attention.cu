// Bidirectional multi-head attention of Eq. 3 with a query subset: the queries
// of the recomputed tokens (I_compute) attend over all T keys of their
// sequence, fresh ones for I_compute and cached ones for I_cache (Eq. 9). The
// full-layer form is the same kernel with every token as a query.
//
// bf16: attention_tc_kernel, tcgen05 tensor cores with the accumulators in
// tensor memory and Q/K/V tiles staged by TMA, for heads of width 64 (MAR-B,
// MAR-L) and 80 (MAR-H).
//
// f32: one warp per query on CUDA cores (fp32 configuration).
#include <cuda.h>

#include <cfloat>

#include "lazymar_internal.cuh"

namespace lm {

bool make_tmap_bf16(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t pitch_bytes,
                    uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swz);

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
// bf16: tcgen05 tensor cores, accumulators in tensor memory
// ---------------------------------------------------------------------------
// One CTA per (128-query tile, head, row). Warps 0-3 run the softmax (thread t
// owns query row t = tensor-memory lane t) and issue the TMA loads; lane 0 of
// warp 4 issues the MMAs. Keys stream in 64-key chunks c:
//   S(c)  = Q K(c)^T      (tcgen05.mma 128 x 64 x DH, K-major operands) into
//                         tensor-memory columns [0, 64);
//   P(c)  = exp2(S(c) * log2(e)/sqrt(d) - m), written as bf16 to shared memory;
//   O    += P(c) V(c)     (A = P K-major, B = the V tile as loaded, MN-major)
//                         into columns [64, 64 + DH), accumulated across chunks.
// The MMA warp issues S(c+1) as soon as the softmax warps have read S(c), so
// the tensor core works while the softmax runs. The running max m is raised
// only when a row's chunk max exceeds it by more than 8 (log2 units): the
// final O / l is the same for any m that is at least every key's score - 8 and
// P stays below 2^8, while O in tensor memory is rescaled only on those
// (rare) raises. K and V have separate two-stage rings: K(c+2) refills as soon
// as S(c) has completed, V(c+1) as soon as O has absorbed P(c-1) V(c-1).
//
// A head of width 80 is a 64-column part (128-byte swizzle, as for width 64)
// and a 16-column remainder (32-byte swizzle: rows of 32 bytes, 8-row groups
// 256 bytes apart), each loaded by its own TMA box. S takes four 16-deep MMAs
// on the first part and one on the remainder; P V takes, per 16 keys, an
// N = 64 MMA on the first part of V into O columns [64, 128) and an N = 16 MMA
// on the remainder into [128, 144).
namespace at2 {
constexpr int QT = 128;   // queries per CTA (MMA M)
constexpr int KC = 64;    // keys per chunk
constexpr int THREADS = 160;
constexpr int Q_BYTES = QT * 128;    // 128 rows x 64 bf16, 128B swizzle
constexpr int KV_BYTES = KC * 128;   // 64 rows x 64 bf16
constexpr int P_BYTES = QT * 128;    // 128 rows x 64 keys
constexpr int Q2_BYTES = QT * 32;    // 128 rows x 16 bf16, 32B swizzle (80-wide heads)
constexpr int KV2_BYTES = KC * 32;   // 64 rows x 16 bf16
constexpr float RESCALE_THRESHOLD = 8.0f;
template <int DH>
struct Cfg {
  static_assert(DH == 64 || DH == 80, "head width 64 or 80");
  static constexpr bool TAIL = DH == 80;
  static constexpr int TAIL_BYTES = TAIL ? Q2_BYTES + 4 * KV2_BYTES : 0;
  static constexpr int SMEM = 1024 + Q_BYTES + 4 * KV_BYTES + P_BYTES + TAIL_BYTES + 256;
  static constexpr uint32_t TMEM_COLS = TAIL ? 256 : 128;  // S [0, 64), O [64, 64 + DH)
  static constexpr uint32_t Q_TX = Q_BYTES + (TAIL ? Q2_BYTES : 0);
  static constexpr uint32_t KV_TX = KV_BYTES + (TAIL ? KV2_BYTES : 0);
  static constexpr int MIN_BLOCKS = TAIL ? 2 : 3;  // shared memory allows three (64) or two (80) per SM
};
// kind::f16, D fp32, A/B bf16, M = 128, N = 64 (or 16); bit 16 marks B as MN-major.
constexpr uint32_t IDESC_S = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(64 >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
constexpr uint32_t IDESC_PV = IDESC_S | (1u << 16);
constexpr uint32_t IDESC_PV16 =
    (1u << 4) | (1u << 7) | (1u << 10) | (1u << 16) | ((uint32_t)(16 >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
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
// 32B swizzle (layout 6), 32-byte rows in 8-row groups 256 B apart. Used for
// the 16-column remainders: as a K-major operand the MMA's 16-deep K step is
// exactly one row of the atom; as the MN-major V remainder its 16 columns are
// one atom along N. Both offsets are the 256 B group stride (the other offset
// never applies to a single atom).
__device__ __forceinline__ uint64_t sw32_desc(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)(256 >> 4) << 16) | ((uint64_t)(256 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)6 << 61);
}
// byte offset of 16-byte chunk c of row r in a 128-byte-row, 128B-swizzled tile
__device__ __forceinline__ uint32_t sw(int r, int c) { return (uint32_t)(r * 128 + (((c ^ r) & 7) << 4)); }
enum { B_Q = 0, B_K = 1, B_V = 3, B_S_FULL = 5, B_S_FREE = 6, B_P_FULL = 7, B_O_DONE = 8, N_BARS = 9 };
}  // namespace at2

template <int DH>
__global__ void __launch_bounds__(at2::THREADS, at2::Cfg<DH>::MIN_BLOCKS)
    attention_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmQ2,
                        const __grid_constant__ CUtensorMap tmK2, const __grid_constant__ CUtensorMap tmV2, bf16* o,
                        int n_q, int T, int D, float scale_log2, unsigned* err) {
  using namespace at2;
  using C = Cfg<DH>;
  constexpr bool TAIL = C::TAIL;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;                    // 16 KB
  uint8_t* sK = sQ + Q_BYTES;            // 2 x 8 KB
  uint8_t* sV = sK + 2 * KV_BYTES;       // 2 x 8 KB
  uint8_t* sP = sV + 2 * KV_BYTES;       // 16 KB (also the output staging tile)
  uint8_t* sQ2 = sP + P_BYTES;           // 80-wide heads: 4 KB, then 2 x 2 KB of K and of V remainders
  uint8_t* sK2 = sQ2 + Q2_BYTES;
  uint8_t* sV2 = sK2 + 2 * KV2_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sP + P_BYTES + C::TAIL_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + N_BARS);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int qt = blockIdx.x, h = blockIdx.y, r = blockIdx.z;
  const int q0 = r * n_q + qt * QT, kv0 = r * T, col = h * DH;
  const int nck = (T + KC - 1) / KC;
  // Softmax warps whose 32 query rows all lie beyond n_q sit out: their rows of
  // S, P and O are never read back (matrix rows are independent).
  const int n_valid = min(QT, n_q - qt * QT);
  const int n_act = (n_valid + 31) / 32;

  if (tid == 0) {
    for (int i = 0; i < N_BARS; ++i) mbar_init(&bars[i], (i == B_S_FREE || i == B_P_FULL) ? (uint32_t)n_act : 1u);
    *abort_flag = 0;
    fence_mbar_init();
    // the descriptors are kernel parameters: fetched while the predecessor grid finishes
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
    if (TAIL) {
      prefetch_tmap(&tmQ2);
      prefetch_tmap(&tmK2);
      prefetch_tmap(&tmV2);
    }
  }
  if (warp == 4) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
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
    mbar_arrive_expect_tx(bar, C::KV_TX);
    tma_load_2d(&tmK, bar, sK + (c & 1) * KV_BYTES, col, kv0 + c * KC);
    if (TAIL) tma_load_2d(&tmK2, bar, sK2 + (c & 1) * KV2_BYTES, col + 64, kv0 + c * KC);
  };
  auto load_v = [&](int c) {
    uint64_t* bar = &bars[B_V + (c & 1)];
    mbar_arrive_expect_tx(bar, C::KV_TX);
    tma_load_2d(&tmV, bar, sV + (c & 1) * KV_BYTES, col, kv0 + c * KC);
    if (TAIL) tma_load_2d(&tmV2, bar, sV2 + (c & 1) * KV2_BYTES, col + 64, kv0 + c * KC);
  };

  if (warp == 4) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint64_t qd = sw128_desc(smem_u32(sQ)), pd = sw128_desc(smem_u32(sP));
      auto issue_s = [&](int c) {
        const uint64_t kd = sw128_desc(smem_u32(sK + (c & 1) * KV_BYTES));
#pragma unroll
        for (int k = 0; k < 4; ++k) umma_bf16(tmem, qd + 2 * k, kd + 2 * k, IDESC_S, k != 0 ? 1u : 0u);
        if (TAIL)
          umma_bf16(tmem, sw32_desc(smem_u32(sQ2)), sw32_desc(smem_u32(sK2 + (c & 1) * KV2_BYTES)), IDESC_S, 1u);
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
        // 16 keys per MMA: 16 rows of the MN-major V tile = 2048 bytes (512
        // bytes of the 32-byte-row remainder).
        const uint64_t vd = sw128_mn_desc(smem_u32(sV + (c & 1) * KV_BYTES));
        const uint64_t vd2 = sw32_desc(smem_u32(sV2 + (c & 1) * KV2_BYTES));
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          umma_bf16(tmem + 64, pd + 2 * k, vd + 128 * k, IDESC_PV, (c > 0 || k > 0) ? 1u : 0u);
          if (TAIL) umma_bf16(tmem + 128, pd + 2 * k, vd2 + 32 * k, IDESC_PV16, (c > 0 || k > 0) ? 1u : 0u);
        }
        umma_commit(&bars[B_O_DONE]);
      }
    }
    __syncwarp();
  } else if (warp < n_act) {
    // ---------------- softmax warps (thread = query row) ----------------
    const uint32_t t_lane = (uint32_t)(warp * 32) << 16;
    if (tid == 0) {
      mbar_arrive_expect_tx(&bars[B_Q], C::Q_TX);
      tma_load_2d(&tmQ, &bars[B_Q], sQ, col, q0);
      if (TAIL) tma_load_2d(&tmQ2, &bars[B_Q], sQ2, col + 64, q0);
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
        // four independent chains of three-input maxima (dependency depth 8
        // instead of 32)
        float mq[4] = {-FLT_MAX, -FLT_MAX, -FLT_MAX, -FLT_MAX};
#pragma unroll
        for (int i = 0; i < 64; i += 8) {
#pragma unroll
          for (int q = 0; q < 4; ++q) mq[q] = fmax3(mq[q], sv[i + 2 * q], sv[i + 2 * q + 1]);
        }
        mloc = fmax3(mq[0], mq[1], fmaxf(mq[2], mq[3]));
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
      // the row sum in four independent paired accumulators
      unsigned long long ps2[4] = {f32x2_pack(0.f, 0.f), f32x2_pack(0.f, 0.f), f32x2_pack(0.f, 0.f),
                                   f32x2_pack(0.f, 0.f)};
      uint32_t pk[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        float x0, x1;
        f32x2_unpack(f32x2_fma(f32x2_pack(sv[2 * i], sv[2 * i + 1]), sc2, nm2), x0, x1);
        const float p0 = exp2_approx(x0), p1 = exp2_approx(x1);
        ps2[i & 3] = f32x2_add(ps2[i & 3], f32x2_pack(p0, p1));
        pk[i] = pack_bf16(p0, p1);
      }
      float ps0, ps1;
      f32x2_unpack(f32x2_add(f32x2_add(ps2[0], ps2[1]), f32x2_add(ps2[2], ps2[3])), ps0, ps1);
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
          if (TAIL) {
            uint32_t rt[16];
            tmem_ld16(tmem + t_lane + 128, rt);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 16; ++i) rt[i] = __float_as_uint(__uint_as_float(rt[i]) * alpha);
            tmem_st16(tmem + t_lane + 128, rt);
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
    // epilogue: O / l for this row, staged through the P tile for whole-row
    // stores of the first 64 columns; the 16-column remainder of an 80-wide
    // head is stored by each thread (32 contiguous bytes)
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
      if (TAIL) {
        uint32_t rt[16];
        tmem_ld16(tmem + t_lane + 128, rt);
        tmem_wait_ld();
        const int qi = qt * QT + tid;
        if (qi < n_q) {
          uint4 t0, t1;
          t0.x = pack_bf16(__uint_as_float(rt[0]) * inv, __uint_as_float(rt[1]) * inv);
          t0.y = pack_bf16(__uint_as_float(rt[2]) * inv, __uint_as_float(rt[3]) * inv);
          t0.z = pack_bf16(__uint_as_float(rt[4]) * inv, __uint_as_float(rt[5]) * inv);
          t0.w = pack_bf16(__uint_as_float(rt[6]) * inv, __uint_as_float(rt[7]) * inv);
          t1.x = pack_bf16(__uint_as_float(rt[8]) * inv, __uint_as_float(rt[9]) * inv);
          t1.y = pack_bf16(__uint_as_float(rt[10]) * inv, __uint_as_float(rt[11]) * inv);
          t1.z = pack_bf16(__uint_as_float(rt[12]) * inv, __uint_as_float(rt[13]) * inv);
          t1.w = pack_bf16(__uint_as_float(rt[14]) * inv, __uint_as_float(rt[15]) * inv);
          uint4* dst = reinterpret_cast<uint4*>(o + (size_t)(r * n_q + qi) * D + col + 64);
          dst[0] = t0;
          dst[1] = t1;
        }
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
    tmem_dealloc(tmem, C::TMEM_COLS);
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
static cudaError_t launch_attn_tc(const Ctx& c, const void* q, const void* k, const void* v, void* o, int rows,
                                  int n_q, int T, int heads) {
  using C = at2::Cfg<DH>;
  if (T < 1) return cudaErrorInvalidValue;  // the kernel's final wait needs at least one key chunk
  const int D = heads * DH;
  const uint64_t pitch = (uint64_t)D * 2;
  CUtensorMap mq, mk, mv, mq2, mk2, mv2;
  if (!make_tmap_bf16(&mq, q, D, (uint64_t)rows * n_q, pitch, 64, at2::QT, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_tmap_bf16(&mk, k, D, (uint64_t)rows * T, pitch, 64, at2::KC, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_tmap_bf16(&mv, v, D, (uint64_t)rows * T, pitch, 64, at2::KC, CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  if (C::TAIL) {
    // 16-column remainders: x = h * 80 + 64 elements = 160 h + 128 bytes, a
    // multiple of 16 bytes as TMA requires
    if (!make_tmap_bf16(&mq2, q, D, (uint64_t)rows * n_q, pitch, 16, at2::QT, CU_TENSOR_MAP_SWIZZLE_32B) ||
        !make_tmap_bf16(&mk2, k, D, (uint64_t)rows * T, pitch, 16, at2::KC, CU_TENSOR_MAP_SWIZZLE_32B) ||
        !make_tmap_bf16(&mv2, v, D, (uint64_t)rows * T, pitch, 16, at2::KC, CU_TENSOR_MAP_SWIZZLE_32B))
      return cudaErrorInvalidValue;
  } else {
    mq2 = mq;
    mk2 = mk;
    mv2 = mv;
  }
  static int attr_set[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    cudaError_t e =
        cudaFuncSetAttribute(attention_tc_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    attr_set[dev] = 1;
  }
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)DH);  // log2(e) / sqrt(d)
  dim3 grid((n_q + at2::QT - 1) / at2::QT, heads, rows);
  return launch_pdl(attention_tc_kernel<DH>, grid, dim3(at2::THREADS), (size_t)C::SMEM, c.stream, mq, mk, mv, mq2,
                    mk2, mv2, static_cast<bf16*>(o), n_q, T, D, scale_log2, c.err);
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
  if (dh == 64) return launch_attn_tc<64>(c, q, k, v, o, rows, n_q, T, heads);
  return launch_attn_tc<80>(c, q, k, v, o, rows, n_q, T, heads);
}

}  // namespace lm
