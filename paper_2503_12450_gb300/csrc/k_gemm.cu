// GEMMs of the MAR block: QKV, attention output, MLP up and down projections
// (Eq. 9's F(X[I_compute]) for the token subset, and the full-layer forms).
//
// bf16: a persistent, warp-specialised tcgen05 kernel. Warp 0 streams A and W
// tiles with TMA (128B swizzle) into a ring of shared-memory stages, warp 1
// issues tcgen05.mma (128 x BN x 16, fp32 accumulators in tensor memory,
// double-buffered so the epilogue of one tile overlaps the main loop of the
// next) and eight epilogue warps drain the accumulators with tcgen05.ld and
// apply the fused epilogue: bias, GELU, fp32 residual add, or the Q/K/V split
// with the K/V rows scattered into the token cache (row_map).
//
// f32: a 64x64 register-tiled CUDA-core kernel with the same epilogues (the
// tensor cores have no fp32 kind; this serves the fp32 configuration).
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include <cstring>

#include "lazymar_internal.cuh"

namespace lm {

// ---------------------------------------------------------------------------
// Epilogue shared by both kernels: NC consecutive columns of one row.
// ---------------------------------------------------------------------------
template <typename T, int NC>
__device__ __forceinline__ void epilogue_apply(const GemmEpi& e, int row, int col0, float* v) {
  if (e.bias) {
    float bv[NC];
    Vec<T, NC>::load(static_cast<const T*>(e.bias) + col0, bv);
#pragma unroll
    for (int i = 0; i < NC; ++i) v[i] += bv[i];
  }
  switch (e.mode) {
    case LAZYMAR_EPI_GELU:
#pragma unroll
      for (int i = 0; i < NC; ++i) v[i] = gelu_erf(v[i]);
      Vec<T, NC>::store(static_cast<T*>(e.out) + (size_t)row * e.ldo + col0, v);
      break;
    case LAZYMAR_EPI_SILU:
#pragma unroll
      for (int i = 0; i < NC; ++i) v[i] = silu(v[i]);
      Vec<T, NC>::store(static_cast<T*>(e.out) + (size_t)row * e.ldo + col0, v);
      break;
    case LAZYMAR_EPI_RESIDUAL: {
      float* o = static_cast<float*>(e.out) + (size_t)row * e.ldo + col0;
      float r[NC];
      Vec<float, NC>::load(o, r);
      if (e.gate) {
        float g[NC];
        Vec<T, NC>::load(static_cast<const T*>(e.gate) + (size_t)row * e.ldg + col0, g);
#pragma unroll
        for (int i = 0; i < NC; ++i) v[i] *= g[i];
      }
#pragma unroll
      for (int i = 0; i < NC; ++i) r[i] += v[i];
      Vec<float, NC>::store(o, r);
      break;
    }
    case LAZYMAR_EPI_QKV: {
      const int part = col0 / e.D;
      const int c = col0 - part * e.D;
      T* dst;
      if (part == 0) {
        dst = static_cast<T*>(e.out) + (size_t)row * e.D + c;
      } else {
        const int drow = e.row_map ? e.row_map[row] : row;
        dst = static_cast<T*>(part == 1 ? e.k_out : e.v_out) + (size_t)drow * e.D + c;
      }
      Vec<T, NC>::store(dst, v);
      break;
    }
    default:
      Vec<T, NC>::store(static_cast<T*>(e.out) + (size_t)row * e.ldo + col0, v);
      break;
  }
}

// ---------------------------------------------------------------------------
// tcgen05 kernel
// ---------------------------------------------------------------------------
namespace tc {
constexpr int BM = 128;  // rows per tile = MMA M (one accumulator lane per row)

// Epilogue kinds: BF16OUT stores bf16 (bias / GELU / Q-K-V split); the two
// residual kinds add into the fp32 residual stream. RESID_WIDE stages whole
// 32-column fp32 chunks (for short K, where the epilogue bounds the kernel, at
// the cost of one pipeline stage); RESID_HALF stages 16-column halves and keeps
// every stage (for long K, where the main loop bounds it).
// RESID_WIDE_GATED is RESID_WIDE with a per-element gate on the product
// (out += gate * y, the adaptive-LayerNorm residual of the diffusion head),
// a separate instantiation so that the ungated kinds carry no gate code.
// BF16OUT_SILU is BF16OUT with the SiLU activation, likewise separate.
enum EpiKind { BF16OUT = 0, RESID_WIDE = 1, RESID_HALF = 2, RESID_WIDE_GATED = 3, BF16OUT_SILU = 4 };
template <int EK>
constexpr bool is_wide() { return EK == RESID_WIDE || EK == RESID_WIDE_GATED; }
template <int EK>
constexpr bool is_bf16out() { return EK == BF16OUT || EK == BF16OUT_SILU; }

// BK: K per pipeline stage (elements), one or two swizzle atoms. A 128-wide
// tile runs 128-deep stages (two atoms, eight MMAs per barrier round trip):
// its 128 x 128 x 16 MMAs are too short to hide the per-stage wait and commit
// at 64 (measured 13-19 % faster); wider tiles keep 64 for a deeper ring.
// F8: E4M3 operands (kind::f8f6f4): a 128-byte atom holds 128 elements and an
// MMA step is K = 32, still 32 bytes; BK = 128 is one atom, the bytes of a
// 64-deep bf16 stage.
template <int BN, int EK, int BK, int F8 = 0>
struct Cfg {
  static constexpr int EB = F8 ? 1 : 2;          // bytes per operand element
  static constexpr int ATOM_E = 128 / EB;        // elements per 128-byte swizzle atom
  static constexpr int ATOMS = BK / ATOM_E;
  // (64-wide tiles, with half the B tile per stage, afford one more stage)
  static constexpr int STAGES = ATOMS == 2 ? (is_wide<EK>() ? 2 : 3) + (BN == 64 ? 1 : 0)
                                          : is_wide<EK>() ? (BN == 256 ? 3 : BN == 192 ? 4 : 5)
                                                             : (BN == 256 ? 4 : BN == 192 ? 5 : 6);
  static constexpr uint32_t A_BYTES = BM * BK * EB;
  static constexpr uint32_t B_BYTES = BN * BK * EB;
  static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  // two accumulator buffers (columns [0, BN) and [BN, 2 BN)); the allocation
  // is a power of two
  static constexpr uint32_t TMEM_COLS = 2 * BN <= 256 ? 256 : 512;
  // Per-warp staging of 32 rows (64 or 128 bytes each), rows padded by 16
  // bytes so that both the row-wise writes and the column-block reads are
  // bank-conflict-lean.
  // Epilogue warps: the bf16-output kinds use four (three for BN = 192) per
  // tensor-memory lane quarter, so more warps share a tile's conversion,
  // GELU and stores; the residual kinds, with more live registers, two.
  static constexpr int EPI_WARPS = !is_bf16out<EK>() ? 8 : (BN == 192 ? 12 : BN == 64 ? 8 : 16);
  static constexpr int THREADS = 64 + EPI_WARPS * 32;
  static constexpr int CHUNKS = BN / 32 / (EPI_WARPS / 4);  // 32-column chunks per warp and tile
  // Per-warp staging of 32 rows: bf16 rows of 64 bytes, 16-byte blocks
  // swizzled by row (conflict-free row-wise writes and column-block reads);
  // fp32 rows of 64 or 128 bytes padded by 16 bytes.
  static constexpr uint32_t ROW_BYTES = is_wide<EK>() ? 128 : 64;
  static constexpr uint32_t STG_PITCH = is_bf16out<EK>() ? 64 : ROW_BYTES + 16;
  static constexpr uint32_t STG_BYTES = 32 * STG_PITCH;
  static constexpr size_t SMEM = 1024 + (size_t)STAGES * STAGE_BYTES + EPI_WARPS * STG_BYTES + 256;
  // Instruction descriptor: D fp32 (bit 4); kind::f16 with A and B bf16
  // (bits 7-9 and 10-12 = 1), or kind::f8f6f4 with A and B E4M3 (format 0);
  // both K-major, N >> 3 at bit 17, M >> 4 at bit 24.
  static constexpr uint32_t IDESC = (1u << 4) | (F8 ? 0u : (1u << 7) | (1u << 10)) | ((uint32_t)(BN >> 3) << 17) |
                                    ((uint32_t)(BM >> 4) << 24);
};

// Shared-memory matrix descriptor of a K-major tile written by TMA with
// SWIZZLE_128B: rows of 128 bytes, 8-row groups 1024 bytes apart (stride byte
// offset), descriptor version 1 (bit 46), layout SWIZZLE_128B (2 at bit 61).
// The leading byte offset is not used by this layout.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// Four packed bf16 values as floats (the gates of four residual columns).
__device__ __forceinline__ float4 bf16x4_to_f4(uint2 u) {
  const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
  const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
  return make_float4(a.x, a.y, b.x, b.y);
}

// Destination row pointer of a bf16 epilogue for tile row `row`, column `col`
// (a 32-column chunk never straddles the Q/K/V parts).
__device__ __forceinline__ bf16* out_row(const GemmEpi& e, int row, int col) {
  if (e.mode != LAZYMAR_EPI_QKV) return static_cast<bf16*>(e.out) + (size_t)row * e.ldo + col;
  const int part = col / e.D;
  const int c = col - part * e.D;
  if (part == 0) return static_cast<bf16*>(e.out) + (size_t)row * e.D + c;
  const int drow = e.row_map ? e.row_map[row] : row;
  return static_cast<bf16*>(part == 1 ? e.k_out : e.v_out) + (size_t)drow * e.D + c;
}
}  // namespace tc

template <int BN, int EK, int BK, int F8 = 0>
__global__ void __launch_bounds__(tc::Cfg<BN, EK, BK, F8>::THREADS, 1)
    gemm_bf16_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                        const __grid_constant__ CUtensorMap tmO0, const __grid_constant__ CUtensorMap tmO1,
                        const __grid_constant__ CUtensorMap tmO2, int tma_out, int M, int N, int K, GemmEpi epi,
                        unsigned* err) {
  using C = tc::Cfg<BN, EK, BK, F8>;
  constexpr bool RESID = !tc::is_bf16out<EK>();
  static_assert(!F8 || EK == tc::BF16OUT, "E4M3 operands: bf16-output epilogue only");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint8_t* sStg = smem + C::STAGES * C::STAGE_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(sStg + C::EPI_WARPS * C::STG_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* acc_full = empty + C::STAGES;
  uint64_t* acc_empty = acc_full + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // Tiles are numbered column-tile fastest: the CTAs running at the same time
  // cover a few row tiles completely, so each activation row tile is fetched
  // from memory once and shared through L2 by the CTAs that use it (the
  // weights, at most a few MB, stay in L2 throughout).
  const int num_m = (M + tc::BM - 1) / tc::BM;
  const int num_n = N / BN;
  const int tiles = num_m * num_n;
  const int KB = K / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], C::EPI_WARPS);
    }
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
    if (tma_out) {
      prefetch_tmap(&tmO0);
      if (epi.mode == LAZYMAR_EPI_QKV) {
        prefetch_tmap(&tmO1);
        prefetch_tmap(&tmO2);
      }
    }
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // Weights are never written by any kernel, so the producer fetches the
  // weight tiles of its first stages before waiting for the predecessor grid;
  // every other access follows pdl_wait().
  int pre = 0;
  if (warp == 0 && lane == 0 && (int)blockIdx.x < tiles) {
    const int n0 = ((int)blockIdx.x % num_n) * BN;
    pre = KB < C::STAGES ? KB : C::STAGES;
    for (int s = 0; s < pre; ++s) {
      mbar_arrive_expect_tx(&full[s], C::STAGE_BYTES);
#pragma unroll
      for (int a = 0; a < C::ATOMS; ++a)
        tma_load_2d(&tmB, &full[s], sB + s * C::B_BYTES + a * (C::B_BYTES / C::ATOMS), s * BK + a * C::ATOM_E, n0);
    }
  }
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < tiles && ok; tile += gridDim.x) {
        const int m0 = (tile / num_n) * tc::BM, n0 = (tile % num_n) * BN;
        for (int kb = 0; kb < KB; ++kb) {
          if (tile == (int)blockIdx.x && kb < pre) {
            // weight tile already in flight on this stage: add the activations
#pragma unroll
            for (int a = 0; a < C::ATOMS; ++a)
              tma_load_2d(&tmA, &full[stage], sA + stage * C::A_BYTES + a * (C::A_BYTES / C::ATOMS),
                          kb * BK + a * C::ATOM_E, m0);
          } else {
            if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, err)) { ok = false; break; }
            mbar_arrive_expect_tx(&full[stage], C::STAGE_BYTES);
#pragma unroll
            for (int a = 0; a < C::ATOMS; ++a) {
              tma_load_2d(&tmA, &full[stage], sA + stage * C::A_BYTES + a * (C::A_BYTES / C::ATOMS),
                          kb * BK + a * C::ATOM_E, m0);
              tma_load_2d(&tmB, &full[stage], sB + stage * C::B_BYTES + a * (C::B_BYTES / C::ATOMS),
                          kb * BK + a * C::ATOM_E, n0);
            }
          }
          if (++stage == C::STAGES) { stage = 0; phase ^= 1u; }
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < tiles && ok; tile += gridDim.x, ++it) {
        const int buf = it & 1;
        const uint32_t use = (uint32_t)(it >> 1) & 1u;
        if (!mbar_wait(&acc_empty[buf], use ^ 1u, abort_flag, err)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(buf * BN);
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, err)) { ok = false; break; }
          tc_fence_after();
          const uint64_t a0 = tc::sw128_desc(smem_u32(sA + stage * C::A_BYTES));
          const uint64_t b0 = tc::sw128_desc(smem_u32(sB + stage * C::B_BYTES));
#pragma unroll
          for (int k = 0; k < C::ATOMS * 4; ++k) {  // +32 bytes per MMA step inside an atom
            const int a = k / 4, ks = k % 4;
            const uint64_t ao = (uint64_t)((a * (C::A_BYTES / C::ATOMS)) >> 4) + 2 * ks;
            const uint64_t bo = (uint64_t)((a * (C::B_BYTES / C::ATOMS)) >> 4) + 2 * ks;
            if (F8)
              umma_e4m3(d_tmem, a0 + ao, b0 + bo, C::IDESC, (kb | k) != 0 ? 1u : 0u);
            else
              umma_bf16(d_tmem, a0 + ao, b0 + bo, C::IDESC, (kb | k) != 0 ? 1u : 0u);
          }
          umma_commit(&empty[stage]);
          if (++stage == C::STAGES) { stage = 0; phase ^= 1u; }
        }
        if (ok) umma_commit(&acc_full[buf]);
      }
    }
    __syncwarp();
  } else {
    // ---------------- epilogue warps ----------------
    // Each warp owns 32 accumulator rows (its TMEM lane quarter) and one of the
    // EPI_WARPS / 4 column ranges of the tile, processed as 32 x 32 chunks
    // (CHUNKS per tile). tcgen05.ld gives one row
    // per thread; each chunk is transposed through the warp's staging buffer
    // (32 rows x 64 bytes: 32 bf16 columns, or 16 fp32 columns at a time) so
    // that every global store and residual load covers 8 rows x 64 contiguous
    // bytes per warp instruction. The residual of the next chunk is loaded
    // while the current one is processed, and the first chunk's before the
    // accumulator is ready.
    const int ew = warp - 2;        // 0 .. EPI_WARPS - 1
    const int quarter = warp & 3;   // tensor-memory lanes this warp may read
    const int half = ew >> 2;       // which column range of the tile (of EPI_WARPS / 4)
    constexpr int CHUNKS = C::CHUNKS;
    uint8_t* stg = sStg + ew * C::STG_BYTES;
    const int cr = lane >> 2;       // row within an 8-row pass
    const int cq = lane & 3;        // 16-byte block within the 64-byte row segment
    float* const res_base = static_cast<float*>(epi.out);
    int it = 0;
    for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x, ++it) {
      const int buf = it & 1;
      const uint32_t use = (uint32_t)(it >> 1) & 1u;
      const int m0 = (tile / num_n) * tc::BM, n0 = (tile % num_n) * BN;
      const int rbase = m0 + quarter * 32;  // first of this warp's 32 rows
      const int c0 = half * CHUNKS;
      // residual of a 32-column chunk in the coalesced layout: [16-col half][pass]
      float4 res[2][4];
      uint2 rbias[2];  // the 4 bias values of this lane's columns in each 16-column half (bf16)
      auto load_res = [&](int col) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          rbias[h] = epi.bias ? *reinterpret_cast<const uint2*>(static_cast<const bf16*>(epi.bias) + col + h * 16 + cq * 4)
                              : make_uint2(0u, 0u);
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            const int row = rbase + p * 8 + cr;
            res[h][p] = row < M ? *reinterpret_cast<const float4*>(res_base + (size_t)row * epi.ldo + col + h * 16 + cq * 4)
                                : make_float4(0.f, 0.f, 0.f, 0.f);
          }
        }
      };
      // RESID_WIDE layout: [pass] with 4 rows x 8 blocks of 16 bytes per pass
      // (gated kind: the gates of the same elements, prefetched alike)
      float4 resw[8];
      uint2 gatew[8];  // 4 bf16 gates each
      uint2 wbias;     // the 4 bias values of this lane's columns (bf16)
      auto load_resw = [&](int col) {
        const int wr = lane >> 3, wq = lane & 7;
        wbias = epi.bias ? *reinterpret_cast<const uint2*>(static_cast<const bf16*>(epi.bias) + col + wq * 4)
                         : make_uint2(0u, 0u);
#pragma unroll
        for (int p = 0; p < 8; ++p) {
          const int row = rbase + p * 4 + wr;
          resw[p] = row < M ? *reinterpret_cast<const float4*>(res_base + (size_t)row * epi.ldo + col + wq * 4)
                            : make_float4(0.f, 0.f, 0.f, 0.f);
          if (EK == tc::RESID_WIDE_GATED)
            gatew[p] = row < M ? *reinterpret_cast<const uint2*>(static_cast<const bf16*>(epi.gate) +
                                                                 (size_t)row * epi.ldg + col + wq * 4)
                               : make_uint2(0u, 0u);
        }
      };
      // bf16-output kinds: the bias of the next 32-column chunk (packed bf16),
      // loaded before it is needed, the first chunk's before the accumulator
      // is ready
      uint4 bpre[4];
      auto load_bias = [&](int col) {
        if (epi.bias) {
          const uint4* bp = reinterpret_cast<const uint4*>(static_cast<const bf16*>(epi.bias) + col);
#pragma unroll
          for (int j = 0; j < 4; ++j) bpre[j] = bp[j];
        }
      };
      if (EK == tc::RESID_HALF) load_res(n0 + c0 * 32);
      if (tc::is_wide<EK>()) load_resw(n0 + c0 * 32);
      if (tc::is_bf16out<EK>() && !F8) load_bias(n0 + c0 * 32);
      const bool ok = mbar_wait(&acc_full[buf], use, abort_flag, err);
      if (__any_sync(0xffffffffu, !ok)) break;
      tc_fence_after();
      // The tensor-memory load of chunk c + 1 is issued as soon as chunk c's
      // accumulator registers have been consumed, and waited for at the top
      // of the next iteration (the wait names the registers, so no use of
      // them moves above it).
      // (Only for the kinds where the extra live registers do not spill: the
      // residual kind over short K and the bf16-output kinds up to 192 wide.
      // The others load and wait at the top of each iteration.)
      constexpr bool PIPE = EK == tc::RESID_WIDE || (tc::is_bf16out<EK>() && BN <= 192);
      uint32_t r[32];
      auto tld = [&](int c) {
        tmem_ld32(tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(buf * BN + c * 32), r);
      };
      // The tile's accumulator buffer goes back to the MMA warp as soon as
      // this warp's last chunk is out of tensor memory, before its stores.
      auto release = [&] {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[buf]);
      };
      if (PIPE) tld(c0);
#pragma unroll 1
      for (int c = c0; c < c0 + CHUNKS; ++c) {
        const int col = n0 + c * 32;
        const bool more = c + 1 < c0 + CHUNKS;
        if (!PIPE) tld(c);
        tmem_wait_ld_regs(r);
        if (tc::is_wide<EK>()) {
          // whole 32-column fp32 chunk: 4 rows x 128 B per warp instruction
          float4* srow = reinterpret_cast<float4*>(stg + lane * C::STG_PITCH);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            srow[j] = make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                  __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
          if (PIPE && more) tld(c + 1);
          if (!more) release();  // the whole accumulator is out of tensor memory
          __syncwarp();
          const int wr = lane >> 3, wq = lane & 7;
          const float4 bq = tc::bf16x4_to_f4(wbias);  // prefetched with the residual
          float4 cur[8];
          uint2 curg[8];
#pragma unroll
          for (int p = 0; p < 8; ++p) {
            cur[p] = resw[p];
            if (EK == tc::RESID_WIDE_GATED) curg[p] = gatew[p];
          }
          if (c + 1 < c0 + CHUNKS) load_resw(col + 32);  // prefetch the next chunk
#pragma unroll
          for (int p = 0; p < 8; ++p) {
            const int lr = p * 4 + wr;
            const int row = rbase + lr;
            const float4 a = *reinterpret_cast<const float4*>(stg + lr * C::STG_PITCH + wq * 16);
            if (row < M) {
              float4 o;
              if (EK == tc::RESID_WIDE_GATED) {
                const float4 gg = tc::bf16x4_to_f4(curg[p]);
                o.x = fmaf(gg.x, a.x + bq.x, cur[p].x);
                o.y = fmaf(gg.y, a.y + bq.y, cur[p].y);
                o.z = fmaf(gg.z, a.z + bq.z, cur[p].z);
                o.w = fmaf(gg.w, a.w + bq.w, cur[p].w);
              } else {
                o.x = cur[p].x + (a.x + bq.x);
                o.y = cur[p].y + (a.y + bq.y);
                o.z = cur[p].z + (a.z + bq.z);
                o.w = cur[p].w + (a.w + bq.w);
              }
              *reinterpret_cast<float4*>(res_base + (size_t)row * epi.ldo + col + wq * 4) = o;
            }
          }
          __syncwarp();
        } else if (EK == tc::RESID_HALF) {
          float4 cur[2][4];
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int p = 0; p < 4; ++p) cur[h][p] = res[h][p];
          const uint2 cbias[2] = {rbias[0], rbias[1]};  // prefetched with the residual
          if (c + 1 < c0 + CHUNKS) load_res(col + 32);  // prefetch the next chunk
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            // stage 16 raw fp32 accumulator columns of this thread's row
            float4* srow = reinterpret_cast<float4*>(stg + lane * C::STG_PITCH);
#pragma unroll
            for (int j = 0; j < 4; ++j)
              srow[j] = make_float4(__uint_as_float(r[16 * h + 4 * j]), __uint_as_float(r[16 * h + 4 * j + 1]),
                                    __uint_as_float(r[16 * h + 4 * j + 2]), __uint_as_float(r[16 * h + 4 * j + 3]));
            if (h == 1 && !more) release();
            __syncwarp();
            const float4 bq = tc::bf16x4_to_f4(cbias[h]);
#pragma unroll
            for (int p = 0; p < 4; ++p) {
              const int lr = p * 8 + cr;
              const int row = rbase + lr;
              const float4 a = *reinterpret_cast<const float4*>(stg + lr * C::STG_PITCH + cq * 16);
              if (row < M) {
                float4 o;
                o.x = cur[h][p].x + (a.x + bq.x);
                o.y = cur[h][p].y + (a.y + bq.y);
                o.z = cur[h][p].z + (a.z + bq.z);
                o.w = cur[h][p].w + (a.w + bq.w);
                *reinterpret_cast<float4*>(res_base + (size_t)row * epi.ldo + col + h * 16 + cq * 4) = o;
              }
            }
            __syncwarp();
          }
        } else {
          // bias (+ GELU) in the row layout, bf16 to the staging buffer, then
          // whole-row-segment stores
          float v[32];
          if (F8) {
            // E4M3 weights carry one scale per output column: 8 columns at a
            // time, so that scales and biases do not hold 64 registers
#pragma unroll
            for (int g = 0; g < 4; ++g) {
              float sv[8], bb[8];
              Vec<float, 8>::load(epi.wscale + col + 8 * g, sv);
              if (epi.bias) {
                Vec<bf16, 8>::load(static_cast<const bf16*>(epi.bias) + col + 8 * g, bb);
              } else {
#pragma unroll
                for (int i = 0; i < 8; ++i) bb[i] = 0.f;
              }
#pragma unroll
              for (int i = 0; i < 8; ++i) v[8 * g + i] = fmaf(__uint_as_float(r[8 * g + i]), sv[i], bb[i]);
            }
          } else {
            if (epi.bias) {
              const uint32_t* bw = reinterpret_cast<const uint32_t*>(bpre);
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                const float2 b2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bw[i]));
                f32x2_unpack(f32x2_add(f32x2_pack(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1])),
                                       f32x2_pack(b2.x, b2.y)),
                             v[2 * i], v[2 * i + 1]);
              }
            } else {
#pragma unroll
              for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
            }
            // the next chunk's bias loads while this chunk is converted and stored
            if (c + 1 < c0 + CHUNKS) load_bias(col + 32);
          }
          if (EK == tc::BF16OUT_SILU) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = silu(v[i]);
          } else if (epi.mode == LAZYMAR_EPI_GELU) {
#pragma unroll
            for (int i = 0; i < 16; ++i) gelu_erf_x2(v[2 * i], v[2 * i + 1]);
          }
          uint4 pk[4];
          {
            uint32_t* w = reinterpret_cast<uint32_t*>(pk);
#pragma unroll
            for (int i = 0; i < 16; ++i) w[i] = pack_bf16(v[2 * i], v[2 * i + 1]);
          }
          if (PIPE && more) tld(c + 1);
          if (!more) release();
          if (tma_out) {
            // the previous chunk's store must have read the staging buffer
            if (lane == 0) bulk_wait_read();
            __syncwarp();
          }
          // row `lane`, 16-byte block j at block j ^ ((lane >> 1) & 3): the
          // TMA 64-byte swizzle of a 32 x 32 bf16 box
#pragma unroll
          for (int j = 0; j < 4; ++j)
            *reinterpret_cast<uint4*>(stg + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4)) = pk[j];
          if (tma_out) {
            // one TMA store of the 32 x 32 chunk; rows beyond M are clipped
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0 && rbase < M) {
              const int part = epi.mode == LAZYMAR_EPI_QKV ? col / epi.D : 0;
              const CUtensorMap* tm = part == 0 ? &tmO0 : part == 1 ? &tmO1 : &tmO2;
              tma_store_2d(tm, stg, col - part * epi.D, rbase);
              bulk_commit();
            }
          } else {
            __syncwarp();
#pragma unroll
            for (int p = 0; p < 4; ++p) {
              const int lr = p * 8 + cr;
              const int row = rbase + lr;
              const uint4 val = *reinterpret_cast<const uint4*>(stg + lr * 64 + ((cq ^ ((lr >> 1) & 3)) << 4));
              if (row < M) *reinterpret_cast<uint4*>(tc::out_row(epi, row, col) + cq * 8) = val;
            }
            __syncwarp();
          }
        }
      }
    }
    if (tma_out && lane == 0) bulk_wait_all();  // stores complete before the CTA exits
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// fp32 CUDA-core kernel: 64 x 64 tile, 256 threads, 4 x 4 outputs per thread
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) gemm_f32_kernel(const float* __restrict__ A, const float* __restrict__ W, int M,
                                                       int N, int K, GemmEpi epi) {
  __shared__ float As[16][64 + 4];
  __shared__ float Ws[16][64 + 4];
  pdl_wait();
  pdl_trigger();
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += 16) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int idx = threadIdx.x + i * 256;
      const int r = idx >> 4, c = idx & 15;
      As[c][r] = (m0 + r < M && k0 + c < K) ? A[(size_t)(m0 + r) * K + k0 + c] : 0.f;
      Ws[c][r] = (n0 + r < N && k0 + c < K) ? W[(size_t)(n0 + r) * K + k0 + c] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = As[kk][ty * 4 + i];
        b[i] = Ws[kk][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  const int col = n0 + tx * 4;
  if (col >= N) return;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int row = m0 + ty * 4 + i;
    if (row < M) epilogue_apply<float, 4>(epi, row, col, acc[i]);
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
static PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D tensor map over a row-major [outer, inner] matrix with the given row
// pitch, box [box_outer, box_inner], out-of-bounds elements read as zero.
static bool make_tmap_2d(CUtensorMapDataType dt, CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                         uint64_t pitch_bytes, uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swz) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {pitch_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  return enc(m, dt, 2, const_cast<void*>(base), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
bool make_tmap_bf16(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t pitch_bytes,
                    uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swz) {
  return make_tmap_2d(CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, m, base, inner, outer, pitch_bytes, box_inner, box_outer, swz);
}

bool gemm_supported(int dtype, int M, int N, int K, const GemmEpi& epi, const char** why) {
  if (M < 0 || N <= 0 || K <= 0) { *why = "M >= 0, N > 0, K > 0 required"; return false; }
  if (epi.mode < LAZYMAR_EPI_BIAS || epi.mode > LAZYMAR_EPI_SILU) { *why = "unknown epilogue"; return false; }
  if (epi.mode == LAZYMAR_EPI_QKV && (epi.D <= 0 || N != 3 * epi.D)) { *why = "QKV epilogue needs N = 3D"; return false; }
  if (epi.gate && (epi.mode != LAZYMAR_EPI_RESIDUAL || epi.ldg < N || epi.ldg % 4 != 0)) {
    *why = "a gate needs the residual epilogue and ldg >= N, ldg % 4 == 0"; return false;
  }
  if (dtype == LAZYMAR_E4M3) {
    if (K % 128 != 0) { *why = "E4M3 GEMM needs K % 128 == 0"; return false; }
    if (N % 128 != 0) { *why = "E4M3 GEMM needs N % 128 == 0"; return false; }
    if (epi.mode == LAZYMAR_EPI_RESIDUAL || epi.mode == LAZYMAR_EPI_SILU) {
      *why = "E4M3 GEMM: bias, GELU or Q/K/V epilogue only"; return false;
    }
    if (!epi.wscale) { *why = "E4M3 GEMM needs the per-column weight scales"; return false; }
    if (epi.mode == LAZYMAR_EPI_QKV && epi.D % 32 != 0) { *why = "QKV epilogue needs D % 32 == 0"; return false; }
    if (epi.mode != LAZYMAR_EPI_QKV && epi.ldo % 8 != 0) { *why = "ldo % 8 == 0 required"; return false; }
  } else if (dtype == LAZYMAR_BF16) {
    if (K % 64 != 0) { *why = "bf16 GEMM needs K % 64 == 0"; return false; }
    if (N % 128 != 0) { *why = "bf16 GEMM needs N % 128 == 0"; return false; }
    if (epi.mode == LAZYMAR_EPI_QKV && epi.D % 32 != 0) { *why = "QKV epilogue needs D % 32 == 0"; return false; }
    if (epi.mode != LAZYMAR_EPI_QKV && epi.ldo % 8 != 0) { *why = "ldo % 8 == 0 required"; return false; }
  } else if (dtype == LAZYMAR_F32) {
    if (K % 4 != 0 || N % 4 != 0) { *why = "f32 GEMM needs K % 4 == 0 and N % 4 == 0"; return false; }
    if (epi.mode == LAZYMAR_EPI_QKV && epi.D % 4 != 0) { *why = "QKV epilogue needs D % 4 == 0"; return false; }
    if (epi.mode != LAZYMAR_EPI_QKV && epi.ldo % 4 != 0) { *why = "ldo % 4 == 0 required"; return false; }
  } else {
    *why = "unknown dtype";
    return false;
  }
  return true;
}

template <int BN, int EK, int BK, int F8 = 0>
static cudaError_t launch_tc(const Ctx& c, const void* A, const void* W, int M, int N, int K, const GemmEpi& epi) {
  using C = tc::Cfg<BN, EK, BK, F8>;
  const CUtensorMapDataType dt = F8 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  CUtensorMap ta, tb;
  if (!make_tmap_2d(dt, &ta, A, (uint64_t)K, (uint64_t)M, (uint64_t)K * C::EB, C::ATOM_E, tc::BM,
                    CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_tmap_2d(dt, &tb, W, (uint64_t)K, (uint64_t)N, (uint64_t)K * C::EB, C::ATOM_E, BN,
                    CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  static int attr_set[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(gemm_bf16_tc_kernel<BN, EK, BK, F8>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
    if (e != cudaSuccess) return e;
    attr_set[dev] = 1;
  }
  // bf16 outputs leave through TMA stores of 32 x 32 boxes (64-byte swizzle),
  // except Q/K/V with a row map, whose K/V rows are scattered
  CUtensorMap to[3];
  std::memset(to, 0, sizeof to);
  int tma_out = 0;
  if (tc::is_bf16out<EK>() && !(epi.mode == LAZYMAR_EPI_QKV && epi.row_map)) {
    tma_out = 1;
    if (epi.mode == LAZYMAR_EPI_QKV) {
      const void* outs[3] = {epi.out, epi.k_out, epi.v_out};
      for (int i = 0; i < 3; ++i)
        if (!make_tmap_bf16(&to[i], outs[i], (uint64_t)epi.D, (uint64_t)M, (uint64_t)epi.D * 2, 32, 32,
                            CU_TENSOR_MAP_SWIZZLE_64B))
          return cudaErrorInvalidValue;
    } else if (!make_tmap_bf16(&to[0], epi.out, (uint64_t)N, (uint64_t)M, (uint64_t)epi.ldo * 2, 32, 32,
                               CU_TENSOR_MAP_SWIZZLE_64B)) {
      return cudaErrorInvalidValue;
    }
  }
  const int tiles = ((M + tc::BM - 1) / tc::BM) * (N / BN);
  const int grid = tiles < c.num_sms ? tiles : c.num_sms;
  return launch_pdl(gemm_bf16_tc_kernel<BN, EK, BK, F8>, dim3(grid), dim3(C::THREADS), C::SMEM, c.stream, ta, tb, to[0], to[1],
                    to[2], tma_out, M, N, K,
                    epi, c.err);
}

// Relative time of one round of tiles of width bn (see launch_gemm).
static int tile_time(int bn, bool resid_half) {
  static const int widths[4] = {256, 192, 128, 64};
  static const int t_bf[4] = {256, 243, 187, 153}, t_rh[4] = {256, 199, 153, 110};
  for (int i = 0; i < 4; ++i)
    if (widths[i] == bn) return resid_half ? t_rh[i] : t_bf[i];
  return 256;
}

// Tile width with the fewest rounds of tiles over the SMs x the time of one
// tile, and that cost.
static int choose_bn(const Ctx& c, int M, int N, const GemmEpi& epi, int K, long* cost) {
  const long mt = (M + tc::BM - 1) / tc::BM;
  const bool resid_half = epi.mode == LAZYMAR_EPI_RESIDUAL && !epi.gate && K >= 2048;
  const int widths[4] = {256, 192, 128, 64};
  int bn = 128;
  long best = -1;
  for (int i = 0; i < 4; ++i) {
    if (N % widths[i] != 0) continue;
    const long rounds = (mt * (N / widths[i]) + c.num_sms - 1) / c.num_sms;
    const long t = rounds * tile_time(widths[i], resid_half);
    if (best < 0 || t < best) {
      best = t;
      bn = widths[i];
    }
  }
  *cost = best;
  return bn;
}

// The epilogue of rows [m0, M) of a GEMM as a GEMM of its own.
static GemmEpi epi_from_row(const GemmEpi& e, int m0) {
  GemmEpi t = e;
  if (e.mode == LAZYMAR_EPI_QKV) {
    t.out = static_cast<bf16*>(e.out) + (size_t)m0 * e.D;
    if (e.row_map) {
      t.row_map = e.row_map + m0;
    } else {
      t.k_out = static_cast<bf16*>(e.k_out) + (size_t)m0 * e.D;
      t.v_out = static_cast<bf16*>(e.v_out) + (size_t)m0 * e.D;
    }
  } else if (e.mode == LAZYMAR_EPI_RESIDUAL) {
    t.out = static_cast<float*>(e.out) + (size_t)m0 * e.ldo;
    if (e.gate) t.gate = static_cast<const bf16*>(e.gate) + (size_t)m0 * e.ldg;
  } else {
    t.out = static_cast<bf16*>(e.out) + (size_t)m0 * e.ldo;
  }
  return t;
}

// Kernels issued by launch_gemm on this thread (a last-wave split issues two).
static thread_local long long t_gemm_kernels = 0;
long long gemm_kernels_issued() { return t_gemm_kernels; }

static cudaError_t launch_bn_impl(const Ctx& c, int dtype, const void* A, const void* W, int M, int N, int K,
                                  const GemmEpi& epi, int bn);
static cudaError_t launch_bn(const Ctx& c, int dtype, const void* A, const void* W, int M, int N, int K,
                             const GemmEpi& epi, int bn) {
  const cudaError_t e = launch_bn_impl(c, dtype, A, W, M, N, K, epi, bn);
  if (e == cudaSuccess) ++t_gemm_kernels;
  return e;
}

static cudaError_t launch_bn_impl(const Ctx& c, int dtype, const void* A, const void* W, int M, int N, int K,
                                  const GemmEpi& epi, int bn) {
  if (dtype == LAZYMAR_E4M3) {
    // E4M3 operands (bf16-output kinds): a 128-element stage is one atom; the
    // tile width follows the bf16 choice
    if (bn == 256) return launch_tc<256, tc::BF16OUT, 128, 1>(c, A, W, M, N, K, epi);
    if (bn == 192) return launch_tc<192, tc::BF16OUT, 128, 1>(c, A, W, M, N, K, epi);
    return launch_tc<128, tc::BF16OUT, 128, 1>(c, A, W, M, N, K, epi);
  }
  const int ek = epi.mode == LAZYMAR_EPI_SILU       ? tc::BF16OUT_SILU
                 : epi.mode != LAZYMAR_EPI_RESIDUAL ? tc::BF16OUT
                 : epi.gate                          ? tc::RESID_WIDE_GATED
                 : K < 2048                          ? tc::RESID_WIDE
                                                     : tc::RESID_HALF;
  if (bn == 192) {
    if (ek == tc::RESID_WIDE) return launch_tc<192, tc::RESID_WIDE, 64>(c, A, W, M, N, K, epi);
    if (ek == tc::RESID_WIDE_GATED) return launch_tc<192, tc::RESID_WIDE_GATED, 64>(c, A, W, M, N, K, epi);
    if (ek == tc::RESID_HALF) return launch_tc<192, tc::RESID_HALF, 64>(c, A, W, M, N, K, epi);
    if (ek == tc::BF16OUT_SILU) return launch_tc<192, tc::BF16OUT_SILU, 64>(c, A, W, M, N, K, epi);
    return launch_tc<192, tc::BF16OUT, 64>(c, A, W, M, N, K, epi);
  }
  if (bn == 256) {
    if (ek == tc::RESID_WIDE) return launch_tc<256, tc::RESID_WIDE, 64>(c, A, W, M, N, K, epi);
    if (ek == tc::RESID_WIDE_GATED) return launch_tc<256, tc::RESID_WIDE_GATED, 64>(c, A, W, M, N, K, epi);
    if (ek == tc::RESID_HALF) return launch_tc<256, tc::RESID_HALF, 64>(c, A, W, M, N, K, epi);
    if (ek == tc::BF16OUT_SILU) return launch_tc<256, tc::BF16OUT_SILU, 64>(c, A, W, M, N, K, epi);
    return launch_tc<256, tc::BF16OUT, 64>(c, A, W, M, N, K, epi);
  }
  if (bn == 64) {
    if (K % 128 == 0) {
      if (ek == tc::RESID_WIDE) return launch_tc<64, tc::RESID_WIDE, 128>(c, A, W, M, N, K, epi);
      if (ek == tc::RESID_WIDE_GATED) return launch_tc<64, tc::RESID_WIDE_GATED, 128>(c, A, W, M, N, K, epi);
      if (ek == tc::RESID_HALF) return launch_tc<64, tc::RESID_HALF, 128>(c, A, W, M, N, K, epi);
      if (ek == tc::BF16OUT_SILU) return launch_tc<64, tc::BF16OUT_SILU, 128>(c, A, W, M, N, K, epi);
      return launch_tc<64, tc::BF16OUT, 128>(c, A, W, M, N, K, epi);
    }
    if (ek == tc::RESID_WIDE) return launch_tc<64, tc::RESID_WIDE, 64>(c, A, W, M, N, K, epi);
    if (ek == tc::RESID_WIDE_GATED) return launch_tc<64, tc::RESID_WIDE_GATED, 64>(c, A, W, M, N, K, epi);
    if (ek == tc::RESID_HALF) return launch_tc<64, tc::RESID_HALF, 64>(c, A, W, M, N, K, epi);
    if (ek == tc::BF16OUT_SILU) return launch_tc<64, tc::BF16OUT_SILU, 64>(c, A, W, M, N, K, epi);
    return launch_tc<64, tc::BF16OUT, 64>(c, A, W, M, N, K, epi);
  }
  if (K % 128 == 0) {
    if (ek == tc::RESID_WIDE) return launch_tc<128, tc::RESID_WIDE, 128>(c, A, W, M, N, K, epi);
    if (ek == tc::RESID_WIDE_GATED) return launch_tc<128, tc::RESID_WIDE_GATED, 128>(c, A, W, M, N, K, epi);
    if (ek == tc::RESID_HALF) return launch_tc<128, tc::RESID_HALF, 128>(c, A, W, M, N, K, epi);
    if (ek == tc::BF16OUT_SILU) return launch_tc<128, tc::BF16OUT_SILU, 128>(c, A, W, M, N, K, epi);
    return launch_tc<128, tc::BF16OUT, 128>(c, A, W, M, N, K, epi);
  }
  if (ek == tc::RESID_WIDE) return launch_tc<128, tc::RESID_WIDE, 64>(c, A, W, M, N, K, epi);
  if (ek == tc::RESID_WIDE_GATED) return launch_tc<128, tc::RESID_WIDE_GATED, 64>(c, A, W, M, N, K, epi);
  if (ek == tc::RESID_HALF) return launch_tc<128, tc::RESID_HALF, 64>(c, A, W, M, N, K, epi);
  if (ek == tc::BF16OUT_SILU) return launch_tc<128, tc::BF16OUT_SILU, 64>(c, A, W, M, N, K, epi);
  return launch_tc<128, tc::BF16OUT, 64>(c, A, W, M, N, K, epi);
}



cudaError_t launch_gemm(const Ctx& c, int dtype, const void* A, const void* W, int M, int N, int K,
                        const GemmEpi& epi, int flags) {
  if (M == 0) return cudaSuccess;
  if (dtype == LAZYMAR_F32) {
    dim3 grid((N + 63) / 64, (M + 63) / 64);
    const cudaError_t e = launch_pdl(gemm_f32_kernel, grid, dim3(256), 0, c.stream, static_cast<const float*>(A),
                                     static_cast<const float*>(W), M, N, K, epi);
    if (e == cudaSuccess) ++t_gemm_kernels;
    return e;
  }
  // Tile width: the one with the fewest rounds of tiles over the SMs x the
  // time of one tile. Relative tile times 187 : 243 : 256 for BN = 128 : 192 :
  // 256 (measured, one round of 128 x BN x 3072 tiles): a narrower tile does
  // proportionally less work per pipeline stage and runs well below the
  // BN = 256 rate. BN = 64 (153, on the line through the 128 and 256 points)
  // wins only when the 128-wide tiles fit in one round with SMs to spare: the
  // few-row GEMMs of the diffusion head. The fp32-residual epilogue over long K
  // (fc2) costs in proportion to the tile width: its measured round times at
  // K = 3072 are 153 : 199 : 256 (110 for 64), under which the full-layer fc2
  // (480 tiles of 256 in 4 rounds, or 640 of 192 in 5) takes the 192-wide tiles.
  if (flags == 2 && N % 256 == 0) return launch_bn(c, dtype, A, W, M, N, K, epi, 256);
  if (flags == 3 && N % 192 == 0) return launch_bn(c, dtype, A, W, M, N, K, epi, 192);
  if (flags == 4) return launch_bn(c, dtype, A, W, M, N, K, epi, 64);
  if (flags != 0) return launch_bn(c, dtype, A, W, M, N, K, epi, 128);
  long cost = 0;
  const int bn = choose_bn(c, M, N, epi, K, &cost);
  // Last-wave split of the fp32-residual GEMM over short K (the
  // out-projection): when its tiles fill several rounds but the last one only
  // partly, the row tiles of the whole waves run as one launch and the
  // remaining rows as a second launch, with the tile width that suits their
  // count (narrower tiles spread them over all SMs), if the model puts the
  // pair at least 2 % below the one launch. Measured on the MAR-B full layer:
  // the partial fourth round of 256-wide tiles costs a whole round (8.2 us),
  // while the last 8 row tiles as 64-wide tiles take 4.9 us (34.1 -> 30.9
  // us). The other kinds lose: the residual over long K (fc2) runs its partial
  // last round faster than a full one (32 tiles of 192 in 10.8 us against
  // 17.1 us), and the full-layer Q/K/V went 55.9 -> 57.6 us split.
  if (dtype == LAZYMAR_BF16 && epi.mode == LAZYMAR_EPI_RESIDUAL && !epi.gate && K < 2048) {
    const long mt = (M + tc::BM - 1) / tc::BM, nn = N / bn;
    const long rounds = (mt * nn + c.num_sms - 1) / c.num_sms;
    const long body_rt = rounds >= 3 ? (rounds - 1) * c.num_sms / nn : 0;  // whole row tiles of the full waves
    if (body_rt > 0 && body_rt < mt) {
      const int Mb = (int)(body_rt * tc::BM);
      long tail_cost = 0;
      const int tail_bn = choose_bn(c, M - Mb, N, epi, K, &tail_cost);
      const long body_rounds = (body_rt * nn + c.num_sms - 1) / c.num_sms;
      const long split_cost = body_rounds * tile_time(bn, false) + tail_cost;
      if (split_cost * 50 <= cost * 49) {
        const cudaError_t e = launch_bn(c, dtype, A, W, Mb, N, K, epi, bn);
        if (e != cudaSuccess) return e;
        return launch_bn(c, dtype, static_cast<const bf16*>(A) + (size_t)Mb * K, W, M - Mb, N, K,
                         epi_from_row(epi, Mb), tail_bn);
      }
    }
  }
  return launch_bn(c, dtype, A, W, M, N, K, epi, bn);
}

}  // namespace lm
