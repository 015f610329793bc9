// Internal declarations shared by the translation units of liblazymar.so:
// device helpers, inline-PTX wrappers for sm_103a (mbarrier, TMA, tcgen05,
// mma.sync, ldmatrix) and the launchers each kernel file exports.
#pragma once

#include <nvtx3/nvToolsExt.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>
#include <utility>

#include "../../include/lazymar.h"

namespace lm {

using bf16 = __nv_bfloat16;

// Bits of the device error word.
enum : unsigned {
  ERR_TIMEOUT = 1u,  // a bounded wait on an mbarrier expired
  ERR_INDEX = 2u,    // an out-of-range or non-increasing token index was clamped
  ERR_LABEL = 4u,    // a class label outside [0, n_classes) was replaced by 0
};

// Upper bound for any single wait on a barrier inside a kernel (wall clock).
constexpr unsigned long long kWaitLimitNs = 2000000000ull;

// Everything a launcher needs besides its own arguments.
struct Ctx {
  cudaStream_t stream;
  unsigned* err;  // device error word
  int num_sms;
};

// ---------------------------------------------------------------------------
// Scalar helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(bf16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float x) { return __float2bfloat16_rn(x); }

// Hardware approximations of 1/x and 2^x (relative error about 2^-22).
__device__ __forceinline__ float rcp_approx(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float exp2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// GELU(x) = x Phi(x) = max(x, 0) - |x| h(|x|), where h(u) = Phi(-u) =
// erfc(u / sqrt 2) / 2 is the normal tail. h is evaluated as 2^P(u) with P a
// degree-5 polynomial fitted to log2 h on u in [0, 6] (weighted least squares
// towards minimax; coefficients from csrc/gen_gelu_poly.py); u is clamped to 6,
// where h < 1e-9. In fp32 the result is within 2.8e-7 * max(1, |x|) of the
// exact erf GELU. Per element: one special-function instruction and eight
// ALU ones (the MLP epilogue applies it to every element of the 4D-wide
// hidden layer and is instruction-bound). The ReLU term is (x + |x|) / 2 so
// that a NaN input stays NaN.
__device__ __forceinline__ float gelu_erf(float x) {
  constexpr float kGeluP0 = -1.000018716e+00f;
  constexpr float kGeluP1 = -1.150941610e+00f;
  constexpr float kGeluP2 = -4.596132934e-01f;
  constexpr float kGeluP3 = -5.220982432e-02f;
  constexpr float kGeluP4 = 7.249599788e-03f;
  constexpr float kGeluP5 = -4.984181724e-04f;
  const float u = fminf(fabsf(x), 6.0f);
  float p = fmaf(kGeluP5, u, kGeluP4);
  p = fmaf(p, u, kGeluP3);
  p = fmaf(p, u, kGeluP2);
  p = fmaf(p, u, kGeluP1);
  p = fmaf(p, u, kGeluP0);
  const float h = exp2_approx(p);
  return fmaf(-u, h, 0.5f * (x + fabsf(x)));
}

// SiLU(x) = x sigmoid(x) = x / (1 + 2^(-x log2 e)); for x below about -88
// the denominator overflows to infinity and the quotient is -0.
__device__ __forceinline__ float silu(float x) {
  return __fdividef(x, 1.f + exp2_approx(-1.4426950408889634f * x));
}

// Three-input maximum (one instruction for two new values).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
// Paired fp32 arithmetic: two lanes of fp32 in one 64-bit register pair, one
// instruction per pair (round to nearest, as the scalar forms).
__device__ __forceinline__ unsigned long long f32x2_pack(float lo, float hi) {
  unsigned long long r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f32x2_unpack(unsigned long long r, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(r));
}
__device__ __forceinline__ unsigned long long f32x2_fma(unsigned long long a, unsigned long long b,
                                                       unsigned long long c) {
  unsigned long long d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ unsigned long long f32x2_add(unsigned long long a, unsigned long long b) {
  unsigned long long d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ unsigned long long f32x2_mul(unsigned long long a, unsigned long long b) {
  unsigned long long d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// gelu_erf of two values with paired fp32 instructions, bit for bit the
// scalar results: the polynomial runs in v = -u with the odd coefficients
// negated (each Horner step is the scalar one with both operands negated, so
// its rounding is the same), and -u h + (x + |x|) / 2 is the scalar fma.
__device__ __forceinline__ void gelu_erf_x2(float& x0, float& x1) {
  constexpr float kGeluP0 = -1.000018716e+00f;
  constexpr float kGeluP1 = -1.150941610e+00f;
  constexpr float kGeluP2 = -4.596132934e-01f;
  constexpr float kGeluP3 = -5.220982432e-02f;
  constexpr float kGeluP4 = 7.249599788e-03f;
  constexpr float kGeluP5 = -4.984181724e-04f;
  const float v0 = fmaxf(-fabsf(x0), -6.0f), v1 = fmaxf(-fabsf(x1), -6.0f);
  const unsigned long long v = f32x2_pack(v0, v1);
  unsigned long long p = f32x2_fma(f32x2_pack(-kGeluP5, -kGeluP5), v, f32x2_pack(kGeluP4, kGeluP4));
  p = f32x2_fma(p, v, f32x2_pack(-kGeluP3, -kGeluP3));
  p = f32x2_fma(p, v, f32x2_pack(kGeluP2, kGeluP2));
  p = f32x2_fma(p, v, f32x2_pack(-kGeluP1, -kGeluP1));
  p = f32x2_fma(p, v, f32x2_pack(kGeluP0, kGeluP0));
  float p0, p1;
  f32x2_unpack(p, p0, p1);
  const unsigned long long h = f32x2_pack(exp2_approx(p0), exp2_approx(p1));
  const unsigned long long half = f32x2_mul(f32x2_add(f32x2_pack(x0, x1), f32x2_pack(fabsf(x0), fabsf(x1))),
                                            f32x2_pack(0.5f, 0.5f));
  f32x2_unpack(f32x2_fma(v, h, half), x0, x1);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Vector load/store of NC consecutive elements converted to/from fp32.
// bf16: NC % 8 == 0 (16-byte chunks); float: NC % 4 == 0.
template <typename T, int NC> struct Vec;
template <int NC> struct Vec<bf16, NC> {
  static_assert(NC % 8 == 0, "bf16 vectors are 8-element chunks");
  __device__ __forceinline__ static void load(const bf16* p, float* v) {
#pragma unroll
    for (int c = 0; c < NC / 8; ++c) {
      uint4 u = reinterpret_cast<const uint4*>(p)[c];
      const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float2 f = __bfloat1622float2(h[i]);
        v[c * 8 + 2 * i] = f.x;
        v[c * 8 + 2 * i + 1] = f.y;
      }
    }
  }
  __device__ __forceinline__ static void store(bf16* p, const float* v) {
#pragma unroll
    for (int c = 0; c < NC / 8; ++c) {
      uint4 u;
      __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
      for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(v[c * 8 + 2 * i], v[c * 8 + 2 * i + 1]);
      reinterpret_cast<uint4*>(p)[c] = u;
    }
  }
};
template <int NC> struct Vec<float, NC> {
  static_assert(NC % 4 == 0, "float vectors are 4-element chunks");
  __device__ __forceinline__ static void load(const float* p, float* v) {
#pragma unroll
    for (int c = 0; c < NC / 4; ++c) {
      float4 f = reinterpret_cast<const float4*>(p)[c];
      v[4 * c] = f.x; v[4 * c + 1] = f.y; v[4 * c + 2] = f.z; v[4 * c + 3] = f.w;
    }
  }
  __device__ __forceinline__ static void store(float* p, const float* v) {
#pragma unroll
    for (int c = 0; c < NC / 4; ++c)
      reinterpret_cast<float4*>(p)[c] = make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
  }
};

// ---------------------------------------------------------------------------
// Programmatic dependent launch
// ---------------------------------------------------------------------------
// Every kernel is launched so that it may start while its predecessor in the
// stream drains: its CTAs can initialise barriers, allocate tensor memory and
// prefetch descriptors early. pdl_wait() must precede the kernel's first access
// to global memory that a predecessor writes or reads; it returns once the
// predecessor grid has completed and its writes are visible. pdl_trigger()
// allows the successor to be scheduled once every CTA of this grid has issued
// it (so a successor never takes an SM a not-yet-started CTA of this grid
// needs). Both are no-ops for a kernel launched without the attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// ---------------------------------------------------------------------------
// Shared-memory barriers and TMA (PTX ISA: mbarrier, cp.async.bulk.tensor)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
// One bounded wait step: the thread is suspended until the phase completes or
// the suspend hint (1 ms) passes, so waiting warps do not take issue slots from
// working ones.
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(1000000u)
      : "memory");
  return ok != 0;
}
// Waits for the phase with the given parity to complete. Gives up (returns
// false) when *abort_flag is raised by another thread of the CTA or after
// kWaitLimitNs, in which case it raises *abort_flag and ERR_TIMEOUT.
__device__ __forceinline__ bool mbar_wait_limit(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                                unsigned* err, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 0) {
      if (*abort_flag) return false;
      if (globaltimer_ns() - t0 > limit_ns) {
        *abort_flag = 1;
        atomicOr(err, ERR_TIMEOUT);
        return false;
      }
    }
  }
}
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          unsigned* err) {
  return mbar_wait_limit(bar, parity, abort_flag, err, kWaitLimitNs);
}
// Orders this thread's view of prior generic-proxy shared-memory accesses
// (made visible to it by a CTA barrier) before its subsequent async-proxy
// operations, e.g. a TMA load that overwrites a stage other warps have read.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void prefetch_tmap(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}
// 2-D tiled TMA load of one box into shared memory, completing on `bar`.
// c0 is the innermost (contiguous) coordinate.
__device__ __forceinline__ void tma_load_2d(const void* tmap, uint64_t* bar, void* dst, int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
      : "memory");
}

// 2-D tiled TMA store of one box from shared memory (bulk-group completion).
__device__ __forceinline__ void tma_store_2d(const void* tmap, const void* src, int c0, int c1) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(tmap)),
               "r"(c0), "r"(c1), "r"(smem_u32(src))
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// Waits until the committed bulk stores of this thread have read their
// shared-memory source (the buffer may be rewritten).
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// Waits until the committed bulk stores of this thread have completed.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// ---------------------------------------------------------------------------
// tcgen05 (5th-generation tensor cores, accumulators in tensor memory)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)),
               "r"(ncols)
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
// D[tmem] (+)= A[smem] * B[smem]^T, bf16 inputs, fp32 accumulate (kind::f16).
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// D[tmem] (+)= A[smem] * B[smem]^T, E4M3 inputs, fp32 accumulate (kind::f8f6f4).
__device__ __forceinline__ void umma_e4m3(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on `bar` once all tcgen05.mma previously issued by this thread complete.
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}
// 32 lanes x 32 consecutive 32-bit columns of tensor memory into registers.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
        "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
// tcgen05.wait::ld naming the destination registers of the outstanding load
// as in/out operands, so that no use of them is scheduled before the wait
// (the load writes them asynchronously): lets a load be issued early, while
// earlier work is still in progress, and waited for where it is needed.
__device__ __forceinline__ void tmem_wait_ld_regs(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                 "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                 "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]),
                 "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
               :
               : "memory");
}
// 32 lanes x 32 consecutive 32-bit columns from registers into tensor memory.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
      "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
      "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// 32 lanes x 16 consecutive 32-bit columns (the 16-column remainder of an 80-wide head).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
}
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

// ---------------------------------------------------------------------------
// Warp-level mma.sync / ldmatrix (attention)
// ---------------------------------------------------------------------------
// Shared- and tensor-memory reads carry a "memory" clobber: without it the
// compiler may move them across the mbarrier wait that makes a TMA-filled
// stage (or a committed accumulator) valid, or across the barrier after which
// the stage is refilled, and read stale data.
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1)
      : "memory");
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// ---------------------------------------------------------------------------
// Launchers (each defined in its own translation unit)
// ---------------------------------------------------------------------------
// GEMM epilogue description (see lazymar_linear).
struct GemmEpi {
  int mode;             // LAZYMAR_EPI_*
  const void* bias;     // [N] in the GEMM dtype, or nullptr
  void* out;            // BIAS/GELU: [M, ldo] dtype; RESIDUAL: [M, ldo] fp32; QKV: Q [M, D]
  int ldo;
  void* k_out;          // QKV: K destination rows
  void* v_out;          // QKV: V destination rows
  const int* row_map;   // QKV: destination row of K/V for row m (nullptr = m)
  int D;                // QKV: width of each of Q, K, V
  // RESIDUAL only: out += gate * y with gate [M, ldg] in the GEMM dtype (the
  // gated residual of an adaptive-LayerNorm block), or nullptr for out += y
  const void* gate;
  int ldg;
  // E4M3 operands only: per-column scale of the weights ([N] fp32), applied
  // to the accumulator before the bias
  const float* wscale;
};
cudaError_t launch_gemm(const Ctx& c, int dtype, const void* A, const void* W, int M, int N, int K,
                        const GemmEpi& epi, int flags);
// Running count of the GEMM kernels launch_gemm has issued on this thread
// (a GEMM split into two launches counts two).
long long gemm_kernels_issued();
// Checks the preconditions of launch_gemm; returns false with a message.
bool gemm_supported(int dtype, int M, int N, int K, const GemmEpi& epi, const char** why);

cudaError_t launch_attention(const Ctx& c, int dtype, const void* q, const void* k, const void* v, void* o,
                             int rows, int n_q, int T, int heads, int dh);
bool attention_supported(int dtype, int heads, int dh, const char** why);

// dtype LAZYMAR_E4M3: bf16 gain/shift, E4M3 output (the A operand of an
// 8-bit GEMM); otherwise gain, shift and output in dtype.
cudaError_t launch_layernorm(const Ctx& c, int dtype, const float* x, const int* row_map, const void* g,
                             const void* b, void* y, float* x_copy, int M, int D, float eps);
// Final LayerNorm of compact rows into the [rows, n_img, D] output cache:
// row m holds token tok = row_map ? row_map[m] : m (tok = r*T + t); buffer
// tokens (t < n_buffer) are skipped.
cudaError_t launch_final_ln(const Ctx& c, int dtype, const float* x, const int* row_map, int T, int n_buffer,
                            int n_img, const void* g, const void* b, void* z, int M, int D, float eps);
cudaError_t launch_embed(const Ctx& c, int dtype, const float* lat, const uint8_t* mask, const int* labels,
                         const void* pos, const void* cls, const void* mask_emb, const void* ew, const void* eb,
                         float* H, int rows, int B, int T, int n_buffer, int n_img, int D, int token_dim,
                         int n_classes);
cudaError_t launch_cast(const Ctx& c, int dtype, const float* x, void* y, size_t n);
// Row i of qc / xc = row row_map[i] of q / x (D columns; D a multiple of 8).
cudaError_t launch_gather_rows(const Ctx& c, int dtype, const void* q, const float* x, const int* row_map, void* qc,
                               float* xc, int M, int D);
// E4M3 copy of a bf16 weight matrix [rows, cols] with one scale per row
// (max |w| / 448): q [rows, cols] bytes, scale [rows] fp32.
cudaError_t launch_quantize_e4m3(const Ctx& c, const void* w, int rows, int cols, void* q, float* scale);

cudaError_t launch_similarity(const Ctx& c, int dtype, const void* cur, void* cache, double* S, int rows, int T,
                              int D, bool copy);
// Diagnostic: one CTA waits on an mbarrier that nothing completes, for at most
// limit_ns (the bounded-wait failure path of every pipelined kernel).
cudaError_t launch_stuck_wait(const Ctx& c, uint64_t limit_ns);
cudaError_t launch_topk(const Ctx& c, const double* S, int rows, int T, int N, int* idx, int* row_map,
                        int rule = 0, const uint8_t* prio = nullptr, const uint32_t* keys = nullptr);
cudaError_t launch_idx_check(const Ctx& c, const int* idx_in, int rows, int T, int N, int* idx, int* row_map);
cudaError_t launch_cfg(const Ctx& c, int dtype, int mode, const void* zc, const void* zu, void* delta,
                       float gamma, size_t n, void* zu_out, void* g_out);

// Up to kMaxCopySegs byte ranges copied by one kernel (the step inputs into
// the handle's staging buffers). Each source is device memory or page-locked
// host memory the device can address.
constexpr int kMaxCopySegs = 6;
struct CopyList {
  const void* src[kMaxCopySegs];
  void* dst[kMaxCopySegs];
  unsigned long long bytes[kMaxCopySegs];
  int n;
};
cudaError_t launch_copy_list(const Ctx& c, const CopyList& L);

// NVTX range for the lifetime of the object (header-only NVTX v3: a no-op
// unless a profiler has attached its tool library).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

// Records `msg` as the calling thread's last error (lazymar_last_error) and
// returns `s`.
lazymar_status report_error(lazymar_status s, const char* msg);

}  // namespace lm
