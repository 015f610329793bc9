// Token selection of Eq. 8.
//
// similarity_kernel: one warp per token, spread over the whole GPU (a row has
// only T tokens, so one CTA per row would leave most SMs idle while streaming
// 2 x rows x T x D elements). Each lane reads 16-byte vectors of the current
// and cached representation and accumulates the dot product and both squared
// norms in fp64. bf16 x bf16 products are exact in fp64, and so are their sums
// for any realistic dynamic range, which makes S independent of the summation
// order: the oracle's fp64 sum gives bit-identical S, hence bit-identical
// selections (similarity_int_kernel computes those sums exactly on the integer
// pipe). fp32 x fp32 products are exact in fp64 too, but a sum of them is
// rounded at every addition, so the kernel's lane-strided order and the
// oracle's pairwise order can differ in the last bits of S (a relative 1e-15
// or so). Two tokens whose similarities lie that close may then be ordered
// differently; every other fp32 selection is identical. The current vector is
// copied over the cached one (the cache now holds this step's values).
//
// topk_kernel: one CTA per row. Each token's rank under the strict total order
// (S ascending, index ascending; NaN counted as -inf) is counted against all T
// similarities held in shared memory as order-preserving integer keys; tokens with rank < N are I_compute. A
// block-wide ballot/prefix scan writes them in ascending index order together
// with the gather/scatter row map r*T + t.
#include <cfloat>

#include "lazymar_internal.cuh"

namespace lm {

template <typename T>
__global__ void __launch_bounds__(256) similarity_kernel(const T* __restrict__ cur, T* __restrict__ cache,
                                                         double* __restrict__ S, long long ntok, int D, int copy) {
  constexpr int V = 16 / sizeof(T);
  pdl_wait();
  pdl_trigger();
  const long long tok = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (tok >= ntok) return;
  const T* a = cur + tok * D;
  T* c = cache + tok * D;
  double dot = 0.0, na = 0.0, nc = 0.0;
  for (int i = lane * V; i < D; i += 32 * V) {
    float av[V], cv[V];
    Vec<T, V>::load(a + i, av);
    Vec<T, V>::load(c + i, cv);
#pragma unroll
    for (int k = 0; k < V; ++k) {
      const double x = (double)av[k], y = (double)cv[k];
      dot = fma(x, y, dot);
      na = fma(x, x, na);
      nc = fma(y, y, nc);
    }
    if (copy) *reinterpret_cast<uint4*>(c + i) = *reinterpret_cast<const uint4*>(a + i);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    dot += __shfl_xor_sync(0xffffffffu, dot, o);
    na += __shfl_xor_sync(0xffffffffu, na, o);
    nc += __shfl_xor_sync(0xffffffffu, nc, o);
  }
  if (lane == 0) {
    const double eps = 1e-8;
    S[tok] = dot / sqrt(fmax(na * nc, eps * eps));
  }
}

// bf16 similarity on the integer pipe (GB300's fp64 rate is a small fraction
// of its integer rate). A bf16 value is M * 2^(E - 134) with an 8-bit integer
// significand M (hidden bit included) and E = max(biased exponent, 1), so a
// product of two is (Ma Mb) * 2^(Ea + Eb - 268) with Ma Mb < 2^16. Each sum
// is taken relative to a base exponent kSpan = 62 - 16 - ceil(log2 D) below
// its largest possible term exponent (from the vectors' largest exponents):
// shifted to the base, every term is an integer below 2^(16 + kSpan) and the
// D-term sum is exact in an int64. Its conversion to double is then the
// correctly rounded exact sum, which equals the fp64 sum of the same products
// whenever that sum is exact. A token with a nonzero term below the base, or
// with an Inf/NaN element, takes the fp64 loop of similarity_kernel instead.
// Each lane keeps its NCH 8-element chunks of both vectors in registers
// (D <= 1280; wider vectors use similarity_kernel).
template <int NCH>
__global__ void __launch_bounds__(256) similarity_int_kernel(const bf16* __restrict__ cur, bf16* __restrict__ cache,
                                                             double* __restrict__ S, long long ntok, int D, int span,
                                                             int copy) {
  pdl_wait();
  pdl_trigger();
  const long long tok = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (tok >= ntok) return;
  const bf16* a = cur + tok * D;
  bf16* c = cache + tok * D;
  uint4 ra[NCH], rc[NCH];
#pragma unroll
  for (int j = 0; j < NCH; ++j) {
    const int i = (lane + 32 * j) * 8;
    if (i < D) {
      ra[j] = *reinterpret_cast<const uint4*>(a + i);
      rc[j] = *reinterpret_cast<const uint4*>(c + i);
    } else {
      ra[j] = make_uint4(0, 0, 0, 0);
      rc[j] = make_uint4(0, 0, 0, 0);
    }
  }
  // largest exponent field of each vector (two bf16 per 32-bit word)
  uint32_t xa = 0, xc = 0;
#pragma unroll
  for (int j = 0; j < NCH; ++j) {
    xa = __vmaxu2(xa, __vmaxu2(ra[j].x & 0x7F807F80u, ra[j].y & 0x7F807F80u));
    xa = __vmaxu2(xa, __vmaxu2(ra[j].z & 0x7F807F80u, ra[j].w & 0x7F807F80u));
    xc = __vmaxu2(xc, __vmaxu2(rc[j].x & 0x7F807F80u, rc[j].y & 0x7F807F80u));
    xc = __vmaxu2(xc, __vmaxu2(rc[j].z & 0x7F807F80u, rc[j].w & 0x7F807F80u));
  }
  int ema = max((int)((xa >> 7) & 0xFFu), (int)((xa >> 23) & 0xFFu));
  int emc = max((int)((xc >> 7) & 0xFFu), (int)((xc >> 23) & 0xFFu));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    ema = max(ema, __shfl_xor_sync(0xffffffffu, ema, o));
    emc = max(emc, __shfl_xor_sync(0xffffffffu, emc, o));
  }
  bool inexact = ema == 255 || emc == 255;  // Inf or NaN present
  ema = max(ema, 1);
  emc = max(emc, 1);
  const int bd = ema + emc - span, ba = 2 * ema - span, bc = 2 * emc - span;
  long long sd = 0, sa = 0, sc = 0;
  if (!inexact) {
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
      const uint32_t wa[4] = {ra[j].x, ra[j].y, ra[j].z, ra[j].w}, wc[4] = {rc[j].x, rc[j].y, rc[j].z, rc[j].w};
#pragma unroll
      for (int h = 0; h < 8; ++h) {
        const uint32_t ya = (wa[h >> 1] >> (16 * (h & 1))) & 0xFFFFu, yc = (wc[h >> 1] >> (16 * (h & 1))) & 0xFFFFu;
        const int ea = (int)((ya >> 7) & 0xFFu), ec = (int)((yc >> 7) & 0xFFu);
        const int Ea = max(ea, 1), Ec = max(ec, 1);
        const uint32_t Ma = (ya & 0x7Fu) | (ea ? 0x80u : 0u), Mc = (yc & 0x7Fu) | (ec ? 0x80u : 0u);
        const uint32_t pd = Ma * Mc, pa = Ma * Ma, pc = Mc * Mc;
        const int hd = Ea + Ec - bd, ha = 2 * Ea - ba, hc = 2 * Ec - bc;
        inexact |= (hd < 0 && pd != 0) | (ha < 0 && pa != 0) | (hc < 0 && pc != 0);
        const long long td = (long long)((unsigned long long)pd << max(hd, 0));
        sd += ((ya ^ yc) & 0x8000u) ? -td : td;
        sa += (long long)((unsigned long long)pa << max(ha, 0));
        sc += (long long)((unsigned long long)pc << max(hc, 0));
      }
    }
  }
  double dot, na, nc;
  if (__any_sync(0xffffffffu, inexact)) {
    // fp64 fallback (the arithmetic of similarity_kernel)
    dot = 0.0, na = 0.0, nc = 0.0;
#pragma unroll 1
    for (int i = lane * 8; i < D; i += 256) {
      float av[8], cv[8];
      Vec<bf16, 8>::load(a + i, av);
      Vec<bf16, 8>::load(c + i, cv);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const double x = (double)av[k], y = (double)cv[k];
        dot = fma(x, y, dot);
        na = fma(x, x, na);
        nc = fma(y, y, nc);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      dot += __shfl_xor_sync(0xffffffffu, dot, o);
      na += __shfl_xor_sync(0xffffffffu, na, o);
      nc += __shfl_xor_sync(0xffffffffu, nc, o);
    }
  } else {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      sd += __shfl_xor_sync(0xffffffffu, sd, o);
      sa += __shfl_xor_sync(0xffffffffu, sa, o);
      sc += __shfl_xor_sync(0xffffffffu, sc, o);
    }
    dot = ldexp((double)sd, bd - 268);
    na = ldexp((double)sa, ba - 268);
    nc = ldexp((double)sc, bc - 268);
  }
  if (copy) {
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
      const int i = (lane + 32 * j) * 8;
      if (i < D) *reinterpret_cast<uint4*>(c + i) = ra[j];
    }
  }
  if (lane == 0) {
    const double eps = 1e-8;
    S[tok] = dot / sqrt(fmax(na * nc, eps * eps));
  }
}

cudaError_t launch_similarity(const Ctx& c, int dtype, const void* cur, void* cache, double* S, int rows, int T, int D,
                              bool copy) {
  const long long ntok = (long long)rows * T;
  if (ntok == 0) return cudaSuccess;
  const unsigned grid = (unsigned)((ntok + 7) / 8);
  if (dtype == LAZYMAR_BF16 && D % 8 == 0 && D <= 1280) {
    int lg = 0;
    while ((1 << lg) < D) ++lg;
    const int span = 62 - 16 - lg;
    const int nch = (D + 255) / 256;
    const bf16* a = static_cast<const bf16*>(cur);
    bf16* k = static_cast<bf16*>(cache);
    const int cp = copy ? 1 : 0;
    if (nch <= 1) return launch_pdl(similarity_int_kernel<1>, dim3(grid), dim3(256), 0, c.stream, a, k, S, ntok, D, span, cp);
    if (nch <= 2) return launch_pdl(similarity_int_kernel<2>, dim3(grid), dim3(256), 0, c.stream, a, k, S, ntok, D, span, cp);
    if (nch <= 3) return launch_pdl(similarity_int_kernel<3>, dim3(grid), dim3(256), 0, c.stream, a, k, S, ntok, D, span, cp);
    if (nch <= 4) return launch_pdl(similarity_int_kernel<4>, dim3(grid), dim3(256), 0, c.stream, a, k, S, ntok, D, span, cp);
    return launch_pdl(similarity_int_kernel<5>, dim3(grid), dim3(256), 0, c.stream, a, k, S, ntok, D, span, cp);
  }
  if (dtype == LAZYMAR_BF16)
    return launch_pdl(similarity_kernel<bf16>, dim3(grid), dim3(256), 0, c.stream, (const bf16*)cur, (bf16*)cache, S,
                      ntok, D, copy ? 1 : 0);
  return launch_pdl(similarity_kernel<float>, dim3(grid), dim3(256), 0, c.stream, (const float*)cur, (float*)cache, S,
                    ntok, D, copy ? 1 : 0);
}

constexpr int kTopkThreads = 512;

// Order-preserving 64-bit key of a similarity: unsigned comparison of keys
// matches numeric comparison of the doubles, with NaN mapped to -inf and -0
// to +0 (so equal similarities give equal keys and the index decides). Keys
// are compared on the integer pipe; GB300's fp64 pipe is far slower.
__device__ __forceinline__ unsigned long long sim_key(double s) {
  if (s != s) s = -HUGE_VAL;
  if (s == 0.0) s = 0.0;
  const unsigned long long u = (unsigned long long)__double_as_longlong(s);
  return (u >> 63) ? ~u : (u | 0x8000000000000000ull);
}

// Selection order (Table 3 strategies): priority descending when given, then
// the rule's key ascending, then token index. Keys: LEAST_SIMILAR (strategy V)
// the order-preserving key of S; MOST_SIMILAR (strategy IV) its complement,
// i.e. S descending (NaN, as -inf, last); RANDOM (strategy III) the caller's
// 32-bit random keys.
__global__ void __launch_bounds__(kTopkThreads) topk_kernel(const double* __restrict__ S, int T, int N,
                                                            int* __restrict__ idx, int* __restrict__ row_map,
                                                            int rule, const uint8_t* __restrict__ prio,
                                                            const uint32_t* __restrict__ rkeys) {
  extern __shared__ unsigned long long sK[];  // T keys, then T priorities, then T flags
  __shared__ int s_wcount[kTopkThreads / 32];
  __shared__ int s_woff[kTopkThreads / 32];
  __shared__ int s_total;
  unsigned char* sP = reinterpret_cast<unsigned char*>(sK + T);
  unsigned char* sel = sP + T;
  const int r = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  pdl_wait();
  pdl_trigger();
  for (int t = tid; t < T; t += kTopkThreads) {
    const size_t i = (size_t)r * T + t;
    unsigned long long k;
    if (rule == LAZYMAR_SELECT_RANDOM) {
      k = rkeys[i];
    } else {
      k = sim_key(S[i]);
      if (rule == LAZYMAR_SELECT_MOST_SIMILAR) k = ~k;
    }
    sK[t] = k;
    sP[t] = prio ? prio[i] : 0;
  }
  __syncthreads();
  // rank of token t under (priority descending, key ascending, index
  // ascending); I_compute = rank < N
  for (int t = tid; t < T; t += kTopkThreads) {
    const unsigned long long kt = sK[t];
    const unsigned pt = sP[t];
    int rank = 0;
    if (prio) {
      for (int u = 0; u < T; ++u) {
        const unsigned long long ku = sK[u];
        const unsigned pu = sP[u];
        rank += (pu > pt) || (pu == pt && ((ku < kt) || (ku == kt && u < t)));
      }
    } else {
      for (int u = 0; u < T; ++u) {
        const unsigned long long ku = sK[u];
        rank += (ku < kt) || (ku == kt && u < t);
      }
    }
    sel[t] = rank < N;
  }
  __syncthreads();
  int base = 0;
  for (int c0 = 0; c0 < T; c0 += kTopkThreads) {
    const int t = c0 + tid;
    const bool f = t < T && sel[t];
    const unsigned bal = __ballot_sync(0xffffffffu, f);
    if (lane == 0) s_wcount[warp] = __popc(bal);
    __syncthreads();
    if (warp == 0) {
      const int v = lane < kTopkThreads / 32 ? s_wcount[lane] : 0;
      int incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += n;
      }
      if (lane < kTopkThreads / 32) s_woff[lane] = incl - v;
      if (lane == 31) s_total = incl;
    }
    __syncthreads();
    if (f) {
      const int pos = base + s_woff[warp] + __popc(bal & ((1u << lane) - 1u));
      idx[(size_t)r * N + pos] = t;
      if (row_map) row_map[(size_t)r * N + pos] = r * T + t;
    }
    base += s_total;
    __syncthreads();
  }
}

cudaError_t launch_topk(const Ctx& c, const double* S, int rows, int T, int N, int* idx, int* row_map, int rule,
                        const uint8_t* prio, const uint32_t* keys) {
  if (rows == 0 || N == 0) return cudaSuccess;
  const size_t smem = (size_t)T * sizeof(unsigned long long) + 2 * (size_t)T;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  return launch_pdl(topk_kernel, dim3(rows), dim3(kTopkThreads), smem, c.stream, S, T, N, idx, row_map, rule, prio,
                    keys);
}

// Caller-chosen I_compute: copied after checking range and strict increase per
// row; a violation is latched as ERR_INDEX and the index is clamped into
// [0, T) so that no later gather or scatter leaves the row.
__global__ void idx_check_kernel(const int* __restrict__ in, int rows, int T, int N, int* __restrict__ idx,
                                 int* __restrict__ row_map, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  const long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x;
  if (i >= (long long)rows * N) return;
  const int r = (int)(i / N), j = (int)(i - (long long)r * N);
  int v = in[i];
  bool ok = v >= 0 && v < T && (j == 0 || in[i - 1] < v);
  if (!ok) {
    atomicOr(err, ERR_INDEX);
    v = v < 0 ? 0 : (v >= T ? T - 1 : v);
  }
  idx[i] = v;
  row_map[i] = r * T + v;
}

cudaError_t launch_idx_check(const Ctx& c, const int* in, int rows, int T, int N, int* idx, int* row_map) {
  const long long n = (long long)rows * N;
  if (n == 0) return cudaSuccess;
  return launch_pdl(idx_check_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, c.stream, in, rows, T, N, idx,
                    row_map, c.err);
}

// ---------------------------------------------------------------------------
// Selection without device allocation
// ---------------------------------------------------------------------------
// Some callers may not allocate device memory once they are running: a
// serving loop that reserves its whole memory budget at start-up and must not
// grow it, or a plug-in whose host framework owns the device allocator and
// forbids direct cudaMalloc. lazymar_select_tokens_noalloc serves them: its
// similarity scratch is this fixed, module-level array, which every GPU that
// loads the library holds until the process exits (8 bytes per token,
// 2 MiB in total).
static __device__ __align__(256) double g_select_scratch[LAZYMAR_SELECT_NOALLOC_MAX_TOKENS];

constexpr int kMaxDevices = 64;

// On the host, the name g_select_scratch denotes a host-side stand-in, not
// device memory: handing it to a kernel would fault or, where the GPU can
// reach host memory, silently use the wrong memory. The device address is
// looked up on every call, with the caller's device current: the lookup
// allocates nothing and costs little, and a cached address would go stale
// when a device reset reloads the module at another address.
static cudaError_t select_scratch(double** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_select_scratch);
  if (e != cudaSuccess) return e;
  *out = static_cast<double*>(p);
  return cudaSuccess;
}

static bool noalloc_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (!p || cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

}  // namespace lm

extern "C" lazymar_status lazymar_select_tokens_noalloc(int dtype, const void* v_cur, void* v_cache, int rows, int T,
                                                        int D, int n_compute, int32_t* idx_out, void* stream) {
  using namespace lm;
  if (dtype != LAZYMAR_F32 && dtype != LAZYMAR_BF16) return report_error(LAZYMAR_ERR_INVALID_ARG, "dtype");
  if (rows < 0 || T < 1 || T > 16384 || D < 8 || D % 8 != 0 || n_compute < 0 || n_compute > T)
    return report_error(LAZYMAR_ERR_INVALID_ARG,
                        "rows >= 0, 1 <= T <= 16384, D % 8 == 0, 0 <= n_compute <= T required");
  if ((long long)rows * T > LAZYMAR_SELECT_NOALLOC_MAX_TOKENS)
    return report_error(LAZYMAR_ERR_INVALID_ARG,
                        "rows * T exceeds LAZYMAR_SELECT_NOALLOC_MAX_TOKENS (262144), the size of the fixed "
                        "scratch; use lazymar_select_tokens");
  if (rows == 0) return LAZYMAR_OK;
  if (!noalloc_device_ptr(v_cur) || !noalloc_device_ptr(v_cache) || (n_compute > 0 && !noalloc_device_ptr(idx_out)))
    return report_error(LAZYMAR_ERR_INVALID_ARG, "v_cur, v_cache and idx_out must be device pointers");
  if ((reinterpret_cast<uintptr_t>(v_cur) | reinterpret_cast<uintptr_t>(v_cache)) & 15u)
    return report_error(LAZYMAR_ERR_INVALID_ARG, "16-byte alignment required");
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return report_error(LAZYMAR_ERR_CUDA, "cudaGetDevice failed or device index out of range");
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return report_error(LAZYMAR_ERR_CUDA, "cudaDeviceGetAttribute failed");
  double* S = nullptr;
  if (select_scratch(&S) != cudaSuccess)
    return report_error(LAZYMAR_ERR_CUDA, "cudaGetSymbolAddress of the selection scratch failed");
  // Every S entry the top-N reads is written by the similarity pass of the
  // same call first, so the scratch needs no clearing between calls.
  const Ctx c{static_cast<cudaStream_t>(stream), nullptr, sms};
  cudaError_t e = launch_similarity(c, dtype, v_cur, v_cache, S, rows, T, D, true);
  if (e == cudaSuccess) e = launch_topk(c, S, rows, T, n_compute, idx_out, nullptr);
  if (e != cudaSuccess) return report_error(LAZYMAR_ERR_CUDA, cudaGetErrorString(e));
  return LAZYMAR_OK;
}

namespace lm {

// ---------------------------------------------------------------------------
// Bounded-wait diagnostic
// ---------------------------------------------------------------------------
// Every pipelined kernel waits on mbarriers with a time limit: on expiry it
// raises its abort flag and ERR_TIMEOUT in the device error word, stops, and
// returns normally, so the context stays usable and the host learns of the
// failure from lazymar_sync / lazymar_device_check. This kernel drives that
// path on purpose: its barrier expects one arrival that never comes.
__global__ void stuck_wait_kernel(unsigned* err, unsigned long long limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  mbar_wait_limit(&bar, 0, &abort_flag, err, limit_ns);
}

cudaError_t launch_stuck_wait(const Ctx& c, uint64_t limit_ns) {
  stuck_wait_kernel<<<1, 32, 0, c.stream>>>(c.err, (unsigned long long)limit_ns);
  return cudaGetLastError();
}

}  // namespace lm
