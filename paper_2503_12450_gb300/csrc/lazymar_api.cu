// C ABI of liblazymar: handle life cycle, the full and cached decoding steps
// (kernel orchestration on the caller's stream), the component entry points and
// host-side bookkeeping (schedule, device error word, per-kernel statistics).
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>
#include <map>
#include <tuple>

#include "lazymar_internal.cuh"

using namespace lm;

namespace lm {
bool layernorm_width_ok(int D);
}

// ---------------------------------------------------------------------------
// Errors
// ---------------------------------------------------------------------------
static thread_local std::string g_last_error;

static lazymar_status fail(lazymar_status s, const std::string& msg) {
  g_last_error = msg;
  return s;
}
namespace lm {
lazymar_status report_error(lazymar_status s, const char* msg) { return fail(s, msg); }
}  // namespace lm

static lazymar_status cuda_fail(cudaError_t e, const char* what) {
  return fail(LAZYMAR_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}
#define LM_CUDA(expr)                                  \
  do {                                                 \
    cudaError_t e_ = (expr);                           \
    if (e_ != cudaSuccess) return cuda_fail(e_, #expr); \
  } while (0)
#define LM_TRY(expr)                      \
  do {                                    \
    lazymar_status s_ = (expr);           \
    if (s_ != LAZYMAR_OK) return s_;      \
  } while (0)

// Device error word of the component entry points (one per device, in this
// module's static device memory; handles use their own word).
static __device__ unsigned g_component_err;

static lazymar_status component_ctx(void* stream, Ctx* c) {
  int dev = 0;
  LM_CUDA(cudaGetDevice(&dev));
  int sms = 0;
  LM_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  void* p = nullptr;
  LM_CUDA(cudaGetSymbolAddress(&p, g_component_err));
  c->stream = static_cast<cudaStream_t>(stream);
  c->err = static_cast<unsigned*>(p);
  c->num_sms = sms;
  return LAZYMAR_OK;
}

static bool is_device_ptr(const void* p) {
  if (!p) return false;
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}
static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

static lazymar_status read_error_word(unsigned* word, cudaStream_t stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  unsigned v = 0;
  LM_CUDA(cudaMemcpy(&v, word, sizeof(unsigned), cudaMemcpyDeviceToHost));
  if (v) LM_CUDA(cudaMemset(word, 0, sizeof(unsigned)));
  if (v & ERR_TIMEOUT) return fail(LAZYMAR_ERR_TIMEOUT, "a bounded device wait expired");
  if (v & ERR_INDEX) return fail(LAZYMAR_ERR_DEVICE, "a token index was out of range or not increasing");
  if (v & ERR_LABEL) return fail(LAZYMAR_ERR_DEVICE, "a class label was out of range");
  return LAZYMAR_OK;
}

// ---------------------------------------------------------------------------
// Handle
// ---------------------------------------------------------------------------
struct BlockDev {
  void *ln1_g, *ln1_b, *w_qkv, *b_qkv, *w_o, *b_o, *ln2_g, *ln2_b, *w1, *b1, *w2, *b2;
};

struct lazymar_handle {
  lazymar_config cfg{};
  int dev = 0, num_sms = 0, T = 0, D = 0, H4 = 0, dh = 0, L = 0, s = 0, max_rows = 0;
  size_t es = 0;
  uint8_t* arena = nullptr;
  size_t arena_bytes = 0;
  // weights (dtype)
  void *pos = nullptr, *cls = nullptr, *memb = nullptr, *ew = nullptr, *eb = nullptr, *lnf_g = nullptr,
       *lnf_b = nullptr;
  std::vector<BlockDev> blk;
  // token cache: keys/values of blocks s..L-1; selection reference; output
  // features of the image tokens; condition cache
  std::vector<void*> Kc, Vc;
  // qkv_e4m3: E4M3 copies of W_qkv of blocks s..L-1 with per-row scales, and
  // the E4M3 LN1 output of the recomputed tokens
  std::vector<uint8_t*> wq8;
  std::vector<float*> wsc;
  uint8_t* A8 = nullptr;
  void *ref = nullptr, *zc = nullptr, *delta = nullptr;
  // scratch
  float *H = nullptr, *Hc = nullptr;
  void *A = nullptr, *Q = nullptr, *Ks = nullptr, *Vs = nullptr, *O = nullptr, *U = nullptr, *Fs = nullptr;
  double* S = nullptr;
  int *idx = nullptr, *row_map = nullptr;
  // staging of host inputs/outputs
  float* st_lat = nullptr;
  uint8_t* st_mask = nullptr;
  int *st_labels = nullptr, *st_idx_in = nullptr, *st_idx_out = nullptr;
  uint8_t* st_prio = nullptr;     // [rows, T] selection priority classes
  uint32_t* st_keys = nullptr;    // [rows, T] selection random keys
  void *st_z = nullptr, *st_g = nullptr;
  unsigned* err = nullptr;
  bool primed = false;
  int last_batch = 0;
  // statistics
  lazymar_stats stats{};
  bool profiling = false;
  struct Ev {
    cudaEvent_t a, b;
    int cls;
  };
  std::vector<Ev> evs;
  size_t ev_used = 0;
  // CUDA graphs of step bodies, keyed by (kind, batch, N, cond reuse, caller indices)
  struct GraphKey {
    int kind, B, N, reuse, idx, sel;  // sel: bit 0 priority given, bit 1 keys given
    bool operator<(const GraphKey& o) const {
      return std::tie(kind, B, N, reuse, idx, sel) < std::tie(o.kind, o.B, o.N, o.reuse, o.idx, o.sel);
    }
  };
  struct GraphEntry {
    cudaGraphExec_t exec = nullptr;
    int eager_runs = 0;
    lazymar_stats delta{};
    std::vector<Ev> evs;   // profiled graphs: the event pairs recorded by its nodes
    bool pending = false;  // profiled graphs: replayed, events not read yet
  };
  std::map<GraphKey, GraphEntry> graphs;
  // Profiled step bodies: captured with an event record around every launch,
  // so that per-kernel times are device times and exclude the host's launch
  // submission (eagerly issued launches can leave the GPU idle between the
  // events of a short kernel).
  std::map<GraphKey, GraphEntry> pgraphs;
  bool use_graphs = true;
  cudaStream_t gstream = nullptr;  // capture stream (graphs replay on the caller's stream)
};

namespace {

struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    int cur = 0;
    if (cudaGetDevice(&cur) == cudaSuccess && cur != dev) {
      prev = cur;
      cudaSetDevice(dev);
    }
  }
  ~DeviceGuard() {
    if (prev >= 0) cudaSetDevice(prev);
  }
};

// Records (when profiling) and counts one kernel launch.
template <class F>
lazymar_status launch(lazymar_handle* h, int cls, double flops, double bytes, cudaStream_t st, const char* what,
                      F&& f) {
  NvtxRange range(what);
  lazymar_handle::Ev* ev = nullptr;
  unsigned ev_flags = cudaEventRecordDefault;
  if (h && h->profiling) {
    if (h->ev_used == h->evs.size()) {
      lazymar_handle::Ev e{};
      LM_CUDA(cudaEventCreate(&e.a));
      LM_CUDA(cudaEventCreate(&e.b));
      h->evs.push_back(e);
    }
    ev = &h->evs[h->ev_used++];
    ev->cls = cls;
    // under stream capture the records must be external to become
    // event-record nodes of the graph (a plain record would only mark a
    // capture dependency)
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    LM_CUDA(cudaStreamIsCapturing(st, &cs));
    ev_flags = cs == cudaStreamCaptureStatusActive ? cudaEventRecordExternal : cudaEventRecordDefault;
    LM_CUDA(cudaEventRecordWithFlags(ev->a, st, ev_flags));
  }
  cudaError_t e = f();
  if (ev) {
    const cudaError_t eb = cudaEventRecordWithFlags(ev->b, st, ev_flags);
    if (eb != cudaSuccess) return cuda_fail(eb, "event record after a launch");
  }
  if (e != cudaSuccess) return cuda_fail(e, what);
  if (h) {
    lazymar_kernel_stats& k = h->stats.k[cls];
    k.launches += 1;
    k.flops += flops;
    k.bytes += bytes;
  }
  return LAZYMAR_OK;
}

struct Bump {
  size_t off = 0;
  size_t take(size_t bytes) {
    const size_t o = off;
    off += (bytes + 255) & ~size_t(255);
    return o;
  }
};

uint16_t f32_to_bf16(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7fffffffu) > 0x7f800000u) return 0x7fc0;
  u += 0x7fffu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

// Copies n fp32 values (host or device pointer) into dst converted to dtype.
lazymar_status upload(void* dst, const float* src, size_t n, int dtype) {
  if (!src) return fail(LAZYMAR_ERR_INVALID_ARG, "a weight pointer is NULL");
  std::vector<float> tmp(n);
  LM_CUDA(cudaMemcpy(tmp.data(), src, n * sizeof(float), cudaMemcpyDefault));
  if (dtype == LAZYMAR_F32) {
    LM_CUDA(cudaMemcpy(dst, tmp.data(), n * sizeof(float), cudaMemcpyHostToDevice));
  } else {
    std::vector<uint16_t> b(n);
    for (size_t i = 0; i < n; ++i) b[i] = f32_to_bf16(tmp[i]);
    LM_CUDA(cudaMemcpy(dst, b.data(), n * sizeof(uint16_t), cudaMemcpyHostToDevice));
  }
  return LAZYMAR_OK;
}

lazymar_status check_config(const lazymar_config* c) {
  if (c->depth < 1 || c->heads < 1 || c->mlp_ratio < 1 || c->n_buffer < 0 || c->n_img < 1 || c->n_classes < 1 ||
      c->max_batch < 1 || !(c->ln_eps > 0.f))
    return fail(LAZYMAR_ERR_INVALID_ARG, "config: non-positive size");
  if (c->dtype != LAZYMAR_F32 && c->dtype != LAZYMAR_BF16) return fail(LAZYMAR_ERR_INVALID_ARG, "config: dtype");
  if (c->criterion != LAZYMAR_CRITERION_VALUE && c->criterion != LAZYMAR_CRITERION_FEATURE)
    return fail(LAZYMAR_ERR_INVALID_ARG, "config: criterion");
  if (c->select_rule < LAZYMAR_SELECT_LEAST_SIMILAR || c->select_rule > LAZYMAR_SELECT_RANDOM)
    return fail(LAZYMAR_ERR_INVALID_ARG, "config: select_rule");
  if (c->sel_layers < 1 || c->sel_layers > c->depth)
    return fail(LAZYMAR_ERR_INVALID_ARG, "config: 1 <= sel_layers <= depth required");
  if (c->token_dim < 1 || c->token_dim > 64) return fail(LAZYMAR_ERR_UNSUPPORTED, "config: token_dim must be 1..64");
  if (c->qkv_e4m3 != 0 && c->qkv_e4m3 != 1) return fail(LAZYMAR_ERR_INVALID_ARG, "config: qkv_e4m3 must be 0 or 1");
  if (c->qkv_e4m3 && (c->dtype != LAZYMAR_BF16 || c->width % 128 != 0))
    return fail(LAZYMAR_ERR_UNSUPPORTED, "config: qkv_e4m3 needs bf16 and width % 128 == 0");
  if (c->width % c->heads != 0) return fail(LAZYMAR_ERR_INVALID_ARG, "config: heads must divide width");
  if (!layernorm_width_ok(c->width))
    return fail(LAZYMAR_ERR_UNSUPPORTED, "config: width must be 128 * {1,2,4,6,8,10,12,16}");
  const char* why = "";
  if (!attention_supported(c->dtype, c->heads, c->width / c->heads, &why)) return fail(LAZYMAR_ERR_UNSUPPORTED, why);
  const long long T = (long long)c->n_buffer + c->n_img;
  if (T > 16384) return fail(LAZYMAR_ERR_UNSUPPORTED, "config: at most 16384 tokens per sequence");
  if ((long long)2 * c->max_batch * T * c->width * c->mlp_ratio >= (1ll << 31))
    return fail(LAZYMAR_ERR_UNSUPPORTED, "config: max_batch too large for 32-bit row indexing");
  return LAZYMAR_OK;
}

}  // namespace

extern "C" lazymar_status lazymar_create(const lazymar_config* cfg, const lazymar_weights* w, lazymar_handle** out) {
  if (!cfg || !w || !out || !w->blocks) return fail(LAZYMAR_ERR_INVALID_ARG, "NULL argument");
  *out = nullptr;
  LM_TRY(check_config(cfg));
  auto* h = new lazymar_handle();
  h->cfg = *cfg;
  h->T = cfg->n_buffer + cfg->n_img;
  h->D = cfg->width;
  h->H4 = cfg->width * cfg->mlp_ratio;
  h->dh = cfg->width / cfg->heads;
  h->L = cfg->depth;
  h->s = cfg->sel_layers;
  h->max_rows = 2 * cfg->max_batch;
  h->es = cfg->dtype == LAZYMAR_BF16 ? 2 : 4;
  auto destroy = [&](lazymar_status s) {
    lazymar_destroy(h);
    return s;
  };
  cudaError_t e = cudaGetDevice(&h->dev);
  if (e != cudaSuccess) return destroy(cuda_fail(e, "cudaGetDevice"));
  e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->dev);
  if (e != cudaSuccess) return destroy(cuda_fail(e, "cudaDeviceGetAttribute"));

  const size_t D = h->D, T = h->T, H4 = h->H4, es = h->es, R = h->max_rows, Bm = cfg->max_batch;
  const size_t rowsT = R * T;
  Bump b;
  // weights
  const size_t o_pos = b.take(T * D * es), o_cls = b.take((size_t)cfg->n_classes * D * es), o_memb = b.take(D * es),
               o_ew = b.take(D * cfg->token_dim * es), o_eb = b.take(D * es), o_lnfg = b.take(D * es),
               o_lnfb = b.take(D * es);
  std::vector<size_t> o_blk(h->L);
  const size_t blk_bytes = (2 * D + 3 * D * D + 3 * D + D * D + D + 2 * D + H4 * D + H4 + D * H4 + D) * es;
  for (int l = 0; l < h->L; ++l) o_blk[l] = b.take(blk_bytes);
  // caches
  std::vector<size_t> o_k(h->L, 0), o_v(h->L, 0);
  for (int l = h->s; l < h->L; ++l) {
    o_k[l] = b.take(rowsT * D * es);
    o_v[l] = b.take(rowsT * D * es);
  }
  std::vector<size_t> o_wq8(h->L, 0), o_wsc(h->L, 0);
  size_t o_A8 = 0;
  if (cfg->qkv_e4m3) {
    for (int l = h->s; l < h->L; ++l) {
      o_wq8[l] = b.take(3 * D * D);
      o_wsc[l] = b.take(3 * D * 4);
    }
    o_A8 = b.take(rowsT * D);
  }
  const size_t o_ref = b.take(rowsT * D * es), o_zc = b.take(R * cfg->n_img * D * es),
               o_delta = b.take(Bm * cfg->n_img * D * es);
  // scratch
  const size_t o_H = b.take(rowsT * D * 4), o_Hc = b.take(rowsT * D * 4), o_A = b.take(rowsT * D * es),
               o_Q = b.take(rowsT * D * es), o_Ks = b.take(rowsT * D * es), o_Vs = b.take(rowsT * D * es),
               o_O = b.take(rowsT * D * es), o_U = b.take(rowsT * H4 * es),
               o_Fs = b.take(cfg->criterion == LAZYMAR_CRITERION_FEATURE ? rowsT * D * es : 0),
               o_S = b.take(rowsT * 8), o_idx = b.take(rowsT * 4), o_map = b.take(rowsT * 4);
  // staging
  const size_t o_lat = b.take(Bm * cfg->n_img * cfg->token_dim * 4), o_mask = b.take(Bm * cfg->n_img),
               o_lab = b.take(Bm * 4), o_iin = b.take(rowsT * 4), o_iout = b.take(rowsT * 4),
               o_prio = b.take(rowsT), o_keys = b.take(rowsT * 4),
               o_stz = b.take(R * cfg->n_img * D * es), o_stg = b.take(Bm * cfg->n_img * D * es),
               o_err = b.take(sizeof(unsigned));
  h->arena_bytes = b.off;
  e = cudaMalloc(&h->arena, h->arena_bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    h->arena = nullptr;
    char msg[160];
    std::snprintf(msg, sizeof msg, "cudaMalloc of %.2f GB failed: %s", h->arena_bytes / 1e9, cudaGetErrorString(e));
    return destroy(fail(LAZYMAR_ERR_OOM, msg));
  }
  uint8_t* a = h->arena;
  h->pos = a + o_pos; h->cls = a + o_cls; h->memb = a + o_memb; h->ew = a + o_ew; h->eb = a + o_eb;
  h->lnf_g = a + o_lnfg; h->lnf_b = a + o_lnfb;
  h->blk.resize(h->L);
  for (int l = 0; l < h->L; ++l) {
    uint8_t* p = a + o_blk[l];
    BlockDev& bd = h->blk[l];
    auto nxt = [&](size_t n) { void* r = p; p += n * es; return r; };
    bd.ln1_g = nxt(D); bd.ln1_b = nxt(D); bd.w_qkv = nxt(3 * D * D); bd.b_qkv = nxt(3 * D);
    bd.w_o = nxt(D * D); bd.b_o = nxt(D); bd.ln2_g = nxt(D); bd.ln2_b = nxt(D);
    bd.w1 = nxt(H4 * D); bd.b1 = nxt(H4); bd.w2 = nxt(D * H4); bd.b2 = nxt(D);
  }
  h->Kc.assign(h->L, nullptr);
  h->Vc.assign(h->L, nullptr);
  for (int l = h->s; l < h->L; ++l) {
    h->Kc[l] = a + o_k[l];
    h->Vc[l] = a + o_v[l];
  }
  h->ref = a + o_ref; h->zc = a + o_zc; h->delta = a + o_delta;
  h->wq8.assign(h->L, nullptr);
  h->wsc.assign(h->L, nullptr);
  if (cfg->qkv_e4m3) {
    for (int l = h->s; l < h->L; ++l) {
      h->wq8[l] = a + o_wq8[l];
      h->wsc[l] = reinterpret_cast<float*>(a + o_wsc[l]);
    }
    h->A8 = a + o_A8;
  }
  h->H = reinterpret_cast<float*>(a + o_H); h->Hc = reinterpret_cast<float*>(a + o_Hc);
  h->A = a + o_A; h->Q = a + o_Q; h->Ks = a + o_Ks; h->Vs = a + o_Vs; h->O = a + o_O; h->U = a + o_U;
  h->Fs = a + o_Fs;
  h->S = reinterpret_cast<double*>(a + o_S);
  h->idx = reinterpret_cast<int*>(a + o_idx); h->row_map = reinterpret_cast<int*>(a + o_map);
  h->st_lat = reinterpret_cast<float*>(a + o_lat); h->st_mask = a + o_mask;
  h->st_labels = reinterpret_cast<int*>(a + o_lab);
  h->st_idx_in = reinterpret_cast<int*>(a + o_iin); h->st_idx_out = reinterpret_cast<int*>(a + o_iout);
  h->st_prio = a + o_prio; h->st_keys = reinterpret_cast<uint32_t*>(a + o_keys);
  h->st_z = a + o_stz; h->st_g = a + o_stg;
  h->err = reinterpret_cast<unsigned*>(a + o_err);

  e = cudaMemset(h->arena, 0, h->arena_bytes);
  if (e != cudaSuccess) return destroy(cuda_fail(e, "cudaMemset"));
  if ((e = cudaStreamCreateWithFlags(&h->gstream, cudaStreamNonBlocking)) != cudaSuccess)
    return destroy(cuda_fail(e, "stream creation"));
  lazymar_status st;
  const int dt = cfg->dtype;
  if ((st = upload(h->pos, w->pos_emb, T * D, dt)) || (st = upload(h->cls, w->class_emb, (size_t)cfg->n_classes * D, dt)) ||
      (st = upload(h->memb, w->mask_emb, D, dt)) || (st = upload(h->ew, w->embed_w, D * cfg->token_dim, dt)) ||
      (st = upload(h->eb, w->embed_b, D, dt)) || (st = upload(h->lnf_g, w->lnf_g, D, dt)) ||
      (st = upload(h->lnf_b, w->lnf_b, D, dt)))
    return destroy(st);
  for (int l = 0; l < h->L; ++l) {
    const lazymar_block_weights& s = w->blocks[l];
    BlockDev& bd = h->blk[l];
    if ((st = upload(bd.ln1_g, s.ln1_g, D, dt)) || (st = upload(bd.ln1_b, s.ln1_b, D, dt)) ||
        (st = upload(bd.w_qkv, s.w_qkv, 3 * D * D, dt)) || (st = upload(bd.b_qkv, s.b_qkv, 3 * D, dt)) ||
        (st = upload(bd.w_o, s.w_o, D * D, dt)) || (st = upload(bd.b_o, s.b_o, D, dt)) ||
        (st = upload(bd.ln2_g, s.ln2_g, D, dt)) || (st = upload(bd.ln2_b, s.ln2_b, D, dt)) ||
        (st = upload(bd.w1, s.w1, H4 * D, dt)) || (st = upload(bd.b1, s.b1, H4, dt)) ||
        (st = upload(bd.w2, s.w2, D * H4, dt)) || (st = upload(bd.b2, s.b2, D, dt)))
      return destroy(st);
  }
  if (cfg->qkv_e4m3) {
    const Ctx qc{h->gstream, h->err, h->num_sms};
    for (int l = h->s; l < h->L; ++l) {
      e = launch_quantize_e4m3(qc, h->blk[l].w_qkv, 3 * (int)D, (int)D, h->wq8[l], h->wsc[l]);
      if (e != cudaSuccess) return destroy(cuda_fail(e, "E4M3 weight quantization"));
    }
    e = cudaStreamSynchronize(h->gstream);
    if (e != cudaSuccess) return destroy(cuda_fail(e, "E4M3 weight quantization"));
  }
  *out = h;
  return LAZYMAR_OK;
}

extern "C" void lazymar_destroy(lazymar_handle* h) {
  if (!h) return;
  DeviceGuard g(h->dev);
  for (auto& kv : h->graphs)
    if (kv.second.exec) cudaGraphExecDestroy(kv.second.exec);
  for (auto& kv : h->pgraphs) {
    if (kv.second.exec) cudaGraphExecDestroy(kv.second.exec);
    for (auto& e : kv.second.evs) {
      cudaEventDestroy(e.a);
      cudaEventDestroy(e.b);
    }
  }
  if (h->gstream) cudaStreamDestroy(h->gstream);
  for (auto& e : h->evs) {
    cudaEventDestroy(e.a);
    cudaEventDestroy(e.b);
  }
  if (h->arena) cudaFree(h->arena);
  delete h;
}

// ---------------------------------------------------------------------------
// Steps
// ---------------------------------------------------------------------------
namespace {

// The address at which the device reads `p`: p itself for device or managed
// memory, the mapping of page-locked host memory, else nullptr (pageable
// host memory, which only a copy can read).
const void* device_view(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) return p;
  if (a.type == cudaMemoryTypeHost) return a.devicePointer;
  return nullptr;
}

// Step inputs always go through the handle's staging buffers, so the device
// work of a step reads fixed addresses and can be replayed from a CUDA graph.
// Inputs the device can address are gathered by one copy kernel (one launch
// on the compute stream instead of a copy-engine operation per input);
// pageable host inputs take a copy each.
struct Stager {
  lazymar_handle* h;
  cudaStream_t st;
  CopyList L{};
  lazymar_status add(void* dst, const void* src, size_t bytes) {
    if (bytes == 0) return LAZYMAR_OK;
    const void* d = device_view(src);
    if (d && L.n < kMaxCopySegs) {
      L.src[L.n] = d;
      L.dst[L.n] = dst;
      L.bytes[L.n] = bytes;
      ++L.n;
      return LAZYMAR_OK;
    }
    LM_CUDA(cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDefault, st));
    return LAZYMAR_OK;
  }
  lazymar_status flush(const Ctx& c) {
    if (L.n == 0) return LAZYMAR_OK;
    return launch(h, LAZYMAR_K_OTHER, 0, 0, c.stream, "stage inputs", [&] { return launch_copy_list(c, L); });
  }
};

lazymar_status stage_inputs(Stager& sg, const lazymar_step_in* in) {
  lazymar_handle* h = sg.h;
  const int B = in->batch;
  const size_t nl = (size_t)B * h->cfg.n_img * h->cfg.token_dim;
  const size_t nm = (size_t)B * h->cfg.n_img;
  LM_TRY(sg.add(h->st_lat, in->latents, nl * 4));
  LM_TRY(sg.add(h->st_mask, in->mask, nm));
  LM_TRY(sg.add(h->st_labels, in->labels, (size_t)B * 4));
  return LAZYMAR_OK;
}

lazymar_status check_step_in(lazymar_handle* h, const lazymar_step_in* in) {
  if (!h || !in) return fail(LAZYMAR_ERR_INVALID_ARG, "NULL handle or inputs");
  if (in->batch < 1 || in->batch > h->cfg.max_batch) return fail(LAZYMAR_ERR_INVALID_ARG, "batch outside 1..max_batch");
  if (!in->latents || !in->mask || !in->labels) return fail(LAZYMAR_ERR_INVALID_ARG, "NULL input tensor");
  return LAZYMAR_OK;
}

double gemm_bytes(const lazymar_handle* h, int M, int N, int K, int mode) {
  const double es = (double)h->es;
  const double out = mode == LAZYMAR_EPI_RESIDUAL ? 8.0 * M * N : es * M * N;
  return es * ((double)M * K + (double)N * K) + out;
}

lazymar_status gemm(lazymar_handle* h, const Ctx& c, const void* A, const void* W, int M, int N, int K,
                    const GemmEpi& e, int dtype = -1) {
  if (M == 0) return LAZYMAR_OK;
  const int dt = dtype < 0 ? h->cfg.dtype : dtype;
  double bytes = gemm_bytes(h, M, N, K, e.mode);
  if (dt == LAZYMAR_E4M3) bytes -= (double)h->es * ((double)M * K + (double)N * K) / 2.0;  // 1-byte operands
  const long long k0 = gemm_kernels_issued();
  LM_TRY(launch(h, LAZYMAR_K_GEMM, 2.0 * M * N * K, bytes, c.stream, "gemm",
                [&] { return launch_gemm(c, dt, A, W, M, N, K, e, 0); }));
  // the statistics count kernels: a split GEMM adds its second launch
  const long long extra = gemm_kernels_issued() - k0 - 1;
  if (extra > 0) h->stats.k[LAZYMAR_K_GEMM].launches += extra;
  return LAZYMAR_OK;
}

lazymar_status layernorm(lazymar_handle* h, const Ctx& c, const float* x, const int* map, const void* g, const void* b,
                         void* y, float* copy, int M, int dtype = -1) {
  if (M == 0) return LAZYMAR_OK;
  const int dt = dtype < 0 ? h->cfg.dtype : dtype;
  const double bytes = (double)M * h->D * (4.0 + (dt == LAZYMAR_E4M3 ? 1.0 : h->es) + (copy ? 4.0 : 0.0));
  return launch(h, LAZYMAR_K_LAYERNORM, 0, bytes, c.stream, "layernorm", [&] {
    return launch_layernorm(c, dt, x, map, g, b, y, copy, M, h->D, h->cfg.ln_eps);
  });
}

lazymar_status attention(lazymar_handle* h, const Ctx& c, const void* k, const void* v, int rows, int n_q,
                         const void* q = nullptr) {
  if (rows == 0 || n_q == 0) return LAZYMAR_OK;
  const double flops = 4.0 * rows * n_q * (double)h->T * h->D;
  const double bytes = (double)h->es * h->D * (2.0 * rows * n_q + 2.0 * rows * h->T);
  return launch(h, LAZYMAR_K_ATTENTION, flops, bytes, c.stream, "attention", [&] {
    return launch_attention(c, h->cfg.dtype, q ? q : h->Q, k, v, h->O, rows, n_q, h->T, h->cfg.heads, h->dh);
  });
}

// One block over every token of `rows` rows (residual stream h->H).
lazymar_status layer_full(lazymar_handle* h, const Ctx& c, int l, int rows, void* kdst, void* vdst) {
  const BlockDev& b = h->blk[l];
  const int M = rows * h->T, D = h->D;
  LM_TRY(layernorm(h, c, h->H, nullptr, b.ln1_g, b.ln1_b, h->A, nullptr, M));
  LM_TRY(gemm(h, c, h->A, b.w_qkv, M, 3 * D, D, GemmEpi{LAZYMAR_EPI_QKV, b.b_qkv, h->Q, D, kdst, vdst, nullptr, D}));
  LM_TRY(attention(h, c, kdst, vdst, rows, h->T));
  LM_TRY(gemm(h, c, h->O, b.w_o, M, D, D, GemmEpi{LAZYMAR_EPI_RESIDUAL, b.b_o, h->H, D, nullptr, nullptr, nullptr, D}));
  LM_TRY(layernorm(h, c, h->H, nullptr, b.ln2_g, b.ln2_b, h->A, nullptr, M));
  LM_TRY(gemm(h, c, h->A, b.w1, M, h->H4, D, GemmEpi{LAZYMAR_EPI_GELU, b.b1, h->U, h->H4, nullptr, nullptr, nullptr, D}));
  LM_TRY(gemm(h, c, h->U, b.w2, M, D, h->H4, GemmEpi{LAZYMAR_EPI_RESIDUAL, b.b2, h->H, D, nullptr, nullptr, nullptr, D}));
  return LAZYMAR_OK;
}

// One block under the token cache (Eq. 9): the N selected tokens of each row
// (compact residual stream h->Hc, gathered from h->H on the first cached
// block); their K/V are scattered into the cache rows row_map, their queries
// attend over all T cached keys/values.
lazymar_status layer_cached(lazymar_handle* h, const Ctx& c, int l, int rows, int N, bool first) {
  const BlockDev& b = h->blk[l];
  const int M = rows * N, D = h->D;
  if (h->cfg.qkv_e4m3) {
    // LN1 to E4M3, then the 8-bit Q/K/V projection with per-channel scales
    const int e8 = LAZYMAR_E4M3;
    if (first)
      LM_TRY(layernorm(h, c, h->H, h->row_map, b.ln1_g, b.ln1_b, h->A8, h->Hc, M, e8));
    else
      LM_TRY(layernorm(h, c, h->Hc, nullptr, b.ln1_g, b.ln1_b, h->A8, nullptr, M, e8));
    GemmEpi qe{LAZYMAR_EPI_QKV, b.b_qkv, h->Q, D, h->Kc[l], h->Vc[l], h->row_map, D};
    qe.wscale = h->wsc[l];
    LM_TRY(gemm(h, c, h->A8, h->wq8[l], M, 3 * D, D, qe, e8));
  } else {
    if (first)
      LM_TRY(layernorm(h, c, h->H, h->row_map, b.ln1_g, b.ln1_b, h->A, h->Hc, M));
    else
      LM_TRY(layernorm(h, c, h->Hc, nullptr, b.ln1_g, b.ln1_b, h->A, nullptr, M));
    LM_TRY(gemm(h, c, h->A, b.w_qkv, M, 3 * D, D,
                GemmEpi{LAZYMAR_EPI_QKV, b.b_qkv, h->Q, D, h->Kc[l], h->Vc[l], h->row_map, D}));
  }
  LM_TRY(attention(h, c, h->Kc[l], h->Vc[l], rows, N));
  LM_TRY(gemm(h, c, h->O, b.w_o, M, D, D, GemmEpi{LAZYMAR_EPI_RESIDUAL, b.b_o, h->Hc, D, nullptr, nullptr, nullptr, D}));
  LM_TRY(layernorm(h, c, h->Hc, nullptr, b.ln2_g, b.ln2_b, h->A, nullptr, M));
  LM_TRY(gemm(h, c, h->A, b.w1, M, h->H4, D, GemmEpi{LAZYMAR_EPI_GELU, b.b1, h->U, h->H4, nullptr, nullptr, nullptr, D}));
  LM_TRY(gemm(h, c, h->U, b.w2, M, D, h->H4, GemmEpi{LAZYMAR_EPI_RESIDUAL, b.b2, h->Hc, D, nullptr, nullptr, nullptr, D}));
  return LAZYMAR_OK;
}

lazymar_status embed(lazymar_handle* h, const Ctx& c, int rows, int B) {
  const double bytes = (double)rows * h->T * h->D * (4.0 + h->es);
  return launch(h, LAZYMAR_K_EMBED, 0, bytes, c.stream, "embed", [&] {
    return launch_embed(c, h->cfg.dtype, h->st_lat, h->st_mask, h->st_labels, h->pos, h->cls, h->memb, h->ew, h->eb, h->H, rows,
                        B, h->T, h->cfg.n_buffer, h->cfg.n_img, h->D, h->cfg.token_dim, h->cfg.n_classes);
  });
}

lazymar_status final_ln(lazymar_handle* h, const Ctx& c, const float* x, const int* map, int M) {
  if (M == 0) return LAZYMAR_OK;
  const double bytes = (double)M * h->D * (4.0 + h->es);
  return launch(h, LAZYMAR_K_LAYERNORM, 0, bytes, c.stream, "final layernorm", [&] {
    return launch_final_ln(c, h->cfg.dtype, x, map, h->T, h->cfg.n_buffer, h->cfg.n_img, h->lnf_g, h->lnf_b, h->zc, M,
                           h->D, h->cfg.ln_eps);
  });
}

lazymar_status cfg(lazymar_handle* h, const Ctx& c, int mode, int B, float gamma, void* zu_out, void* g_out) {
  const size_t n = (size_t)B * h->cfg.n_img * h->D;
  const uint8_t* zc = static_cast<const uint8_t*>(h->zc);
  const double bytes = (double)n * h->es * (mode == LAZYMAR_CFG_GUIDE ? 3.0 : 4.0);
  return launch(h, LAZYMAR_K_CFG, 0, bytes, c.stream, "cfg", [&] {
    return launch_cfg(c, h->cfg.dtype, mode, zc, zc + n * h->es, h->delta, gamma, n, zu_out, g_out);
  });
}

// Resolves an output pointer: device pointers on a 16-byte boundary (the
// kernels store 16-byte vectors) are written directly, any other pointer
// through the staging buffer `st` and a copy at the end.
void* out_target(void* user, void* st) {
  return user == nullptr ? nullptr : (is_device_ptr(user) && aligned16(user) ? user : st);
}

// Target of the guided output, which the CFG kernel writes: the caller's
// buffer when it is device memory, or page-locked host memory mapped into the
// device's address space (cudaHostAlloc / cudaHostRegister under unified
// addressing), which the kernel then writes directly (no staging and no
// separate device-to-host copy); otherwise the staging buffer, copied out
// afterwards.
void* guided_target(void* user, void* st) {
  if (user == nullptr) return nullptr;
  if (is_device_ptr(user)) return aligned16(user) ? user : st;
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, user) != cudaSuccess) {
    cudaGetLastError();
    return st;
  }
  if (a.type == cudaMemoryTypeHost && a.devicePointer && aligned16(a.devicePointer)) return a.devicePointer;
  return st;
}

// Device work of a full step up to the output cache (everything but the CFG
// combine, which takes gamma and stays outside any graph).
lazymar_status full_body(lazymar_handle* h, const Ctx& c, int B) {
  const int rows = 2 * B, s = h->s;
  LM_TRY(embed(h, c, rows, B));
  for (int l = 0; l < h->L; ++l) {
    const bool value_ref = l == s - 1 && h->cfg.criterion == LAZYMAR_CRITERION_VALUE;
    void* kdst = l >= s ? h->Kc[l] : h->Ks;
    void* vdst = l >= s ? h->Vc[l] : (value_ref ? h->ref : h->Vs);
    LM_TRY(layer_full(h, c, l, rows, kdst, vdst));
    if (l == s - 1 && h->cfg.criterion == LAZYMAR_CRITERION_FEATURE) {
      const size_t n = (size_t)rows * h->T * h->D;
      LM_TRY(launch(h, LAZYMAR_K_OTHER, 0, n * (4.0 + h->es), c.stream, "cast",
                    [&] { return launch_cast(c, h->cfg.dtype, h->H, h->ref, n); }));
    }
  }
  return final_ln(h, c, h->H, nullptr, rows * h->T);
}

// Device work of a cached step up to the output cache.
//
// Under the value criterion the output of block s-1 is read only for the
// selected tokens (blocks s..L-1 see no other token's features, and the cache
// keeps K/V of blocks >= s only). So block s-1 runs LN1 and the Q/K/V
// projection over all tokens (its keys and values, and the value matrix Eq. 8
// compares), then attention, out-projection and MLP for the selected tokens
// alone. The feature criterion compares block s-1's output features, which
// then run over all tokens.
lazymar_status cached_body(lazymar_handle* h, const Ctx& c, int rows, int N, bool has_idx, int sel) {
  const int s = h->s, T = h->T, D = h->D;
  const bool value = h->cfg.criterion == LAZYMAR_CRITERION_VALUE;
  LM_TRY(embed(h, c, rows, h->last_batch));
  for (int l = 0; l < s - (value ? 1 : 0); ++l) LM_TRY(layer_full(h, c, l, rows, h->Ks, h->Vs));
  if (value) {
    const BlockDev& b = h->blk[s - 1];
    const int M = rows * T;
    LM_TRY(layernorm(h, c, h->H, nullptr, b.ln1_g, b.ln1_b, h->A, nullptr, M));
    LM_TRY(gemm(h, c, h->A, b.w_qkv, M, 3 * D, D, GemmEpi{LAZYMAR_EPI_QKV, b.b_qkv, h->Q, D, h->Ks, h->Vs, nullptr, D}));
  }
  // Eq. 8: similarity of block s-1's representation with the reference, then
  // the reference takes this step's values.
  const void* cur = h->Vs;
  if (h->cfg.criterion == LAZYMAR_CRITERION_FEATURE) {
    const size_t n = (size_t)rows * T * D;
    LM_TRY(launch(h, LAZYMAR_K_OTHER, 0, n * (4.0 + h->es), c.stream, "cast",
                  [&] { return launch_cast(c, h->cfg.dtype, h->H, h->Fs, n); }));
    cur = h->Fs;
  }
  LM_TRY(launch(h, LAZYMAR_K_SELECT, 0, 3.0 * rows * T * D * h->es + 8.0 * rows * T, c.stream, "similarity",
                [&] { return launch_similarity(c, h->cfg.dtype, cur, h->ref, h->S, rows, T, D, true); }));
  if (has_idx) {
    LM_TRY(launch(h, LAZYMAR_K_SELECT, 0, 12.0 * rows * N, c.stream, "index check",
                  [&] { return launch_idx_check(c, h->st_idx_in, rows, T, N, h->idx, h->row_map); }));
  } else if (N > 0) {
    LM_TRY(launch(h, LAZYMAR_K_SELECT, 0, 8.0 * rows * T + 8.0 * rows * N, c.stream, "topk",
                  [&] {
                    return launch_topk(c, h->S, rows, T, N, h->idx, h->row_map, h->cfg.select_rule,
                                       (sel & 1) ? h->st_prio : nullptr, (sel & 2) ? h->st_keys : nullptr);
                  }));
  }
  if (N > 0) {
    if (value) {
      // rest of block s-1 on the selected tokens: their queries and residual
      // rows gathered (queries into the free LayerNorm buffer)
      const BlockDev& b = h->blk[s - 1];
      const int M = rows * N;
      LM_TRY(launch(h, LAZYMAR_K_OTHER, 0, (double)M * D * (h->es + 4.0) * 2.0, c.stream, "gather", [&] {
        return launch_gather_rows(c, h->cfg.dtype, h->Q, h->H, h->row_map, h->A, h->Hc, M, D);
      }));
      LM_TRY(attention(h, c, h->Ks, h->Vs, rows, N, h->A));
      LM_TRY(gemm(h, c, h->O, b.w_o, M, D, D, GemmEpi{LAZYMAR_EPI_RESIDUAL, b.b_o, h->Hc, D, nullptr, nullptr, nullptr, D}));
      LM_TRY(layernorm(h, c, h->Hc, nullptr, b.ln2_g, b.ln2_b, h->A, nullptr, M));
      LM_TRY(gemm(h, c, h->A, b.w1, M, h->H4, D, GemmEpi{LAZYMAR_EPI_GELU, b.b1, h->U, h->H4, nullptr, nullptr, nullptr, D}));
      LM_TRY(gemm(h, c, h->U, b.w2, M, D, h->H4, GemmEpi{LAZYMAR_EPI_RESIDUAL, b.b2, h->Hc, D, nullptr, nullptr, nullptr, D}));
    }
    for (int l = s; l < h->L; ++l) LM_TRY(layer_cached(h, c, l, rows, N, l == s && !value));
    LM_TRY(final_ln(h, c, h->Hc, h->row_map, rows * N));
  }
  return LAZYMAR_OK;
}

void add_stats(lazymar_stats& a, const lazymar_stats& d, double sign) {
  for (int i = 0; i < LAZYMAR_K_COUNT; ++i) {
    a.k[i].launches += (long long)sign * d.k[i].launches;
    a.k[i].flops += sign * d.k[i].flops;
    a.k[i].bytes += sign * d.k[i].bytes;
  }
}

// Reads the event pairs of a replayed profiled graph into the statistics.
lazymar_status drain_profiled(lazymar_handle* h, lazymar_handle::GraphEntry& ge) {
  if (!ge.pending) return LAZYMAR_OK;
  ge.pending = false;
  if (ge.evs.empty()) return LAZYMAR_OK;
  LM_CUDA(cudaEventSynchronize(ge.evs.back().b));
  for (const auto& e : ge.evs) {
    float ms = 0.f;
    LM_CUDA(cudaEventElapsedTime(&ms, e.a, e.b));
    h->stats.k[e.cls].ms += ms;
    h->stats.k[e.cls].timed_launches += 1;
  }
  return LAZYMAR_OK;
}

// Runs a step body: eagerly on the caller's stream on its first use (and
// always with graphs disabled); from then on as a CUDA graph, captured on the
// second use and replayed afterwards. Capture and replay run on the handle's
// own stream, joined to the caller's stream by events (the legacy default
// stream cannot be captured). While profiling, the body is captured with its
// per-launch events into a separate graph on its first use and replayed from
// there (the events are read by lazymar_get_stats, or before the same graph
// is replayed again).
template <class F>
lazymar_status run_body(lazymar_handle* h, cudaStream_t st, const lazymar_handle::GraphKey& key, F&& body) {
  if (!h->use_graphs) return body(Ctx{st, h->err, h->num_sms});
  lazymar_handle::GraphEntry& ge = h->profiling ? h->pgraphs[key] : h->graphs[key];
  if (!h->profiling && !ge.exec && ge.eager_runs++ == 0) return body(Ctx{st, h->err, h->num_sms});
  LM_TRY(drain_profiled(h, ge));
  // captured on the handle's own stream (the caller's may be the legacy
  // stream, which cannot be captured), replayed on the caller's stream
  cudaStream_t gs = h->gstream;
  if (!ge.exec) {
    const lazymar_stats before = h->stats;
    const size_t ev_base = h->ev_used;
    LM_CUDA(cudaStreamBeginCapture(gs, cudaStreamCaptureModeThreadLocal));
    const lazymar_status s = body(Ctx{gs, h->err, h->num_sms});
    cudaGraph_t g = nullptr;
    const cudaError_t e = cudaStreamEndCapture(gs, &g);
    // events recorded by the captured launches belong to the graph
    ge.evs.assign(h->evs.begin() + ev_base, h->evs.begin() + h->ev_used);
    h->evs.erase(h->evs.begin() + ev_base, h->evs.begin() + h->ev_used);
    h->ev_used = ev_base;
    if (s != LAZYMAR_OK || e != cudaSuccess) {
      if (g) cudaGraphDestroy(g);
      h->stats = before;
      return s != LAZYMAR_OK ? s : cuda_fail(e, "cudaStreamEndCapture");
    }
    const cudaError_t ei = cudaGraphInstantiate(&ge.exec, g, 0);
    cudaGraphDestroy(g);
    if (ei != cudaSuccess) {
      ge.exec = nullptr;
      h->stats = before;
      return cuda_fail(ei, "cudaGraphInstantiate");
    }
    ge.delta = h->stats;
    add_stats(ge.delta, before, -1.0);
    h->stats = before;
  }
  LM_CUDA(cudaGraphLaunch(ge.exec, st));
  add_stats(h->stats, ge.delta, 1.0);
  ge.pending = h->profiling;
  return LAZYMAR_OK;
}

}  // namespace

extern "C" lazymar_status lazymar_full_step(lazymar_handle* h, const lazymar_step_in* in, float gamma, void* z_out,
                                            void* guided_out, void* stream) {
  NvtxRange range("lazymar_full_step");
  LM_TRY(check_step_in(h, in));
  DeviceGuard dg(h->dev);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const Ctx c{st, h->err, h->num_sms};
  const int B = in->batch;
  Stager sg{h, st};
  LM_TRY(stage_inputs(sg, in));
  LM_TRY(sg.flush(c));
  LM_TRY(run_body(h, st, lazymar_handle::GraphKey{0, B, 0, 0, 0, 0}, [&](const Ctx& cc) { return full_body(h, cc, B); }));
  void* g_dst = guided_target(guided_out, h->st_g);
  LM_TRY(cfg(h, c, LAZYMAR_CFG_REFRESH, B, gamma, nullptr, g_dst));
  const size_t zbytes = (size_t)2 * B * h->cfg.n_img * h->D * h->es;
  if (z_out) LM_CUDA(cudaMemcpyAsync(z_out, h->zc, zbytes, cudaMemcpyDefault, st));
  if (guided_out && g_dst == h->st_g)
    LM_CUDA(cudaMemcpyAsync(guided_out, g_dst, zbytes / 2, cudaMemcpyDefault, st));
  h->primed = true;
  h->last_batch = B;
  return LAZYMAR_OK;
}

extern "C" lazymar_status lazymar_cached_step(lazymar_handle* h, const lazymar_step_in* in, int n_compute,
                                              int use_cond_cache, float gamma, const int32_t* idx_in,
                                              int32_t* idx_out, void* z_out, void* guided_out, void* stream) {
  NvtxRange range(use_cond_cache ? "lazymar_cached_step (condition cache reused)" : "lazymar_cached_step");
  LM_TRY(check_step_in(h, in));
  if (n_compute < 0 || n_compute > h->T) return fail(LAZYMAR_ERR_INVALID_ARG, "n_compute outside 0..T");
  if (!h->primed) return fail(LAZYMAR_ERR_STATE, "cached step before any full step");
  if (in->batch != h->last_batch) return fail(LAZYMAR_ERR_STATE, "batch differs from the last full step");
  DeviceGuard dg(h->dev);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const Ctx c{st, h->err, h->num_sms};
  const int B = in->batch, rows = use_cond_cache ? B : 2 * B, N = n_compute, D = h->D;
  Stager sg{h, st};
  LM_TRY(stage_inputs(sg, in));
  const bool has_idx = idx_in != nullptr && N > 0;
  if (has_idx) LM_TRY(sg.add(h->st_idx_in, idx_in, (size_t)rows * N * 4));
  // selection inputs (Table 3 rules): priority classes and random keys
  const bool sel_rule = !has_idx && N > 0;
  const bool has_prio = sel_rule && in->select_priority != nullptr;
  const bool has_keys = sel_rule && h->cfg.select_rule == LAZYMAR_SELECT_RANDOM;
  if (has_keys && !in->select_keys)
    return fail(LAZYMAR_ERR_INVALID_ARG, "LAZYMAR_SELECT_RANDOM needs select_keys on cached steps");
  const size_t rowsT = (size_t)rows * h->T;
  if (has_prio) LM_TRY(sg.add(h->st_prio, in->select_priority, rowsT));
  if (has_keys) LM_TRY(sg.add(h->st_keys, in->select_keys, rowsT * 4));
  LM_TRY(sg.flush(c));
  const int sel = (has_prio ? 1 : 0) | (has_keys ? 2 : 0);
  LM_TRY(run_body(h, st, lazymar_handle::GraphKey{1, B, N, use_cond_cache ? 1 : 0, has_idx ? 1 : 0, sel},
                  [&](const Ctx& cc) { return cached_body(h, cc, rows, N, has_idx, sel); }));

  const size_t n_el = (size_t)B * h->cfg.n_img * D;
  void* z_dst = out_target(z_out, h->st_z);
  void* g_dst = guided_target(guided_out, h->st_g);
  uint8_t* z8 = static_cast<uint8_t*>(z_dst);
  if (use_cond_cache) {
    LM_TRY(cfg(h, c, LAZYMAR_CFG_REUSE, B, gamma, z8 ? z8 + n_el * h->es : nullptr, g_dst));
    if (z8) LM_CUDA(cudaMemcpyAsync(z8, h->zc, n_el * h->es, cudaMemcpyDeviceToDevice, st));
  } else {
    LM_TRY(cfg(h, c, LAZYMAR_CFG_REFRESH, B, gamma, nullptr, g_dst));
    if (z8) LM_CUDA(cudaMemcpyAsync(z8, h->zc, 2 * n_el * h->es, cudaMemcpyDeviceToDevice, st));
  }
  if (z_out && z_dst != z_out) LM_CUDA(cudaMemcpyAsync(z_out, z_dst, 2 * n_el * h->es, cudaMemcpyDefault, st));
  if (guided_out && g_dst == h->st_g)
    LM_CUDA(cudaMemcpyAsync(guided_out, g_dst, n_el * h->es, cudaMemcpyDefault, st));
  if (idx_out && N > 0) LM_CUDA(cudaMemcpyAsync(idx_out, h->idx, (size_t)rows * N * 4, cudaMemcpyDefault, st));
  return LAZYMAR_OK;
}

extern "C" lazymar_status lazymar_set_graphs(lazymar_handle* h, int enable) {
  if (!h) return fail(LAZYMAR_ERR_INVALID_ARG, "NULL handle");
  h->use_graphs = enable != 0;
  return LAZYMAR_OK;
}

// ---------------------------------------------------------------------------
// Component entry points
// ---------------------------------------------------------------------------
extern "C" lazymar_status lazymar_select_tokens_ex(int dtype, const void* v_cur, void* v_cache, int rows, int T,
                                                   int D, int n_compute, int rule, const uint8_t* priority,
                                                   const uint32_t* keys, int32_t* idx_out, void* stream) {
  if (dtype != LAZYMAR_F32 && dtype != LAZYMAR_BF16) return fail(LAZYMAR_ERR_INVALID_ARG, "dtype");
  if (rule < LAZYMAR_SELECT_LEAST_SIMILAR || rule > LAZYMAR_SELECT_RANDOM) return fail(LAZYMAR_ERR_INVALID_ARG, "rule");
  if (rows < 0 || T < 1 || T > 16384 || D < 8 || D % 8 != 0 || n_compute < 0 || n_compute > T)
    return fail(LAZYMAR_ERR_INVALID_ARG, "rows >= 0, 1 <= T <= 16384, D % 8 == 0, 0 <= n_compute <= T required");
  if (rows == 0) return LAZYMAR_OK;
  if (!is_device_ptr(v_cur) || !is_device_ptr(v_cache) || (n_compute > 0 && !is_device_ptr(idx_out)))
    return fail(LAZYMAR_ERR_INVALID_ARG, "v_cur, v_cache and idx_out must be device pointers");
  if (priority && !is_device_ptr(priority)) return fail(LAZYMAR_ERR_INVALID_ARG, "priority must be a device pointer");
  if (rule == LAZYMAR_SELECT_RANDOM && !is_device_ptr(keys))
    return fail(LAZYMAR_ERR_INVALID_ARG, "LAZYMAR_SELECT_RANDOM needs device keys");
  if (!aligned16(v_cur) || !aligned16(v_cache)) return fail(LAZYMAR_ERR_INVALID_ARG, "16-byte alignment required");
  Ctx c;
  LM_TRY(component_ctx(stream, &c));
  double* S = nullptr;
  LM_CUDA(cudaMallocAsync(reinterpret_cast<void**>(&S), (size_t)rows * T * sizeof(double), c.stream));
  cudaError_t e = launch_similarity(c, dtype, v_cur, v_cache, S, rows, T, D, true);
  if (e == cudaSuccess)
    e = launch_topk(c, S, rows, T, n_compute, idx_out, nullptr, rule, priority,
                    rule == LAZYMAR_SELECT_RANDOM ? keys : nullptr);
  cudaError_t e2 = cudaFreeAsync(S, c.stream);
  if (e != cudaSuccess) return cuda_fail(e, "select kernels");
  if (e2 != cudaSuccess) return cuda_fail(e2, "cudaFreeAsync");
  return LAZYMAR_OK;
}

extern "C" lazymar_status lazymar_select_tokens(int dtype, const void* v_cur, void* v_cache, int rows, int T, int D,
                                                int n_compute, int32_t* idx_out, void* stream) {
  return lazymar_select_tokens_ex(dtype, v_cur, v_cache, rows, T, D, n_compute, LAZYMAR_SELECT_LEAST_SIMILAR, nullptr,
                                  nullptr, idx_out, stream);
}

extern "C" lazymar_status lazymar_cfg_combine(int dtype, int mode, const void* z_cond, const void* z_uncond,
                                              void* delta, float gamma, size_t n, void* z_uncond_out,
                                              void* guided_out, void* stream) {
  if (dtype != LAZYMAR_F32 && dtype != LAZYMAR_BF16) return fail(LAZYMAR_ERR_INVALID_ARG, "dtype");
  if (mode < LAZYMAR_CFG_GUIDE || mode > LAZYMAR_CFG_REUSE) return fail(LAZYMAR_ERR_INVALID_ARG, "mode");
  if (n == 0) return LAZYMAR_OK;
  if (!is_device_ptr(z_cond)) return fail(LAZYMAR_ERR_INVALID_ARG, "z_cond must be a device pointer");
  if (mode != LAZYMAR_CFG_REUSE && !is_device_ptr(z_uncond))
    return fail(LAZYMAR_ERR_INVALID_ARG, "z_uncond must be a device pointer");
  if (mode != LAZYMAR_CFG_GUIDE && !is_device_ptr(delta)) return fail(LAZYMAR_ERR_INVALID_ARG, "delta must be a device pointer");
  if ((guided_out && !is_device_ptr(guided_out)) || (z_uncond_out && !is_device_ptr(z_uncond_out)))
    return fail(LAZYMAR_ERR_INVALID_ARG, "outputs must be device pointers");
  const void* ps[] = {z_cond, z_uncond, delta, z_uncond_out, guided_out};
  for (const void* p : ps)
    if (p && !aligned16(p)) return fail(LAZYMAR_ERR_INVALID_ARG, "16-byte alignment required");
  Ctx c;
  LM_TRY(component_ctx(stream, &c));
  cudaError_t e = launch_cfg(c, dtype, mode, z_cond, z_uncond, delta, gamma, n, z_uncond_out, guided_out);
  return e == cudaSuccess ? LAZYMAR_OK : cuda_fail(e, "cfg kernel");
}

extern "C" lazymar_status lazymar_linear(int dtype, int epilogue, const void* a, const void* w, const void* bias, int M,
                                         int N, int K, void* out, int ldo, void* k_out, void* v_out,
                                         const int32_t* row_map, int flags, void* stream) {
  if (epilogue < LAZYMAR_EPI_BIAS || epilogue > LAZYMAR_EPI_SILU) return fail(LAZYMAR_ERR_INVALID_ARG, "epilogue");
  if (flags < 0 || flags > 4) return fail(LAZYMAR_ERR_INVALID_ARG, "flags");
  GemmEpi e{epilogue, bias, out, ldo, k_out, v_out, row_map, epilogue == LAZYMAR_EPI_QKV ? N / 3 : 0};
  const char* why = "";
  if (!gemm_supported(dtype, M, N, K, e, &why)) return fail(LAZYMAR_ERR_UNSUPPORTED, why);
  if (epilogue != LAZYMAR_EPI_QKV && ldo < N) return fail(LAZYMAR_ERR_INVALID_ARG, "ldo < N");
  if (M == 0) return LAZYMAR_OK;
  if (!is_device_ptr(a) || !is_device_ptr(w) || !is_device_ptr(out) || (bias && !is_device_ptr(bias)))
    return fail(LAZYMAR_ERR_INVALID_ARG, "a, w, bias and out must be device pointers");
  if (epilogue == LAZYMAR_EPI_QKV && (!is_device_ptr(k_out) || !is_device_ptr(v_out)))
    return fail(LAZYMAR_ERR_INVALID_ARG, "k_out and v_out must be device pointers");
  const void* ps[] = {a, w, bias, out, k_out, v_out};
  for (const void* p : ps)
    if (p && !aligned16(p)) return fail(LAZYMAR_ERR_INVALID_ARG, "16-byte alignment required");
  Ctx c;
  LM_TRY(component_ctx(stream, &c));
  cudaError_t err = launch_gemm(c, dtype, a, w, M, N, K, e, flags);
  return err == cudaSuccess ? LAZYMAR_OK : cuda_fail(err, "gemm kernel");
}

extern "C" lazymar_status lazymar_linear_e4m3(int epilogue, const void* a, const void* w, const float* wscale,
                                              const void* bias, int M, int N, int K, void* out, int ldo, void* k_out,
                                              void* v_out, const int32_t* row_map, int flags, void* stream) {
  if (epilogue != LAZYMAR_EPI_BIAS && epilogue != LAZYMAR_EPI_GELU && epilogue != LAZYMAR_EPI_QKV)
    return fail(LAZYMAR_ERR_INVALID_ARG, "epilogue: BIAS, GELU or QKV");
  if (flags < 0 || flags > 4) return fail(LAZYMAR_ERR_INVALID_ARG, "flags");
  GemmEpi e{epilogue, bias, out, ldo, k_out, v_out, row_map, epilogue == LAZYMAR_EPI_QKV ? N / 3 : 0};
  e.wscale = wscale;
  const char* why = "";
  if (!gemm_supported(LAZYMAR_E4M3, M, N, K, e, &why)) return fail(LAZYMAR_ERR_UNSUPPORTED, why);
  if (epilogue != LAZYMAR_EPI_QKV && ldo < N) return fail(LAZYMAR_ERR_INVALID_ARG, "ldo < N");
  if (M == 0) return LAZYMAR_OK;
  if (!is_device_ptr(a) || !is_device_ptr(w) || !is_device_ptr(wscale) || !is_device_ptr(out) ||
      (bias && !is_device_ptr(bias)))
    return fail(LAZYMAR_ERR_INVALID_ARG, "a, w, wscale, bias and out must be device pointers");
  if (epilogue == LAZYMAR_EPI_QKV && (!is_device_ptr(k_out) || !is_device_ptr(v_out)))
    return fail(LAZYMAR_ERR_INVALID_ARG, "k_out and v_out must be device pointers");
  const void* ps[] = {a, w, wscale, bias, out, k_out, v_out};
  for (const void* p : ps)
    if (p && !aligned16(p)) return fail(LAZYMAR_ERR_INVALID_ARG, "16-byte alignment required");
  Ctx c;
  LM_TRY(component_ctx(stream, &c));
  cudaError_t err = launch_gemm(c, LAZYMAR_E4M3, a, w, M, N, K, e, flags);
  return err == cudaSuccess ? LAZYMAR_OK : cuda_fail(err, "E4M3 gemm kernel");
}

extern "C" lazymar_status lazymar_quantize_e4m3(const void* w, int rows, int cols, void* q, float* scale,
                                                void* stream) {
  if (rows < 0 || cols < 8 || cols % 8 != 0) return fail(LAZYMAR_ERR_INVALID_ARG, "rows >= 0, cols % 8 == 0 required");
  if (rows == 0) return LAZYMAR_OK;
  if (!is_device_ptr(w) || !is_device_ptr(q) || !is_device_ptr(scale))
    return fail(LAZYMAR_ERR_INVALID_ARG, "device pointers required");
  if (!aligned16(w) || (reinterpret_cast<uintptr_t>(q) & 7u))
    return fail(LAZYMAR_ERR_INVALID_ARG, "w 16-byte and q 8-byte alignment required");
  Ctx c;
  LM_TRY(component_ctx(stream, &c));
  cudaError_t e = launch_quantize_e4m3(c, w, rows, cols, q, scale);
  return e == cudaSuccess ? LAZYMAR_OK : cuda_fail(e, "E4M3 quantization kernel");
}

extern "C" lazymar_status lazymar_attention(int dtype, const void* q, const void* k, const void* v, void* o, int rows,
                                            int n_q, int T, int heads, int head_dim, void* stream) {
  const char* why = "";
  if (!attention_supported(dtype, heads, head_dim, &why)) return fail(LAZYMAR_ERR_UNSUPPORTED, why);
  if (rows < 0 || n_q < 0 || T < 1) return fail(LAZYMAR_ERR_INVALID_ARG, "rows >= 0, n_q >= 0, T >= 1 required");
  if (dtype == LAZYMAR_F32 && T > 8192) return fail(LAZYMAR_ERR_UNSUPPORTED, "f32 attention supports T <= 8192");
  if (rows == 0 || n_q == 0) return LAZYMAR_OK;
  if (!is_device_ptr(q) || !is_device_ptr(k) || !is_device_ptr(v) || !is_device_ptr(o))
    return fail(LAZYMAR_ERR_INVALID_ARG, "q, k, v and o must be device pointers");
  const void* ps[] = {q, k, v, o};
  for (const void* p : ps)
    if (!aligned16(p)) return fail(LAZYMAR_ERR_INVALID_ARG, "16-byte alignment required");
  Ctx c;
  LM_TRY(component_ctx(stream, &c));
  cudaError_t e = launch_attention(c, dtype, q, k, v, o, rows, n_q, T, heads, head_dim);
  return e == cudaSuccess ? LAZYMAR_OK : cuda_fail(e, "attention kernel");
}

extern "C" lazymar_status lazymar_layernorm(int dtype, const float* x, const int32_t* row_map, const void* g,
                                            const void* b, void* y, int M, int D, float eps, void* stream) {
  if (dtype != LAZYMAR_F32 && dtype != LAZYMAR_BF16 && dtype != LAZYMAR_E4M3)
    return fail(LAZYMAR_ERR_INVALID_ARG, "dtype");
  if (M < 0 || !layernorm_width_ok(D) || !(eps > 0.f))
    return fail(LAZYMAR_ERR_UNSUPPORTED, "M >= 0, D = 128 * {1,2,4,6,8,10,12,16}, eps > 0 required");
  if (M == 0) return LAZYMAR_OK;
  if (!is_device_ptr(x) || !is_device_ptr(g) || !is_device_ptr(b) || !is_device_ptr(y) ||
      (row_map && !is_device_ptr(row_map)))
    return fail(LAZYMAR_ERR_INVALID_ARG, "device pointers required");
  Ctx c;
  LM_TRY(component_ctx(stream, &c));
  cudaError_t e = launch_layernorm(c, dtype, x, row_map, g, b, y, nullptr, M, D, eps);
  return e == cudaSuccess ? LAZYMAR_OK : cuda_fail(e, "layernorm kernel");
}

// ---------------------------------------------------------------------------
// Host logic, errors, statistics
// ---------------------------------------------------------------------------
extern "C" int lazymar_plan_step(int k, int k0, int tau, int tau_cfg, int use_cond_cache) {
  if (k < 0 || k0 < 0 || tau < 1 || tau_cfg < 0) return -1;
  if (k < k0 || (k - k0) % tau == 0) return 1;
  const bool reuse = use_cond_cache && tau_cfg > 0 && (k - k0) % tau_cfg != 0;
  return reuse ? 2 : 0;
}

extern "C" lazymar_status lazymar_sync(lazymar_handle* h, void* stream) {
  if (!h) return fail(LAZYMAR_ERR_INVALID_ARG, "NULL handle");
  DeviceGuard dg(h->dev);
  return read_error_word(h->err, static_cast<cudaStream_t>(stream));
}

extern "C" lazymar_status lazymar_read_reference(lazymar_handle* h, int rows, void* dst, void* stream) {
  if (!h || !dst) return fail(LAZYMAR_ERR_INVALID_ARG, "NULL handle or destination");
  if (rows < 1 || rows > h->max_rows) return fail(LAZYMAR_ERR_INVALID_ARG, "rows outside 1..2 max_batch");
  if (!h->primed) return fail(LAZYMAR_ERR_STATE, "no full step has run yet");
  DeviceGuard dg(h->dev);
  const size_t bytes = (size_t)rows * h->T * h->D * h->es;
  LM_CUDA(cudaMemcpyAsync(dst, h->ref, bytes, cudaMemcpyDefault, static_cast<cudaStream_t>(stream)));
  return LAZYMAR_OK;
}

extern "C" lazymar_status lazymar_selftest_wait(int limit_us, void* stream) {
  if (limit_us < 1 || limit_us > 1000000) return fail(LAZYMAR_ERR_INVALID_ARG, "limit_us outside 1..1000000");
  Ctx c;
  LM_TRY(component_ctx(stream, &c));
  cudaError_t e = launch_stuck_wait(c, (uint64_t)limit_us * 1000ull);
  return e == cudaSuccess ? LAZYMAR_OK : cuda_fail(e, "stuck-wait kernel");
}

extern "C" lazymar_status lazymar_device_check(void* stream) {
  Ctx c;
  LM_TRY(component_ctx(stream, &c));
  return read_error_word(c.err, c.stream);
}

extern "C" lazymar_status lazymar_set_profiling(lazymar_handle* h, int enable) {
  if (!h) return fail(LAZYMAR_ERR_INVALID_ARG, "NULL handle");
  h->profiling = enable != 0;
  return LAZYMAR_OK;
}

extern "C" lazymar_status lazymar_get_stats(lazymar_handle* h, lazymar_stats* out) {
  if (!h || !out) return fail(LAZYMAR_ERR_INVALID_ARG, "NULL argument");
  DeviceGuard dg(h->dev);
  for (auto& kv : h->pgraphs) LM_TRY(drain_profiled(h, kv.second));
  if (h->ev_used > 0) {
    LM_CUDA(cudaEventSynchronize(h->evs[h->ev_used - 1].b));
    for (size_t i = 0; i < h->ev_used; ++i) {
      float ms = 0.f;
      LM_CUDA(cudaEventElapsedTime(&ms, h->evs[i].a, h->evs[i].b));
      h->stats.k[h->evs[i].cls].ms += ms;
      h->stats.k[h->evs[i].cls].timed_launches += 1;
    }
    h->ev_used = 0;
  }
  *out = h->stats;
  return LAZYMAR_OK;
}

extern "C" lazymar_status lazymar_reset_stats(lazymar_handle* h) {
  if (!h) return fail(LAZYMAR_ERR_INVALID_ARG, "NULL handle");
  lazymar_stats tmp;
  LM_TRY(lazymar_get_stats(h, &tmp));  // drains pending events
  h->stats = lazymar_stats{};
  return LAZYMAR_OK;
}

extern "C" const char* lazymar_status_string(lazymar_status s) {
  switch (s) {
    case LAZYMAR_OK: return "ok";
    case LAZYMAR_ERR_INVALID_ARG: return "invalid argument";
    case LAZYMAR_ERR_OOM: return "out of device memory";
    case LAZYMAR_ERR_CUDA: return "CUDA error";
    case LAZYMAR_ERR_STATE: return "invalid state";
    case LAZYMAR_ERR_TIMEOUT: return "device wait timed out";
    case LAZYMAR_ERR_UNSUPPORTED: return "unsupported shape";
    case LAZYMAR_ERR_DEVICE: return "device-side argument error";
  }
  return "unknown status";
}

extern "C" const char* lazymar_last_error(void) { return g_last_error.c_str(); }
