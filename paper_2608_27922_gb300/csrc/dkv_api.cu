// Host implementation of the C ABI declared in include/dkv.h.
#include "../../include/dkv.h"
#include <nvtx3/nvToolsExt.h>
#include "dkv_internal.h"

#include <cmath>
#include <cstring>
#include <map>
#include <mutex>
#include <new>
#include <string>
#include <algorithm>
#include <vector>

namespace dkv {

// ------------------------------------------------------------------ timing hook
struct Timer {
  bool on = false;
  bool attend_only = false;   // bracket only the attention launches
  struct Rec {
    std::string name;
    cudaEvent_t a, b;
  };
  std::vector<Rec> pending;
  std::vector<cudaEvent_t> pool;
  std::map<std::string, std::pair<int, double>> acc;
  std::vector<std::string> order;
  std::string cur;
  cudaEvent_t cur_a = nullptr;

  cudaEvent_t get() {
    if (!pool.empty()) {
      cudaEvent_t e = pool.back();
      pool.pop_back();
      return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
  }
  void drain() {
    for (auto& r : pending) {
      cudaEventSynchronize(r.b);
      float ms = 0.f;
      cudaEventElapsedTime(&ms, r.a, r.b);
      auto it = acc.find(r.name);
      if (it == acc.end()) {
        acc[r.name] = {1, (double)ms};
        order.push_back(r.name);
      } else {
        it->second.first += 1;
        it->second.second += ms;
      }
      pool.push_back(r.a);
      pool.push_back(r.b);
    }
    pending.clear();
  }
  ~Timer() {
    for (auto& r : pending) { cudaEventDestroy(r.a); cudaEventDestroy(r.b); }
    for (auto e : pool) cudaEventDestroy(e);
  }
};

// Inside a stream capture a plain event record only orders the graph; an external
// record keeps the timestamp when the graph is replayed.
static void record(cudaEvent_t e, cudaStream_t s) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &st) == cudaSuccess && st == cudaStreamCaptureStatusActive)
    cudaEventRecordWithFlags(e, s, cudaEventRecordExternal);
  else
    cudaEventRecord(e, s);
}

// NVTX: every kernel launch sits in a range named after it, every ABI call in one named
// after the call (host-side ranges; free unless a profiler is attached).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

void timer_begin(Timer* t, const char* name, cudaStream_t s) {
  nvtxRangePushA(name);   // popped by timer_end
  if (!t || !t->on) return;
  if (t->attend_only && std::strncmp(name, "attend", 6) != 0) {   // counted, not timed
    auto it = t->acc.find(name);
    if (it == t->acc.end()) {
      t->acc[name] = {1, 0.0};
      t->order.push_back(name);
    } else {
      it->second.first += 1;
    }
    return;
  }
  t->cur = name;
  t->cur_a = t->get();
  record(t->cur_a, s);
}

void timer_end(Timer* t, cudaStream_t s) {
  nvtxRangePop();
  if (!t || !t->on || !t->cur_a) return;
  cudaEvent_t b = t->get();
  record(b, s);
  t->pending.push_back({t->cur, t->cur_a, b});
  t->cur_a = nullptr;
}

// ------------------------------------------------------------------ workspace
static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

size_t ws_layout(int H, int d, int M_max, int n_max, int bf16, int kv, Ws* out, char* base) {
  const size_t es = bf16 ? 2 : 4;
  const int hist_stride = ((n_max + 2) + 3) & ~3;
  const int snap_stride = n_max / SNAP + 2;
  const int feas_words = (n_max + 1 + 31) / 32;
  size_t off = 0;
  auto take = [&](size_t bytes) -> char* {
    char* p = base ? base + off : nullptr;
    off += align256(bytes);
    return p;
  };
  const size_t Hh = (size_t)H, Nm = (size_t)n_max, Mm = (size_t)M_max;
  Ws w{};
  w.L = (DevLayer*)take(Hh * sizeof(DevLayer));   // room for up to H layers
  w.hd = (DevHead*)take(Hh * sizeof(DevHead));
  w.budgets = (int32_t*)take(Hh * 4);
  w.cnorm = (float*)take(Hh * Nm * 4);
  w.score = (float*)take(Hh * Nm * 4);
  w.perm = (int32_t*)take(Hh * Nm * 4);
  w.kperm = take(Hh * Nm * d * es);
  w.kperm_norm = (float*)take(Hh * Nm * 4);
  w.cross = (int32_t*)take(Hh * Mm * 4);
  w.hist = (int32_t*)take(Hh * hist_stride * 4);
  w.feas = (uint32_t*)take(Hh * feas_words * 4);
  w.snap = (float*)take(Hh * Mm * snap_stride * 4);
  w.rho_t = (float*)take(Hh * Mm * 4);
  w.evict_list = (int32_t*)take(Hh * Nm * 4);
  w.surv_list = (int32_t*)take(Hh * Mm * 4);
  w.kevict = take(Hh * Nm * d * es);
  w.kevict_norm = (float*)take(Hh * Nm * 4);
  w.ksurv = take(Hh * Mm * d * es);
  w.ksurv_norm = (float*)take(Hh * Mm * 4);
  w.slot_new = (int32_t*)take(Hh * Nm * 4);
  w.cext = take(Hh * Nm * 64);
  w.kperm_ext = take(Hh * Nm * 64);
  w.bext = take(Hh * Mm * 64);
  w.ksurv_ext = take(Hh * Mm * 64);
  w.kevict_ext = take(Hh * Nm * 64);
  if (kv) {
    w.vperm = take(Hh * Nm * d * es);
    w.vsurv = take(Hh * Mm * d * es);
    w.vevict = take(Hh * Nm * d * es);
  }
  const int sort_stride = (n_max + 255) / 256 * 256;
  w.sortbuf = (unsigned long long*)take(Hh * (size_t)sort_stride * 8);
  const int invb_stride = (M_max + 3) & ~3;   // 16-byte rows for the bulk copies
  w.invb = (float*)take((Hh * (size_t)invb_stride + 256) * 4);   // a whole 256-column tile past the end
  const int part_stride = (M_max > n_max ? M_max : n_max);
  const int cnt_stride = (part_stride + 127) / 128;
  w.part = (float*)take(2 * Hh * part_stride * 4);
  w.cnt = (int32_t*)take(Hh * cnt_stride * 4);
  w.tile_head = (int32_t*)take(Hh * ((Mm + 127) / 128) * 4);
  w.tile_first = (int32_t*)take(Hh * 4);
  w.pair_head = (int32_t*)take(Hh * (((Mm + 127) / 128 + 1) / 2) * 4);
  w.pair_first = (int32_t*)take(Hh * 4);
  w.head_order = (int32_t*)take(Hh * 4);
  w.loop_stride = (int64_t)(Hh * std::max((Mm + 127) / 128, (Nm + 127) / 128));
  w.loop_list = (int32_t*)take(3 * (size_t)w.loop_stride * 4);
  w.loop_ctr = (int32_t*)take(3 * 2 * 4);
  w.part_stride = part_stride;
  w.cnt_stride = cnt_stride;
  w.invb_stride = invb_stride;
  w.sort_stride = sort_stride;
  w.hist_stride = hist_stride;
  w.snap_stride = snap_stride;
  w.feas_words = feas_words;
  if (out) *out = w;
  return off;
}

}  // namespace dkv

using namespace dkv;

struct dkv_bank_s {
  Bank b{};
  Ws w{};
  KParams kp{};
  dkv_params_t params{};
  std::vector<int32_t> budgets;
  bool tc = false;
  int state = 0;   // 0: idle, 1: admitted, 2: evicted
  int n_layers = 1;
  const int32_t* src_map = nullptr;   // provenance source index of each candidate (sequential admission)
  // commit runs the survivor pass and the new-baselines pass side by side (they touch
  // disjoint slots): the latter on this library-owned stream, forked and joined by events
  cudaStream_t side = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  ~dkv_bank_s() {
    if (ev_fork) cudaEventDestroy(ev_fork);
    if (ev_join) cudaEventDestroy(ev_join);
    if (side) cudaStreamDestroy(side);
  }
  const void* Kc = nullptr;
  const void* Vc = nullptr;
  int N = 0;
  int64_t step = 0;
  cudaStream_t last = nullptr;
  Timer timer;
  int device = 0;
};

namespace {

constexpr int kMaxH = 4096;
constexpr int kMaxM = 262144;
constexpr int kMaxN = 16384;

dkv_status_t cuda_status(cudaError_t e) { return e == cudaSuccess ? DKV_OK : DKV_ERR_CUDA; }

bool aligned(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

std::once_flag g_smem_once;
cudaError_t g_smem_err = cudaSuccess;

}  // namespace

extern "C" {

const char* dkv_status_str(dkv_status_t s) {
  switch (s) {
    case DKV_OK: return "ok";
    case DKV_ERR_ARG: return "invalid argument";
    case DKV_ERR_SHAPE: return "unsupported shape";
    case DKV_ERR_STATE: return "call out of order";
    case DKV_ERR_CUDA: return "CUDA error";
    case DKV_ERR_NOMEM: return "workspace too small";
    case DKV_ERR_TIMEOUT: return "device wait timed out";
    case DKV_ERR_UNSUPPORTED: return "unsupported on this device or dtype";
    case DKV_ERR_DEVICE: return "device-side consistency check failed";
  }
  return "unknown status";
}

int32_t dkv_version(void) { return 200; }   // 0.2.0: dkv_params_t.descriptor, admit_rope

dkv_status_t dkv_params_default(dkv_params_t* out, int32_t d) {
  if (!out || d <= 0) return DKV_ERR_ARG;
  out->tau = 2.0f;
  out->sigma = std::sqrt((float)d / 2.0f);
  out->p = 2.0f;
  out->eps = 1.0f;
  out->delta = 1e-6f;
  out->sync_heads = 1;
  out->score_mode = DKV_SCORE_TENSOR;
  out->order = DKV_ORDER_SCORE;
  out->eviction = DKV_EVICT_MANDATORY_DENSEST;
  out->refresh_baselines = 0;
  out->layer_heads = 0;
  out->descriptor = DKV_DESC_K;
  return DKV_OK;
}

size_t dkv_bank_workspace_size_ex(int32_t H, int32_t d, const int32_t* budgets, int32_t n_max, int32_t dtype,
                                  const dkv_params_t* params) {
  if (H < 1 || H > kMaxH || (d != 64 && d != 128) || !budgets || n_max < 1 || n_max > kMaxN) return 0;
  if (dtype != DKV_DTYPE_BF16 && dtype != DKV_DTYPE_FP32) return 0;
  const int kv = params ? params->descriptor : DKV_DESC_K;
  if (kv != DKV_DESC_K && kv != DKV_DESC_KV) return 0;
  int M_max = 0;
  for (int h = 0; h < H; ++h) {
    if (budgets[h] < 1 || budgets[h] > kMaxM) return 0;
    M_max = budgets[h] > M_max ? budgets[h] : M_max;
  }
  return ws_layout(H, d, M_max, n_max, dtype == DKV_DTYPE_BF16, kv, nullptr, nullptr);
}

size_t dkv_bank_workspace_size(int32_t H, int32_t d, const int32_t* budgets, int32_t n_max, int32_t dtype) {
  return dkv_bank_workspace_size_ex(H, d, budgets, n_max, dtype, nullptr);
}

dkv_status_t dkv_bank_create(dkv_bank_t* out, int32_t H, int32_t d, const int32_t* budgets, int32_t n_max,
                             int32_t dtype, const dkv_params_t* params, const dkv_buffers_t* buf) {
  if (!out || !budgets || !params || !buf) return DKV_ERR_ARG;
  *out = nullptr;
  if (H < 1 || H > kMaxH || (d != 64 && d != 128) || n_max < 1 || n_max > kMaxN) return DKV_ERR_SHAPE;
  if (dtype != DKV_DTYPE_BF16 && dtype != DKV_DTYPE_FP32) return DKV_ERR_ARG;
  const dkv_params_t& p = *params;
  if (!(p.tau > 1.0f) || !(p.eps > 0.0f) || !(p.delta > 0.0f) || !(p.sigma >= 0.0f) ||
      !(p.p == 1.0f || p.p == 2.0f || p.p == 4.0f) || (p.sync_heads != 0 && p.sync_heads != 1) ||
      (p.score_mode != DKV_SCORE_TENSOR && p.score_mode != DKV_SCORE_FP32) ||
      p.layer_heads < 0 || p.layer_heads > H || (p.layer_heads > 0 && H % p.layer_heads != 0) ||
      (p.order != DKV_ORDER_SCORE && p.order != DKV_ORDER_SOURCE) ||
      (p.eviction != DKV_EVICT_MANDATORY_DENSEST && p.eviction != DKV_EVICT_DENSEST &&
       p.eviction != DKV_EVICT_MANDATORY_SOURCE) ||
      (p.refresh_baselines != 0 && p.refresh_baselines != 1) ||
      (p.descriptor != DKV_DESC_K && p.descriptor != DKV_DESC_KV) ||
      !std::isfinite(p.tau) || !std::isfinite(p.sigma) || !std::isfinite(p.eps) || !std::isfinite(p.delta))
    return DKV_ERR_ARG;
  int M_max = 0;
  for (int h = 0; h < H; ++h) {
    if (budgets[h] < 1 || budgets[h] > kMaxM) return DKV_ERR_SHAPE;
    M_max = budgets[h] > M_max ? budgets[h] : M_max;
  }
  if (!buf->k || !buf->v || !buf->rho || !buf->base || !buf->knorm || !buf->prov_step || !buf->prov_src ||
      !buf->occupancy || !buf->workspace)
    return DKV_ERR_ARG;
  if (!aligned(buf->k, 16) || !aligned(buf->v, 16) || !aligned(buf->workspace, 256)) return DKV_ERR_ARG;
  const int bf16 = dtype == DKV_DTYPE_BF16;
  const int kv = p.descriptor == DKV_DESC_KV;
  const size_t need = ws_layout(H, d, M_max, n_max, bf16, kv, nullptr, nullptr);
  if (buf->workspace_bytes < need) return DKV_ERR_NOMEM;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DKV_ERR_CUDA;
  cudaDeviceProp prop;
  if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess) return DKV_ERR_CUDA;
  if (prop.major != 10 || prop.minor != 3) return DKV_ERR_UNSUPPORTED;   // built for sm_103a only
  const bool want_tc = p.score_mode == DKV_SCORE_TENSOR;
  if (want_tc && !tc_supported(d, bf16)) return DKV_ERR_UNSUPPORTED;
  std::call_once(g_smem_once, [] {
    cudaError_t e = simt_set_smem_limits();
    if (e == cudaSuccess) e = update_set_smem_limits();
    if (e == cudaSuccess) e = tc_set_smem_limits();
    g_smem_err = e;
  });
  if (g_smem_err != cudaSuccess) return DKV_ERR_CUDA;

  dkv_bank_s* bk = new (std::nothrow) dkv_bank_s();
  if (!bk) return DKV_ERR_ARG;
  bk->device = dev;
  bk->params = p;
  if (!(bk->params.sigma > 0.0f)) bk->params.sigma = std::sqrt((float)(kv ? 2 * d : d) / 2.0f);
  bk->budgets.assign(budgets, budgets + H);
  bk->tc = want_tc;
  Bank& b = bk->b;
  b.k = buf->k; b.v = buf->v; b.rho = buf->rho; b.base = buf->base; b.knorm = buf->knorm;
  b.prov_step = buf->prov_step; b.prov_src = buf->prov_src; b.occ = buf->occupancy;
  b.H = H; b.d = d; b.M_max = M_max; b.n_max = n_max; b.bf16 = bf16;
  ws_layout(H, d, M_max, n_max, bf16, kv, &bk->w, (char*)buf->workspace);
  bk->w.layer_heads = p.layer_heads > 0 ? p.layer_heads : H;
  bk->n_layers = H / bk->w.layer_heads;
  const float sg = bk->params.sigma;
  bk->kp.inv_s2 = 1.0f / (sg * sg);
  bk->kp.eps = p.eps;
  bk->kp.tau = p.tau;
  bk->kp.delta = p.delta;
  bk->kp.p = (int)p.p;
  bk->kp.sync_heads = p.sync_heads;
  bk->kp.order = p.order;
  bk->kp.eviction = p.eviction;
  bk->kp.refresh = p.refresh_baselines;
  if (cudaStreamCreateWithFlags(&bk->side, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&bk->ev_fork, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&bk->ev_join, cudaEventDisableTiming) != cudaSuccess) {
    delete bk;
    return DKV_ERR_CUDA;
  }
  // workspace header: zeroed layer state and the per-head budgets (one-time, synchronous)
  cudaError_t e = cudaMemset(bk->w.L, 0, sizeof(DevLayer) * bk->n_layers);
  if (e == cudaSuccess) e = cudaMemset(bk->w.hd, 0, sizeof(DevHead) * H);
  if (e == cudaSuccess) e = cudaMemset(bk->w.cnt, 0, sizeof(int32_t) * H * bk->w.cnt_stride);
  if (e == cudaSuccess) e = cudaMemcpy(bk->w.budgets, budgets, sizeof(int32_t) * H, cudaMemcpyHostToDevice);
  // the 128-row tiles of every head's budget, head-major (grids of the passes over bank rows)
  std::vector<int32_t> tile_head, tile_first(H);
  for (int h = 0; h < H; ++h) {
    tile_first[h] = (int32_t)tile_head.size();
    tile_head.insert(tile_head.end(), (size_t)(budgets[h] + 127) / 128, h);
  }
  bk->w.n_mtiles = (int)tile_head.size();
  if (e == cudaSuccess)
    e = cudaMemcpy(bk->w.tile_head, tile_head.data(), sizeof(int32_t) * tile_head.size(), cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(bk->w.tile_first, tile_first.data(), sizeof(int32_t) * H, cudaMemcpyHostToDevice);
  // pairs of those tiles (the units of the two-row-tile crossing pass); the heads by
  // decreasing budget (the persistent score pass takes the largest units first, so that
  // its fixed stride ends on small ones)
  std::vector<int32_t> pair_head, pair_first(H), head_order(H);
  for (int h = 0; h < H; ++h) {
    pair_first[h] = (int32_t)pair_head.size();
    pair_head.insert(pair_head.end(), (size_t)((budgets[h] + 127) / 128 + 1) / 2, h);
    head_order[h] = h;
  }
  std::stable_sort(head_order.begin(), head_order.end(),
                   [&](int32_t a, int32_t b) { return budgets[a] > budgets[b]; });
  bk->w.n_mpairs = (int)pair_head.size();
  if (e == cudaSuccess)
    e = cudaMemcpy(bk->w.head_order, head_order.data(), sizeof(int32_t) * H, cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(bk->w.pair_head, pair_head.data(), sizeof(int32_t) * pair_head.size(), cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(bk->w.pair_first, pair_first.data(), sizeof(int32_t) * H, cudaMemcpyHostToDevice);
  if (e != cudaSuccess) {
    delete bk;
    return DKV_ERR_CUDA;
  }
  *out = bk;
  return DKV_OK;
}

void dkv_bank_destroy(dkv_bank_t bank) { delete bank; }

dkv_status_t dkv_bank_reset(dkv_bank_t bank, void* stream) {
  if (!bank) return DKV_ERR_ARG;
  if (bank->state != 0) return DKV_ERR_STATE;
  cudaStream_t s = (cudaStream_t)stream;
  bank->last = s;
  return cuda_status(cudaMemsetAsync(bank->b.occ, 0, sizeof(int32_t) * bank->b.H, s));
}

static dkv_status_t admit_impl(dkv_bank_t bank, const void* Kc, const void* Vc, int32_t N, int64_t step,
                               const RopeArgs* rope, void* stream) {
  NvtxRange nvtx_range("dkv_bank_admit");
  if (!bank || !Kc || !Vc) return DKV_ERR_ARG;
  if (bank->state != 0) return DKV_ERR_STATE;
  if (N < 1 || N > bank->b.n_max) return DKV_ERR_SHAPE;
  if (step < 0 || step > 0x7fffffffLL) return DKV_ERR_ARG;
  if (!aligned(Kc, 16) || !aligned(Vc, 16)) return DKV_ERR_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  const Bank& b = bank->b;
  const Ws& w = bank->w;
  Timer* t = &bank->timer;
  bank->last = s;
  cudaError_t e = launch_cand_norms(b, w, Kc, Vc, N, step, bank->kp, rope, s, t);
  if (rope) Kc = w.kevict;   // the re-zeroed keys, same [H][N][d] layout
  if (e == cudaSuccess)
    if (bank->kp.order == DKV_ORDER_SCORE)   // source order needs no scores (App. E)
      e = bank->tc ? launch_score_tc(b, w, Kc, Vc, N, bank->kp, s, t) : launch_score_fp32(b, w, Kc, Vc, N, bank->kp, s, t);
  if (e == cudaSuccess) e = launch_sort(b, w, Kc, Vc, bank->kp.order == DKV_ORDER_SOURCE, s, t);
  if (e == cudaSuccess) e = bank->tc ? launch_cross_tc(b, w, bank->kp, s, t) : launch_cross_fp32(b, w, bank->kp, s, t);
  if (e == cudaSuccess) e = launch_rstar(b, w, bank->kp, s, t);
  if (e != cudaSuccess) return DKV_ERR_CUDA;
  bank->state = 1;
  bank->Kc = Kc;
  bank->Vc = Vc;
  bank->N = N;
  bank->step = step;
  return DKV_OK;
}

dkv_status_t dkv_bank_admit(dkv_bank_t bank, const void* Kc, const void* Vc, int32_t N, int64_t step,
                            void* stream) {
  return admit_impl(bank, Kc, Vc, N, step, nullptr, stream);
}

dkv_status_t dkv_bank_admit_rope(dkv_bank_t bank, const void* Kc, const void* Vc, int32_t N, int64_t step,
                                 const int32_t* t_coord, const float* theta, int32_t layout, void* stream) {
  if (!bank) return DKV_ERR_ARG;
  if (!t_coord || !theta || !aligned(t_coord, 4) || !aligned(theta, 4)) return DKV_ERR_ARG;
  if (layout != DKV_ROPE_INTERLEAVED && layout != DKV_ROPE_HALF) return DKV_ERR_ARG;
  const RopeArgs ra{theta, t_coord, layout};
  return admit_impl(bank, Kc, Vc, N, step, &ra, stream);
}

dkv_status_t dkv_bank_evict(dkv_bank_t bank, void* stream) {
  NvtxRange nvtx_range("dkv_bank_evict");
  if (!bank) return DKV_ERR_ARG;
  if (bank->state != 1) return DKV_ERR_STATE;
  cudaStream_t s = (cudaStream_t)stream;
  const Bank& b = bank->b;
  const Ws& w = bank->w;
  Timer* t = &bank->timer;
  const KParams& kp = bank->kp;
  bank->last = s;
  bank->state = 2;
  cudaError_t e = bank->tc ? launch_project_tc(b, w, kp, s, t) : launch_project_fp32(b, w, kp, s, t);
  if (e == cudaSuccess) e = launch_select(b, w, kp.eviction, s, t);
  return cuda_status(e);
}

dkv_status_t dkv_bank_commit(dkv_bank_t bank, void* stream) {
  NvtxRange nvtx_range("dkv_bank_commit");
  if (!bank) return DKV_ERR_ARG;
  if (bank->state != 2) return DKV_ERR_STATE;
  cudaStream_t s = (cudaStream_t)stream;
  const Bank& b = bank->b;
  const Ws& w = bank->w;
  Timer* t = &bank->timer;
  const KParams& kp = bank->kp;
  bank->last = s;
  bank->state = 0;
  cudaError_t e = launch_commit(b, w, bank->Vc, bank->N, bank->src_map, s, t);
  if (t->on && !t->attend_only) {
    // every launch timed: the two passes one after the other on `stream`, so that each
    // launch's time is its own
    if (e == cudaSuccess) e = bank->tc ? launch_subtract_tc(b, w, kp, s, t) : launch_subtract_fp32(b, w, kp, s, t);
    if (e == cudaSuccess) e = bank->tc ? launch_newbase_tc(b, w, kp, s, t) : launch_newbase_fp32(b, w, kp, s, t);
    return cuda_status(e);
  }
  // Eq. C.4 (survivors) on `stream` beside Eq. 5 (admitted states) on the handle's own
  // stream: disjoint slots, read-only inputs; `stream` waits for both
  if (e == cudaSuccess) e = cudaEventRecord(bank->ev_fork, s);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(bank->side, bank->ev_fork, 0);
  if (e == cudaSuccess)
    e = bank->tc ? launch_newbase_tc(b, w, kp, bank->side, t) : launch_newbase_fp32(b, w, kp, bank->side, t);
  if (e == cudaSuccess) e = cudaEventRecord(bank->ev_join, bank->side);
  if (e == cudaSuccess) e = bank->tc ? launch_subtract_tc(b, w, kp, s, t) : launch_subtract_fp32(b, w, kp, s, t);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(s, bank->ev_join, 0);
  return cuda_status(e);
}

dkv_status_t dkv_bank_compress(dkv_bank_t bank, void* stream) {
  if (!bank) return DKV_ERR_ARG;
  if (bank->state != 1) return DKV_ERR_STATE;
  const dkv_status_t st = dkv_bank_evict(bank, stream);
  return st != DKV_OK ? st : dkv_bank_commit(bank, stream);
}

// ---- sequential admission (within-block competition)
namespace {
struct SeqScratch {
  char *kseq, *vseq, *k1, *v1;
  int32_t *srcseq, *src1;
};
size_t seq_layout(int H, int d, int n_max, int bf16, SeqScratch* out, char* base) {
  const size_t es = bf16 ? 2 : 4, rb = (size_t)d * es;
  size_t off = 0;
  auto take = [&](size_t bytes) -> char* {
    char* p = base ? base + off : nullptr;
    off += (bytes + 255) & ~(size_t)255;
    return p;
  };
  SeqScratch sc{};
  sc.kseq = take((size_t)H * n_max * rb);
  sc.vseq = take((size_t)H * n_max * rb);
  sc.srcseq = (int32_t*)take((size_t)H * n_max * 4);
  sc.k1 = take((size_t)H * rb);
  sc.v1 = take((size_t)H * rb);
  sc.src1 = (int32_t*)take((size_t)H * 4);
  if (out) *out = sc;
  return off;
}
}  // namespace

size_t dkv_sequential_scratch_size(int32_t H, int32_t d, int32_t n_max, int32_t dtype) {
  if (H < 1 || H > kMaxH || (d != 64 && d != 128) || n_max < 1 || n_max > kMaxN) return 0;
  if (dtype != DKV_DTYPE_BF16 && dtype != DKV_DTYPE_FP32) return 0;
  return seq_layout(H, d, n_max, dtype == DKV_DTYPE_BF16, nullptr, nullptr);
}

dkv_status_t dkv_bank_update_sequential(dkv_bank_t bank, const void* Kc, const void* Vc, int32_t N, int64_t step,
                                        void* scratch, size_t scratch_bytes, void* stream) {
  NvtxRange nvtx_range("dkv_bank_update_sequential");
  if (!bank || !Kc || !Vc || !scratch) return DKV_ERR_ARG;
  if (bank->state != 0) return DKV_ERR_STATE;
  if (N < 1 || N > bank->b.n_max) return DKV_ERR_SHAPE;
  if (step < 0 || step > 0x7fffffffLL) return DKV_ERR_ARG;
  if (!aligned(Kc, 16) || !aligned(Vc, 16) || !aligned(scratch, 256)) return DKV_ERR_ARG;
  const Bank& b = bank->b;
  if (scratch_bytes < seq_layout(b.H, b.d, b.n_max, b.bf16, nullptr, nullptr)) return DKV_ERR_NOMEM;
  cudaStream_t s = (cudaStream_t)stream;
  bank->last = s;
  // every head empty: the whole block initialises the bank (Alg. 1, m = 0), as by default
  std::vector<int32_t> occ(b.H);
  if (cudaStreamSynchronize(s) != cudaSuccess ||
      cudaMemcpy(occ.data(), b.occ, sizeof(int32_t) * b.H, cudaMemcpyDeviceToHost) != cudaSuccess)
    return DKV_ERR_CUDA;
  int n_empty = 0;
  for (int h = 0; h < b.H; ++h) n_empty += occ[h] == 0;
  if (n_empty == b.H) {
    const dkv_status_t st = dkv_bank_admit(bank, Kc, Vc, N, step, stream);
    return st != DKV_OK ? st : dkv_bank_compress(bank, stream);
  }
  if (n_empty > 0) return DKV_ERR_STATE;
  // the block's order against the bank at block start, then its rows in that order
  SeqScratch sc;
  seq_layout(b.H, b.d, b.n_max, b.bf16, &sc, (char*)scratch);
  const Ws& w = bank->w;
  Timer* t = &bank->timer;
  const KParams& kp = bank->kp;
  cudaError_t e = launch_cand_norms(b, w, Kc, Vc, N, step, kp, nullptr, s, t);
  if (e == cudaSuccess && kp.order == DKV_ORDER_SCORE)
    e = bank->tc ? launch_score_tc(b, w, Kc, Vc, N, kp, s, t) : launch_score_fp32(b, w, Kc, Vc, N, kp, s, t);
  if (e == cudaSuccess) e = launch_sort(b, w, Kc, Vc, kp.order == DKV_ORDER_SOURCE, s, t);
  if (e == cudaSuccess) e = launch_seq_gather(b, w, Kc, Vc, N, sc.kseq, sc.vseq, sc.srcseq, s);
  if (e != cudaSuccess) return DKV_ERR_CUDA;
  // one one-candidate update per position j: the j-th candidate of every head
  const size_t rb = (size_t)b.d * (b.bf16 ? 2 : 4);
  for (int j = 0; j < N; ++j) {
    e = cudaMemcpy2DAsync(sc.k1, rb, sc.kseq + j * rb, (size_t)N * rb, rb, b.H, cudaMemcpyDeviceToDevice, s);
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(sc.v1, rb, sc.vseq + j * rb, (size_t)N * rb, rb, b.H, cudaMemcpyDeviceToDevice, s);
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(sc.src1, 4, sc.srcseq + j, (size_t)N * 4, 4, b.H, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return DKV_ERR_CUDA;
    dkv_status_t st = dkv_bank_admit(bank, sc.k1, sc.v1, 1, step, stream);
    if (st != DKV_OK) return st;
    bank->src_map = sc.src1;
    st = dkv_bank_compress(bank, stream);
    bank->src_map = nullptr;
    if (st != DKV_OK) return st;
  }
  return DKV_OK;
}

dkv_status_t dkv_bank_attend(dkv_bank_t bank, const void* Q, int32_t Nq, const void* Kw, const void* Vw,
                             int32_t W, void* O, void* stream) {
  NvtxRange nvtx_range("dkv_bank_attend");
  if (!bank || !Q || !O) return DKV_ERR_ARG;
  if (Nq < 1 || Nq > (1 << 20) || W < 0 || W > (1 << 20)) return DKV_ERR_SHAPE;
  if (W > 0 && (!Kw || !Vw)) return DKV_ERR_ARG;
  if (!aligned(Q, 16) || !aligned(O, 16) || (W > 0 && (!aligned(Kw, 16) || !aligned(Vw, 16)))) return DKV_ERR_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  bank->last = s;
  cudaError_t e = bank->tc ? launch_attend_tc(bank->b, bank->w.L, Q, Nq, Kw, Vw, W, O, s, &bank->timer)
                           : launch_attend_fp32(bank->b, Q, Nq, Kw, Vw, W, O, s, &bank->timer);
  return cuda_status(e);
}

dkv_status_t dkv_bank_import(dkv_bank_t bank, const int32_t* occupancy, void* stream) {
  NvtxRange nvtx_range("dkv_bank_import");
  if (!bank || !occupancy) return DKV_ERR_ARG;
  if (bank->state != 0) return DKV_ERR_STATE;
  for (int h = 0; h < bank->b.H; ++h)
    if (occupancy[h] < 0 || occupancy[h] > bank->budgets[h]) return DKV_ERR_SHAPE;
  cudaStream_t s = (cudaStream_t)stream;
  bank->last = s;
  cudaError_t e = cudaMemcpyAsync(bank->b.occ, occupancy, sizeof(int32_t) * bank->b.H, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = launch_bank_norms(bank->b, bank->w, bank->kp, s, &bank->timer);
  if (e == cudaSuccess) e = launch_inv_base(bank->b, bank->w, s);
  return cuda_status(e);
}

dkv_status_t dkv_bank_export(dkv_bank_t bank, const dkv_buffers_t* dst) {
  NvtxRange nvtx_range("dkv_bank_export");
  if (!bank || !dst) return DKV_ERR_ARG;
  if (bank->state != 0) return DKV_ERR_STATE;
  cudaStream_t s = bank->last;
  const Bank& b = bank->b;
  const size_t rows = (size_t)b.H * b.M_max;
  const size_t esz = b.bf16 ? 2 : 4;
  struct Item {
    void* to;
    const void* from;
    size_t bytes;
  } items[] = {
      {dst->k, b.k, rows * b.d * esz},          {dst->v, b.v, rows * b.d * esz},
      {dst->rho, b.rho, rows * 4},              {dst->base, b.base, rows * 4},
      {dst->prov_step, b.prov_step, rows * 8},  {dst->prov_src, b.prov_src, rows * 4},
      {dst->occupancy, b.occ, (size_t)b.H * 4},
  };
  cudaError_t e = cudaSuccess;
  for (const Item& it : items)   // one copy per array; the direction follows from the pointers
    if (e == cudaSuccess && it.to) e = cudaMemcpyAsync(it.to, it.from, it.bytes, cudaMemcpyDefault, s);
  const cudaError_t es = cudaStreamSynchronize(s);
  return cuda_status(e != cudaSuccess ? e : es);
}

dkv_status_t dkv_bank_sync(dkv_bank_t bank) {
  if (!bank) return DKV_ERR_ARG;
  cudaError_t e = cudaStreamSynchronize(bank->last);
  if (e != cudaSuccess) return DKV_ERR_CUDA;
  int32_t err = 0;
  e = cudaMemcpy(&err, &bank->w.L->err, sizeof(int32_t), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return DKV_ERR_CUDA;
  if (err != 0) {
    const int32_t zero[2] = {0, 0};
    cudaMemcpy(&bank->w.L->err, zero, sizeof(zero), cudaMemcpyHostToDevice);
    return err == DEV_TIMEOUT ? DKV_ERR_TIMEOUT : DKV_ERR_DEVICE;
  }
  return DKV_OK;
}

dkv_status_t dkv_bank_stats(dkv_bank_t bank, dkv_layer_stats_t* layer, dkv_head_stats_t* heads) {
  if (!bank || !layer) return DKV_ERR_ARG;
  if (cudaStreamSynchronize(bank->last) != cudaSuccess) return DKV_ERR_CUDA;
  std::vector<DevLayer> L(bank->n_layers);
  if (cudaMemcpy(L.data(), bank->w.L, sizeof(DevLayer) * bank->n_layers, cudaMemcpyDeviceToHost) != cudaSuccess)
    return DKV_ERR_CUDA;
  for (int l = 0; l < bank->n_layers; ++l) {
    layer[l].r_star = L[l].r_star;
    layer[l].rmax = L[l].rmax;
    layer[l].n_candidates = L[l].N;
    layer[l].empty_init = L[l].empty_all;
  }
  if (heads) {
    std::vector<DevHead> hd(bank->b.H);
    if (cudaMemcpy(hd.data(), bank->w.hd, sizeof(DevHead) * bank->b.H, cudaMemcpyDeviceToHost) != cudaSuccess)
      return DKV_ERR_CUDA;
    for (int h = 0; h < bank->b.H; ++h) {
      heads[h].occupancy_before = hd[h].m_old;
      heads[h].occupancy_after = hd[h].m_new;
      heads[h].admitted = hd[h].r;
      heads[h].evicted = hd[h].e;
      heads[h].mandatory = hd[h].n_mand;
      heads[h].pre_violators = hd[h].n_pre;
    }
  }
  return DKV_OK;
}

dkv_status_t dkv_bank_occupancy(dkv_bank_t bank, int32_t* occupancy) {
  if (!bank || !occupancy) return DKV_ERR_ARG;
  if (cudaStreamSynchronize(bank->last) != cudaSuccess) return DKV_ERR_CUDA;
  return cuda_status(cudaMemcpy(occupancy, bank->b.occ, sizeof(int32_t) * bank->b.H, cudaMemcpyDeviceToHost));
}

dkv_status_t dkv_bank_intermediates(dkv_bank_t bank, dkv_intermediates_t* out) {
  if (!bank || !out) return DKV_ERR_ARG;
  out->score = bank->w.score;
  out->perm = bank->w.perm;
  out->cross = bank->w.cross;
  out->rho_tilde = bank->w.rho_t;
  out->slot_new = bank->w.slot_new;
  out->n_max = bank->b.n_max;
  out->M_max = bank->b.M_max;
  return DKV_OK;
}

dkv_status_t dkv_bank_set_timing(dkv_bank_t bank, int32_t enable) {
  if (!bank) return DKV_ERR_ARG;
  if (enable < 0 || enable > 2) return DKV_ERR_ARG;
  bank->timer.drain();
  bank->timer.on = enable != 0;
  bank->timer.attend_only = enable == 2;
  if (!enable) {
    bank->timer.acc.clear();
    bank->timer.order.clear();
  }
  return DKV_OK;
}

dkv_status_t dkv_bank_kernel_times(dkv_bank_t bank, int32_t max_kernels, char* names, int32_t* launches,
                                   double* total_ms, int32_t* n_kernels) {
  if (!bank || !n_kernels || max_kernels < 0 || (max_kernels > 0 && (!names || !launches || !total_ms)))
    return DKV_ERR_ARG;
  bank->timer.drain();
  const auto& order = bank->timer.order;
  *n_kernels = (int32_t)order.size();
  for (int i = 0; i < (int)order.size() && i < max_kernels; ++i) {
    const auto& v = bank->timer.acc[order[i]];
    std::strncpy(names + 48 * i, order[i].c_str(), 47);
    names[48 * i + 47] = 0;
    launches[i] = v.first;
    total_ms[i] = v.second;
  }
  return DKV_OK;
}

}  // extern "C"
