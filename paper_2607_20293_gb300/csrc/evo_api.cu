// Host side of the C ABI declared in include/evo.h: configuration checks,
// weight packing, launch geometry, schedule upload and the FLOP accountant.
//
// Packing.  For cluster rank c, every unit's weights are cut into the two
// slices that CTA c multiplies by (first GEMM: columns; second GEMM: rows),
// stored contiguously per CTA and per layer so that the kernel's producer warp
// fetches each refreshed unit's slice with a few bulk copies:
//   SA  : [q_h | k_h | v_c] columns of W_qkv (h = head of c, v_c = c's value
//         columns), then rows c*E/C.. of W_o
//   CA  : q_h columns of W_q, then rows c*E/C.. of W_o
//   FFN : columns c*4E/C.. of W_1, then rows c*4E/C.. of W_2
// bf16 slices are laid out in mma.sync B-fragment order (k-tiles of 16 rows,
// n-tiles of 8 columns, 8 bytes per lane) so that a warp reads a fragment
// with one conflict-free 8-byte load per lane; fp32 slices are row-major.

#include "../../include/evo.h"
#include "evo_internal.h"

#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>
#include <vector>

using namespace evo;

struct evo_handle {
  evo_config cfg;
  GuardList guards;             // guard bands of the handle's activation buffers
  int device = 0;
  int L = 0, E = 0, U = 0, T = 0, H = 0, A = 0;
  JobParams base{};
  int shape = -1;               // compiled loop-kernel shape (evo_shapes.h)
  int max_batch = 0;
  int max_clusters = 0;
  int smem_limit = 0;
  int es = 4;
  // device memory
  float* wf32 = nullptr;
  int* woff_d = nullptr;
  uint8_t* wpack = nullptr;
  float* vec = nullptr;
  float* stab = nullptr;
  float* kstep = nullptr;
  float* kv_time = nullptr;
  float* kv_obs = nullptr;
  float* cond_scratch = nullptr;   // 6E floats per condition token
  // condition path of small calls (bf16 models): bf16 weight copy, k|v bias, partial sums, counters
  __nv_bfloat16* cond_w16 = nullptr;
  float* cond_bkv = nullptr;
  float* cond_part = nullptr;
  unsigned* cond_count = nullptr;
  void* cache = nullptr;
  uint8_t* sched = nullptr;
  size_t sched_cap = 0;
  int* status = nullptr;      // [0] = kernel status bits, [1] = schedule check of the last device lattice
  float* pop_x = nullptr;
  // host staging for host-memory schedules
  uint8_t* stage = nullptr;
  cudaEvent_t stage_ev = nullptr;
  std::vector<uint8_t> last_sched;
  int last_rows = -1;
  bool last_valid = false;
  cudaStream_t last_stream = nullptr;
  cudaEvent_t prof_start = nullptr, prof_stop = nullptr;
  int woff[W_COUNT];
  // batch-wide path (null when the configuration has none)
  WideState* wide = nullptr;
  long long wide_rows = 1024;
  int last_path = 0;
  long long last_kernels = 0;
  int last_cond_kernels = 4;          // kernels of the last call's condition path
  // Further cluster decompositions of the same model (automatic cluster size
  // only): a smaller cluster is slower per job but more clusters run at once,
  // so a call takes the decomposition with the fewest estimated job rounds.
  struct Alt {
    JobParams base{};
    int shape = -1, max_clusters = 0;
    uint8_t* wpack = nullptr;
  };
  Alt alt[2];
  int n_alt = 0;
  const JobParams* last_base = nullptr;   // decomposition of the last cluster launch
  JobParams replan{};                     // a population call's plan with fewer samples per job
  int last_mc = 0;
};

namespace {

// One NVTX range per public call (host side: covers staging and every launch
// the call issues), so that a profiler timeline groups a call's kernels.  NVTX
// is header-only and does nothing unless a tool is attached.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
};

}  // namespace

namespace evo {

cudaError_t guarded_malloc(void** user, size_t bytes, GuardList* list) {
  unsigned char* base = nullptr;
  cudaError_t e = cudaMalloc(&base, bytes + 2 * GUARD_BYTES);
  if (e != cudaSuccess) return e;
  e = cudaMemset(base, GUARD_FILL, GUARD_BYTES);
  if (e == cudaSuccess) e = cudaMemset(base + GUARD_BYTES + bytes, GUARD_FILL, GUARD_BYTES);
  if (e != cudaSuccess) {
    cudaFree(base);
    return e;
  }
  list->push_back({base, bytes});
  *user = base + GUARD_BYTES;
  return cudaSuccess;
}

void guarded_free(void* user) {
  if (user) cudaFree(static_cast<unsigned char*>(user) - GUARD_BYTES);
}

int guards_check(const GuardList& list) {
  std::vector<unsigned char> h(GUARD_BYTES);
  for (const GuardedRegion& r : list)
    for (int side = 0; side < 2; ++side) {
      const unsigned char* g = r.base + (side ? GUARD_BYTES + r.bytes : 0);
      if (cudaMemcpy(h.data(), g, GUARD_BYTES, cudaMemcpyDeviceToHost) != cudaSuccess) return -1;
      for (unsigned char c : h)
        if (c != GUARD_FILL) return 1;
    }
  return 0;
}

}  // namespace evo

namespace {

// CUDA runtime error of the most recent failed call on this thread
thread_local int g_last_cuda_error = 0;

#define EVO_CUDA(x)                                   \
  do {                                                \
    cudaError_t _e = (x);                             \
    if (_e != cudaSuccess) {                          \
      g_last_cuda_error = (int)_e;                    \
      return EVO_ERR_CUDA;                            \
    }                                                 \
  } while (0)

bool config_ok(const evo_config* c) {
  if (!c) return false;
  if (c->n_layer <= 0 || c->n_layer > 21) return false;          // 3L units tracked in a 64-bit mask
  if (c->n_emb <= 0 || c->n_head <= 0 || c->n_emb % c->n_head) return false;
  if (c->n_emb % 64 || c->n_emb > 512) return false;             // LayerNorm: float4 chunks over half a warp
  if (c->horizon <= 0 || c->horizon > 32 || c->horizon % 4) return false;
  if (c->action_dim <= 0 || c->action_dim > 16) return false;
  if (c->n_obs <= 0 || c->n_obs > 31 || c->obs_dim <= 0) return false;
  if (c->n_steps <= 0 || c->train_steps <= 0 || c->train_steps % c->n_steps) return false;
  if (c->sampler != EVO_SAMPLER_DDPM && c->sampler != EVO_SAMPLER_DDIM) return false;
  if (c->dtype != EVO_DTYPE_F32 && c->dtype != EVO_DTYPE_BF16) return false;
  if (c->empty_cache != EVO_EMPTY_ZERO && c->empty_cache != EVO_EMPTY_FORCE) return false;
  if (c->cluster < 0 || c->cluster > MAX_CLUSTER || c->job_samples < 0) return false;
  const int dh = c->n_emb / c->n_head;
  if (dh % 4 || dh > 128) return false;
  return true;
}

// The FLOP accountant is arithmetic on the shapes only: any positive model
// (the kernels' limits above do not apply)
bool flops_config_ok(const evo_config* c) {
  return c && c->n_layer > 0 && c->n_layer <= 21 && c->n_emb > 0 && c->n_head > 0 && c->n_emb % c->n_head == 0 &&
         c->horizon > 0 && c->action_dim > 0 && c->n_obs >= 0 && c->obs_dim > 0 && c->n_steps > 0 &&
         (c->empty_cache == EVO_EMPTY_ZERO || c->empty_cache == EVO_EMPTY_FORCE);
}

void weight_offsets(const evo_config* c, int* wo) {
  const int E = c->n_emb, A = c->action_dim, D = c->obs_dim, H = c->horizon, Cm = 1 + c->n_obs;
  int o = 0;
  auto take = [&](int id, int n) { wo[id] = o; o += n; };
  take(W_OBS_W, D * E);
  take(W_OBS_B, E);
  take(W_COND_POS, Cm * E);
  take(W_CM_W1, E * 4 * E);
  take(W_CM_B1, 4 * E);
  take(W_CM_W2, 4 * E * E);
  take(W_CM_B2, E);
  take(W_IN_W, A * E);
  take(W_IN_B, E);
  take(W_POS, H * E);
  wo[W_LAYER0] = o;
  int lo = 0;
  auto ltake = [&](int id, int n) { wo[id] = lo; lo += n; };
  ltake(WL_LN1G, E);
  ltake(WL_LN1B, E);
  ltake(WL_SA_WQKV, E * 3 * E);
  ltake(WL_SA_BQKV, 3 * E);
  ltake(WL_SA_WO, E * E);
  ltake(WL_SA_BO, E);
  ltake(WL_LN2G, E);
  ltake(WL_LN2B, E);
  ltake(WL_CA_WQ, E * E);
  ltake(WL_CA_BQ, E);
  ltake(WL_CA_WKV, E * 2 * E);
  ltake(WL_CA_BKV, 2 * E);
  ltake(WL_CA_WO, E * E);
  ltake(WL_CA_BO, E);
  ltake(WL_LN3G, E);
  ltake(WL_LN3B, E);
  ltake(WL_FF_W1, E * 4 * E);
  ltake(WL_FF_B1, 4 * E);
  ltake(WL_FF_W2, 4 * E * E);
  ltake(WL_FF_B2, E);
  wo[W_LAYER_STRIDE] = lo;
  o += c->n_layer * lo;
  take(W_LNF_G, E);
  take(W_LNF_B, E);
  take(W_HEAD_W, E * A);
  take(W_HEAD_B, A);
  wo[W_TOTAL] = o;
}

inline uint16_t f2bf(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7f800000u) == 0x7f800000u) return (uint16_t)(u >> 16);   // inf / nan kept
  u += 0x7fffu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

inline int rup(int x, int a) { return (x + a - 1) / a * a; }

// decomposition constraints for a cluster of C CTAs
bool cluster_ok(const evo_config* c, int C) {
  const int E = c->n_emb, dh = E / c->n_head;
  if (C < 1 || E % C) return false;
  const int Ec = E / C, hid = 4 * E / C;
  if (Ec % 4 || Ec > dh || dh % Ec || Ec > 64) return false;
  if (c->dtype == EVO_DTYPE_BF16 && (Ec % 8 || hid % 16)) return false;
  return true;
}

// sampler coefficients per loop step: inv_sqrt_ab, sqrt_1mab, c_x0, c_xt, sigma, sqrt_ab, sqrt_ab_prev, sqrt_1mab_prev
void sampler_table(const evo_config* c, std::vector<float>& tab, std::vector<float>& kstep) {
  const int Ttr = c->train_steps, T = c->n_steps, stride = Ttr / T;
  std::vector<double> ac(Ttr);
  double prod = 1.0;
  const double pi = 3.14159265358979323846;
  auto f = [&](double s) {
    const double v = std::cos((s + 0.008) / 1.008 * pi / 2);
    return v * v;
  };
  for (int i = 0; i < Ttr; ++i) {
    const double beta = std::min(1.0 - f((i + 1) / (double)Ttr) / f(i / (double)Ttr), 0.999);
    prod *= (1.0 - beta);
    ac[i] = prod;
  }
  tab.assign((size_t)T * 8, 0.f);
  kstep.assign(T, 0.f);
  for (int t = 0; t < T; ++t) {
    const int k = (T - 1 - t) * stride;
    const int prev = k - stride;
    const double ab = ac[k], abp = prev >= 0 ? ac[prev] : 1.0;
    const double alpha = ab / abp, beta = 1.0 - alpha;
    float* r = &tab[(size_t)t * 8];
    r[0] = (float)(1.0 / std::sqrt(ab));
    r[1] = (float)std::sqrt(1.0 - ab);
    r[2] = (float)(std::sqrt(abp) * beta / (1.0 - ab));
    r[3] = (float)(std::sqrt(alpha) * (1.0 - abp) / (1.0 - ab));
    const double var = std::max((1.0 - abp) / (1.0 - ab) * beta, 1e-20);
    r[4] = k > 0 ? (float)std::sqrt(var) : 0.f;
    r[5] = (float)std::sqrt(ab);
    r[6] = (float)std::sqrt(abp);
    r[7] = (float)std::sqrt(1.0 - abp);
    kstep[t] = (float)k;
  }
}

int64_t flops_of(const evo_config* c, const uint8_t* S, int rows) {
  const int64_t E = c->n_emb, H = c->horizon, Cm = 1 + c->n_obs, A = c->action_dim, D = c->obs_dim;
  const int64_t fsa = 2 * H * E * 3 * E + 4 * H * H * E + 2 * H * E * E;
  const int64_t fca = 2 * H * E * E + 4 * Cm * E * E + 4 * H * Cm * E + 2 * H * E * E;
  const int64_t fff = 16 * H * E * E;
  const int64_t fix = 2 * c->n_obs * D * E + 16 * Cm * E * E + 4 * H * A * E;
  const int T = c->n_steps, U = 3 * c->n_layer;
  int64_t total = (int64_t)T * fix;
  for (int b = 0; b < U; ++b) {
    const int row = rows == U ? b : b / 3;
    int64_t n = 0;
    for (int t = 0; t < T; ++t) n += S[(size_t)row * T + t];
    if (c->empty_cache == EVO_EMPTY_FORCE && T > 0 && S[(size_t)row * T] == 0) n += 1;
    const int u = b % 3;
    total += n * (u == 0 ? fsa : (u == 1 ? fca : fff));
  }
  return total;
}

bool is_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

bool lattice_ok(const uint8_t* S, size_t n) {
  for (size_t i = 0; i < n; ++i)
    if (S[i] > 1) return false;
  return true;
}

inline bool pow2(int x) { return x > 0 && (x & (x - 1)) == 0; }
inline int ilog2(int x) {
  int l = 0;
  while ((1 << l) < x) ++l;
  return l;
}

// Fill p's decomposition fields for g samples per job and the ring geometry
// (slot bytes, slots) of the compiled shape; returns shared bytes or -1.
int plan(const evo_config* c, int C, int g, int slot, int nslot, int smem_limit, JobParams& p) {
  const int E = c->n_emb, dh = E / c->n_head, H = c->horizon;
  const int es = c->dtype == EVO_DTYPE_BF16 ? 2 : 4;
  auto r84 = [](int x) { return x + ((12 - x % 8) % 8); };      // smallest y >= x with y % 8 == 4
  p.L = c->n_layer;
  p.E = E;
  p.nh = c->n_head;
  p.dh = dh;
  p.H = H;
  p.A = c->action_dim;
  p.n_obs = c->n_obs;
  p.T = c->n_steps;
  p.U = 3 * c->n_layer;
  p.Cm = 1 + c->n_obs;
  p.C = C;
  p.Ec = E / C;
  p.hid = 4 * E / C;
  p.g = g;
  p.M = g * H;
  p.Mp = rup(p.M, 16);
  if (!pow2(p.Ec) || !pow2(H) || !pow2(g)) return -1;
  p.lEc = ilog2(p.Ec);
  p.lH = ilog2(H);
  p.blk = p.M * p.Ec + 4;
  p.lda = es == 2 ? E + 8 : E + 4;
  p.n1[0] = 2 * dh + p.Ec;
  p.n1[1] = dh;
  p.n1[2] = p.hid;
  p.ldg1 = r84(p.n1[0]);
  p.kvw = r84(dh + p.Ec);
  p.kp_o = rup(p.Ec, 16);
  p.kp_h = rup(p.hid, 16);
  p.ldh = es == 2 ? p.kp_h + 8 : p.kp_h;
  p.ldo = es == 2 ? p.kp_o + 8 : p.kp_o;
  for (int u = 0; u < 3; ++u) p.hdr1[u] = rup(p.n1[u] + p.Ec, 4) * 4;
  p.sampler = c->sampler;
  p.force = c->empty_cache == EVO_EMPTY_FORCE;
  p.invE = 1.0f / (float)E;
  if (p.Cm > 32 || p.M * p.Ec > 4 * NCT) return -1;
  if (g * p.Cm * (dh / 4 + p.Ec / 4) > NCT) return -1;     // one memory key/value chunk per thread
  if (es == 2 && p.Cm > 16) return -1;                      // tensor-core attention pads memory keys to 16
  if (p.A > 16) return -1;                                  // action dimensions of the fused head
  // head partials per row: sum, sum of squares, A dots (4-padded)
  p.npr = rup(2 + p.A, 4);
  if (es == 2) {
    if (p.Mp > 32) return -1;
  } else {
    const int nmax = std::max(std::max(p.n1[0], p.n1[2]), E);
    if (p.M * nmax > 16 * NCT) return -1;
  }
  // a ring slot must hold any piece-1 header plus one k-tile, and one k-tile of piece 2
  int need = 16 * E * es;
  for (int u = 0; u < 3; ++u) need = std::max(need, p.hdr1[u] + 16 * p.n1[u] * es);
  if (slot < need) return -1;
  p.slot_bytes = slot;
  p.nslot = nslot;
  p.wait_limit = WAIT_CYCLES_DEFAULT;
  // preference: caches on chip, per-step memory keys/values, double-buffered
  // head exchange, head weights on chip
  for (int cache_smem = 1; cache_smem >= 0; --cache_smem)
    for (int kvall = 1; kvall >= 0; --kvall)
      for (int head_sep = 1; head_sep >= 0; --head_sep) {
        if (!head_sep && p.M * p.npr > p.blk) continue;     // one head landing block per ablk block
        p.kv_slots = kvall ? p.L : 1;
        p.head_sep = head_sep;
        const int total = smem_layout(p, es, cache_smem);
        if (total <= smem_limit) return total;
      }
  return -1;
}

}  // namespace

extern "C" {

const char* evo_status_string(evo_status s) {
  switch (s) {
    case EVO_OK: return "ok";
    case EVO_ERR_ARG: return "invalid argument";
    case EVO_ERR_SHAPE: return "unsupported shape or batch";
    case EVO_ERR_SCHEDULE: return "invalid schedule lattice";
    case EVO_ERR_CUDA: return "CUDA runtime error";
    case EVO_ERR_TIMEOUT: return "device wait timed out";
    case EVO_ERR_OOM: return "device out of memory";
    case EVO_ERR_UNSUPPORTED: return "unsupported on this device";
    case EVO_ERR_CORRUPT: return "guard band overwritten or device index check failed";
  }
  return "unknown status";
}

size_t evo_weight_count(const evo_config* cfg) {
  if (!config_ok(cfg)) return 0;
  int wo[W_COUNT];
  weight_offsets(cfg, wo);
  return (size_t)wo[W_TOTAL];
}

evo_status evo_flops_cfg(const evo_config* cfg, const uint8_t* S, int32_t S_rows, int64_t* out) {
  if (!flops_config_ok(cfg) || !S || !out) return EVO_ERR_ARG;
  const int U = 3 * cfg->n_layer;
  if (S_rows != U && S_rows != cfg->n_layer) return EVO_ERR_SCHEDULE;
  if (!lattice_ok(S, (size_t)S_rows * cfg->n_steps)) return EVO_ERR_SCHEDULE;
  *out = flops_of(cfg, S, S_rows);
  return EVO_OK;
}

evo_status evo_flops(const evo_handle* h, const uint8_t* S, int32_t S_rows, int64_t* out) {
  if (!h) return EVO_ERR_ARG;
  return evo_flops_cfg(&h->cfg, S, S_rows, out);
}

evo_status evo_schedule_from_positions(const int16_t* bt, int32_t K, int32_t n_units, int32_t T, uint8_t* S_out) {
  if ((!bt && K > 0) || !S_out || K < 0 || n_units <= 0 || T <= 0) return EVO_ERR_ARG;
  std::vector<uint8_t> s((size_t)n_units * T, 0);
  for (int i = 0; i < K; ++i) {
    const int b = bt[2 * i], t = bt[2 * i + 1];
    if (b < 0 || b >= n_units || t < 0 || t >= T) return EVO_ERR_SCHEDULE;
    uint8_t& cell = s[(size_t)b * T + t];
    if (cell) return EVO_ERR_SCHEDULE;
    cell = 1;
  }
  std::memcpy(S_out, s.data(), s.size());
  return EVO_OK;
}

evo_status evo_schedule_fixed_interval(int32_t n_units, int32_t T, int32_t M, uint8_t* S_out) {
  if (!S_out || n_units <= 0 || T <= 0 || M < 1 || M > T) return EVO_ERR_ARG;
  std::memset(S_out, 0, (size_t)n_units * T);
  for (int b = 0; b < n_units; ++b)
    for (int i = 0; i < M; ++i) S_out[(size_t)b * T + (long long)i * T / M] = 1;
  return EVO_OK;
}

evo_status evo_get_launch_info(const evo_handle* h, int32_t* cluster, int32_t* job_samples, int32_t* max_clusters,
                               int32_t* smem_bytes) {
  if (!h) return EVO_ERR_ARG;
  const JobParams& b = h->last_base ? *h->last_base : h->base;
  if (cluster) *cluster = b.C;
  if (job_samples) *job_samples = b.g;
  if (max_clusters) *max_clusters = h->last_base ? h->last_mc : h->max_clusters;
  if (smem_bytes) *smem_bytes = b.sm.total;
  return EVO_OK;
}

evo_status evo_destroy(evo_handle* h) {
  if (!h) return EVO_ERR_ARG;
  wide_destroy(h->wide);
  cudaFree(h->wf32);
  cudaFree(h->woff_d);
  cudaFree(h->wpack);
  for (int i = 0; i < h->n_alt; ++i) cudaFree(h->alt[i].wpack);
  cudaFree(h->vec);
  cudaFree(h->stab);
  cudaFree(h->kstep);
  cudaFree(h->kv_time);
  cudaFree(h->kv_obs);
  cudaFree(h->cond_scratch);
  cudaFree(h->cond_w16);
  cudaFree(h->cond_bkv);
  cudaFree(h->cond_part);
  cudaFree(h->cond_count);
  guarded_free(h->cache);
  cudaFree(h->sched);
  cudaFree(h->status);
  cudaFree(h->pop_x);
  if (h->stage) cudaFreeHost(h->stage);
  if (h->stage_ev) cudaEventDestroy(h->stage_ev);
  delete h;
  return EVO_OK;
}

evo_status evo_create(const float* weights, size_t n_floats, const evo_config* cfg, int32_t max_batch,
                      evo_handle** out) {
  if (!weights || !cfg || !out || max_batch <= 0) return EVO_ERR_ARG;
  *out = nullptr;
  if (!config_ok(cfg)) return EVO_ERR_SHAPE;
  if (n_floats != evo_weight_count(cfg)) return EVO_ERR_SHAPE;
  int dev = 0;
  EVO_CUDA(cudaGetDevice(&dev));
  int cc_major = 0, smem_optin = 0, cluster_ok_attr = 0;
  EVO_CUDA(cudaDeviceGetAttribute(&cc_major, cudaDevAttrComputeCapabilityMajor, dev));
  EVO_CUDA(cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev));
  EVO_CUDA(cudaDeviceGetAttribute(&cluster_ok_attr, cudaDevAttrClusterLaunch, dev));
  if (cc_major < 10 || !cluster_ok_attr) return EVO_ERR_UNSUPPORTED;

  evo_handle* h = new evo_handle();
  h->cfg = *cfg;
  h->device = dev;
  h->L = cfg->n_layer;
  h->E = cfg->n_emb;
  h->U = 3 * cfg->n_layer;
  h->T = cfg->n_steps;
  h->H = cfg->horizon;
  h->A = cfg->action_dim;
  h->es = cfg->dtype == EVO_DTYPE_BF16 ? 2 : 4;
  h->max_batch = max_batch;
  h->smem_limit = smem_optin;
  weight_offsets(cfg, h->woff);
  const int E = h->E, L = h->L, U = h->U, T = h->T, H = h->H, A = h->A;
  const int dh = E / cfg->n_head;

  // ---- decomposition ------------------------------------------------------
  const int g = cfg->job_samples > 0 ? cfg->job_samples : 1;
  int C = cfg->cluster, slot = 0, nslot = 0;
  if (C == 0) {
    // the largest cluster with a compiled kernel for this shape
    const int cap = std::min(MAX_CLUSTER, std::max(1, E / 16));
    for (C = cap; C >= 1; C >>= 1)
      if (cluster_ok(cfg, C) && shape_find(cfg->dtype, E, cfg->n_head, H, C, g, &slot, &nslot) >= 0) break;
  }
  if (C < 1 || !cluster_ok(cfg, C)) {
    delete h;
    return EVO_ERR_SHAPE;
  }
  h->shape = shape_find(cfg->dtype, E, cfg->n_head, H, C, g, &slot, &nslot);
  if (h->shape < 0) {
    delete h;
    return EVO_ERR_UNSUPPORTED;
  }
  JobParams& p = h->base;
  const int smem = plan(cfg, C, g, slot, nslot, smem_optin, p);
  if (smem < 0) {
    delete h;
    return EVO_ERR_UNSUPPORTED;
  }
  {
    int mc = 0;
    cudaError_t e = job_kernel_prepare(h->shape, smem, &mc);
    if (e != cudaSuccess || mc <= 0) {
      cudaGetLastError();
      delete h;
      return EVO_ERR_UNSUPPORTED;
    }
    h->max_clusters = mc;
  }

  // ---- weights -------------------------------------------------------------
  auto fail = [&](evo_status s) {
    evo_destroy(h);
    return s;
  };
  const size_t wbytes = n_floats * sizeof(float);
  if (cudaMalloc(&h->wf32, wbytes) != cudaSuccess) return fail(EVO_ERR_OOM);
  if (cudaMemcpy(h->wf32, weights, wbytes, cudaMemcpyHostToDevice) != cudaSuccess) return fail(EVO_ERR_CUDA);
  if (cudaMalloc(&h->woff_d, sizeof(h->woff)) != cudaSuccess) return fail(EVO_ERR_OOM);
  if (cudaMemcpy(h->woff_d, h->woff, sizeof(h->woff), cudaMemcpyHostToDevice) != cudaSuccess)
    return fail(EVO_ERR_CUDA);

  const int* wo = h->woff;
  auto W = [&](int id) { return weights + wo[id]; };
  auto WL = [&](int l, int id) { return weights + wo[W_LAYER0] + (size_t)l * wo[W_LAYER_STRIDE] + wo[id]; };
  const int es = h->es;
  // packed weights of one decomposition (fills p.poff, p.layer_stride, p.cta_stride)
  auto pack_for = [&](JobParams& p, uint8_t** dst) -> evo_status {
  const int C = p.C;
  const int Ec = p.Ec, hid = p.hid;
  // piece sizes (bytes) and offsets within one layer block
  const long long sz[3][2] = {{p.hdr1[0] + (long long)E * p.n1[0] * es, (long long)p.kp_o * E * es},
                              {p.hdr1[1] + (long long)E * p.n1[1] * es, (long long)p.kp_o * E * es},
                              {p.hdr1[2] + (long long)E * p.n1[2] * es, (long long)p.kp_h * E * es}};
  long long off = 0;
  for (int u = 0; u < 3; ++u)
    for (int q = 0; q < 2; ++q) {
      p.poff[u][q] = off;
      off += sz[u][q];
    }
  p.layer_stride = off;
  p.cta_stride = off * L;
  std::vector<uint8_t> pack((size_t)p.cta_stride * C, 0);
  auto put = [&](uint8_t* dst, int K, int N, auto get) {
    if (es == 2) {
      uint16_t* d = reinterpret_cast<uint16_t*>(dst);
      const int NT = N / 8;
      for (int kt = 0; kt < K / 16; ++kt)
        for (int nt = 0; nt < NT; ++nt)
          for (int lane = 0; lane < 32; ++lane)
            for (int i = 0; i < 4; ++i) {
              const int k = kt * 16 + (lane % 4) * 2 + (i % 2) + (i / 2) * 8;
              const int n = nt * 8 + lane / 4;
              d[(((size_t)kt * NT + nt) * 32 + lane) * 4 + i] = f2bf(get(k, n));
            }
    } else {
      float* d = reinterpret_cast<float*>(dst);
      for (int k = 0; k < K; ++k)
        for (int n = 0; n < N; ++n) d[(size_t)k * N + n] = get(k, n);
    }
  };
  // piece 1 = [float32 header][k-tiles], header = the first GEMM's bias
  // columns and this CTA's columns of the second GEMM's bias; piece 2 =
  // [k-tiles].  The unit's LayerNorm affine is folded into the first GEMM:
  // LN(a) W + b = xhat (g o W) + (beta W + b), xhat = (a - mean) * rstd, so the
  // k-tiles hold g_k W[k][n] and the bias beta W + b (summed in double).
  auto header = [&](uint8_t* dst, const float* beta, const float* bias, int nbias, auto colmap, auto wcol,
                    const float* bias2) {
    float* d = reinterpret_cast<float*>(dst);
    for (int i = 0; i < nbias; ++i) {
      double v = (double)bias[colmap(i)];
      for (int k = 0; k < E; ++k) v += (double)beta[k] * (double)wcol(k, i);
      d[i] = (float)v;
    }
    for (int i = 0; i < Ec; ++i) d[nbias + i] = bias2[i];
  };
  for (int c = 0; c < C; ++c) {
    const int h0 = (c * Ec) / dh;
    auto qkv_col = [&](int n) { return n < dh ? h0 * dh + n : (n < 2 * dh ? E + h0 * dh + (n - dh) : 2 * E + c * Ec + (n - 2 * dh)); };
    for (int l = 0; l < L; ++l) {
      uint8_t* base = pack.data() + (size_t)c * p.cta_stride + (size_t)l * p.layer_stride;
      const float* wqkv = WL(l, WL_SA_WQKV);
      const float* wo1 = WL(l, WL_SA_WO);
      const float* wq = WL(l, WL_CA_WQ);
      const float* wo2 = WL(l, WL_CA_WO);
      const float* w1 = WL(l, WL_FF_W1);
      const float* w2 = WL(l, WL_FF_W2);
      const float* g1 = WL(l, WL_LN1G);
      const float* g2 = WL(l, WL_LN2G);
      const float* g3 = WL(l, WL_LN3G);
      auto sa_w = [&](int k, int n) { return wqkv[(size_t)k * 3 * E + qkv_col(n)]; };
      auto ca_w = [&](int k, int n) { return wq[(size_t)k * E + h0 * dh + n]; };
      auto ff_w = [&](int k, int n) { return w1[(size_t)k * 4 * E + c * hid + n]; };
      // SA
      header(base + p.poff[0][0], WL(l, WL_LN1B), WL(l, WL_SA_BQKV), p.n1[0], qkv_col, sa_w, WL(l, WL_SA_BO) + c * Ec);
      put(base + p.poff[0][0] + p.hdr1[0], E, p.n1[0], [&](int k, int n) { return g1[k] * sa_w(k, n); });
      put(base + p.poff[0][1], p.kp_o, E, [&](int k, int n) { return k < Ec ? wo1[(size_t)(c * Ec + k) * E + n] : 0.f; });
      // CA
      header(base + p.poff[1][0], WL(l, WL_LN2B), WL(l, WL_CA_BQ), p.n1[1], [&](int n) { return h0 * dh + n; }, ca_w,
             WL(l, WL_CA_BO) + c * Ec);
      put(base + p.poff[1][0] + p.hdr1[1], E, p.n1[1], [&](int k, int n) { return g2[k] * ca_w(k, n); });
      put(base + p.poff[1][1], p.kp_o, E, [&](int k, int n) { return k < Ec ? wo2[(size_t)(c * Ec + k) * E + n] : 0.f; });
      // FFN
      header(base + p.poff[2][0], WL(l, WL_LN3B), WL(l, WL_FF_B1), p.n1[2], [&](int n) { return c * hid + n; }, ff_w,
             WL(l, WL_FF_B2) + c * Ec);
      put(base + p.poff[2][0] + p.hdr1[2], E, p.n1[2], [&](int k, int n) { return g3[k] * ff_w(k, n); });
      put(base + p.poff[2][1], p.kp_h, E, [&](int k, int n) { return k < hid ? w2[(size_t)(c * hid + k) * E + n] : 0.f; });
    }
  }
  if (cudaMalloc(dst, pack.size()) != cudaSuccess) return EVO_ERR_OOM;
  if (cudaMemcpy(*dst, pack.data(), pack.size(), cudaMemcpyHostToDevice) != cudaSuccess) return EVO_ERR_CUDA;
  return EVO_OK;
  };
  {
    const evo_status ps = pack_for(p, &h->wpack);
    if (ps != EVO_OK) return fail(ps);
  }
  // smaller-cluster decompositions (automatic cluster size, one sample per job)
  if (cfg->cluster == 0 && g == 1) {
    for (int C2 = C / 2; C2 >= 4 && h->n_alt < 2; C2 /= 2) {
      int slot2 = 0, nslot2 = 0;
      if (!cluster_ok(cfg, C2)) continue;
      const int sh = shape_find(cfg->dtype, E, cfg->n_head, H, C2, 1, &slot2, &nslot2);
      if (sh < 0) continue;
      evo_handle::Alt& a = h->alt[h->n_alt];
      const int sm2 = plan(cfg, C2, 1, slot2, nslot2, smem_optin, a.base);
      if (sm2 < 0) continue;
      int mc = 0;
      if (job_kernel_prepare(sh, sm2, &mc) != cudaSuccess || mc <= 0) {
        cudaGetLastError();
        continue;
      }
      a.shape = sh;
      a.max_clusters = mc;
      const evo_status ps = pack_for(a.base, &a.wpack);
      ++h->n_alt;                                     // evo_destroy frees its weights
      if (ps != EVO_OK) return fail(ps);
    }
  }

  // float32 vectors
  std::vector<float> vec;
  auto vtake = [&](long long& dst, size_t n) {
    dst = (long long)vec.size();
    vec.resize(vec.size() + n, 0.f);
  };
  vtake(p.v_inw, (size_t)A * E);
  vtake(p.v_inb, E);
  vtake(p.v_pos, (size_t)H * E);
  vtake(p.v_lnfg, E);
  vtake(p.v_lnfb, E);
  vtake(p.v_headw, (size_t)E * A);
  vtake(p.v_headb, A);
  vtake(p.v_headG, A);
  vtake(p.v_headB, A);
  std::memcpy(&vec[p.v_inw], W(W_IN_W), (size_t)A * E * 4);
  std::memcpy(&vec[p.v_inb], W(W_IN_B), E * 4);
  std::memcpy(&vec[p.v_pos], W(W_POS), (size_t)H * E * 4);
  std::memcpy(&vec[p.v_lnfg], W(W_LNF_G), E * 4);
  std::memcpy(&vec[p.v_lnfb], W(W_LNF_B), E * 4);
  for (int e = 0; e < E; ++e)   // W_head transposed: [A][E]
    for (int a = 0; a < A; ++a) vec[p.v_headw + (size_t)a * E + e] = W(W_HEAD_W)[(size_t)e * A + a];
  std::memcpy(&vec[p.v_headb], W(W_HEAD_B), A * 4);
  // LN_f folded into the head: (LN(a) . W)_a = rstd (sum_e a_e g_e W_ea - mean G_a) + B_a
  for (int a = 0; a < A; ++a) {
    double G = 0.0, B = 0.0;
    for (int e = 0; e < E; ++e) {
      G += (double)W(W_LNF_G)[e] * (double)W(W_HEAD_W)[(size_t)e * A + a];
      B += (double)W(W_LNF_B)[e] * (double)W(W_HEAD_W)[(size_t)e * A + a];
    }
    vec[p.v_headG + a] = (float)G;
    vec[p.v_headB + a] = (float)B;
  }
  if (cudaMalloc(&h->vec, vec.size() * 4) != cudaSuccess) return fail(EVO_ERR_OOM);
  if (cudaMemcpy(h->vec, vec.data(), vec.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess)
    return fail(EVO_ERR_CUDA);

  // sampler table, timestep-token keys/values
  std::vector<float> tab, kst;
  sampler_table(cfg, tab, kst);
  if (cudaMalloc(&h->stab, tab.size() * 4) != cudaSuccess) return fail(EVO_ERR_OOM);
  if (cudaMalloc(&h->kstep, kst.size() * 4) != cudaSuccess) return fail(EVO_ERR_OOM);
  cudaMemcpy(h->stab, tab.data(), tab.size() * 4, cudaMemcpyHostToDevice);
  cudaMemcpy(h->kstep, kst.data(), kst.size() * 4, cudaMemcpyHostToDevice);
  if (cudaMalloc(&h->kv_time, (size_t)T * L * 2 * E * 4) != cudaSuccess) return fail(EVO_ERR_OOM);
  // per-call buffers
  const size_t cap_samples = (size_t)max_batch + 32;
  const size_t cond_tokens = std::max((size_t)T, cap_samples * cfg->n_obs);
  if (cudaMalloc(&h->cond_scratch, cond_tokens * 6 * E * sizeof(float)) != cudaSuccess) return fail(EVO_ERR_OOM);
  if (launch_time_table(h->wf32, h->woff_d, h->woff, h->kstep, T, L, E, h->cond_scratch, h->kv_time, 0) != cudaSuccess)
    return fail(EVO_ERR_CUDA);

  if (cudaMalloc(&h->kv_obs, cap_samples * cfg->n_obs * L * 2 * E * 4) != cudaSuccess) return fail(EVO_ERR_OOM);
  if (es == 2 && cond_fast_ok(E, L, 1)) {
    // bf16 copy of the condition matmuls for calls of a few tokens
    std::vector<uint16_t> w16((size_t)8 * E * E + (size_t)E * L * 2 * E);
    std::vector<float> bkv((size_t)L * 2 * E);
    const float* w1 = W(W_CM_W1);
    const float* w2 = W(W_CM_W2);
    for (size_t i = 0; i < (size_t)4 * E * E; ++i) w16[i] = f2bf(w1[i]);
    for (size_t i = 0; i < (size_t)4 * E * E; ++i) w16[(size_t)4 * E * E + i] = f2bf(w2[i]);
    uint16_t* wkv = w16.data() + (size_t)8 * E * E;
    for (int l = 0; l < L; ++l) {
      const float* src = WL(l, WL_CA_WKV);
      for (int k = 0; k < E; ++k)
        for (int j = 0; j < 2 * E; ++j) wkv[(size_t)k * L * 2 * E + (size_t)l * 2 * E + j] = f2bf(src[(size_t)k * 2 * E + j]);
      std::memcpy(&bkv[(size_t)l * 2 * E], WL(l, WL_CA_BKV), (size_t)2 * E * 4);
    }
    if (cudaMalloc(&h->cond_w16, w16.size() * 2) != cudaSuccess) return fail(EVO_ERR_OOM);
    if (cudaMalloc(&h->cond_bkv, bkv.size() * 4) != cudaSuccess) return fail(EVO_ERR_OOM);
    if (cudaMalloc(&h->cond_part, cond_fast_part_floats(E, L, 32) * 4) != cudaSuccess) return fail(EVO_ERR_OOM);
    if (cudaMalloc(&h->cond_count, 768 * sizeof(unsigned)) != cudaSuccess) return fail(EVO_ERR_OOM);
    cudaMemcpy(h->cond_w16, w16.data(), w16.size() * 2, cudaMemcpyHostToDevice);
    cudaMemcpy(h->cond_bkv, bkv.data(), bkv.size() * 4, cudaMemcpyHostToDevice);
    cudaMemset(h->cond_count, 0, 768 * sizeof(unsigned));
  }
  if (guarded_malloc(&h->cache, cap_samples * H * (size_t)U * E * es, &h->guards) != cudaSuccess)
    return fail(EVO_ERR_OOM);
  h->sched_cap = cap_samples * U * T;
  if (cudaMalloc(&h->sched, h->sched_cap) != cudaSuccess) return fail(EVO_ERR_OOM);
  if (cudaMalloc(&h->status, 2 * sizeof(int)) != cudaSuccess) return fail(EVO_ERR_OOM);
  cudaMemset(h->status, 0, 2 * sizeof(int));
  if (cudaMalloc(&h->pop_x, cap_samples * H * A * 4) != cudaSuccess) return fail(EVO_ERR_OOM);
  if (cudaMallocHost(&h->stage, h->sched_cap) != cudaSuccess) return fail(EVO_ERR_OOM);
  if (cudaEventCreateWithFlags(&h->stage_ev, cudaEventDisableTiming) != cudaSuccess) return fail(EVO_ERR_CUDA);
  if (cfg->wide_rows >= 0 && wide_supported(cfg)) {
    // every call's rows (population: (P+1) * N_obs samples) and lattices fit
    const int ws = wide_create(&h->wide, cfg, weights, h->wf32, h->woff, (long long)max_batch * H, max_batch + 1);
    if (ws == EVO_ERR_OOM || ws == EVO_ERR_CUDA) return fail((evo_status)ws);
    if (cfg->wide_rows > 0) h->wide_rows = cfg->wide_rows;
  }
  if (cudaDeviceSynchronize() != cudaSuccess) return fail(EVO_ERR_CUDA);

  p.stab = h->stab;
  p.kv_time = h->kv_time;
  p.kv_obs = h->kv_obs;
  p.wpack = h->wpack;
  p.vec = h->vec;
  p.cache = h->cache;
  p.status = h->status;
  for (int i = 0; i < h->n_alt; ++i) {
    JobParams& q = h->alt[i].base;
    q.v_inw = p.v_inw;
    q.v_inb = p.v_inb;
    q.v_pos = p.v_pos;
    q.v_lnfg = p.v_lnfg;
    q.v_lnfb = p.v_lnfb;
    q.v_headw = p.v_headw;
    q.v_headb = p.v_headb;
    q.v_headG = p.v_headG;
    q.v_headB = p.v_headB;
    q.stab = p.stab;
    q.kv_time = p.kv_time;
    q.kv_obs = p.kv_obs;
    q.wpack = h->alt[i].wpack;
    q.vec = p.vec;
    q.cache = p.cache;
    q.status = p.status;
  }
  // with a cluster of 4 at hand the cluster path stays ahead of the batch-wide
  // one up to about 2048 action-token rows
  if (cfg->wide_rows == 0 && h->n_alt > 0 && h->alt[h->n_alt - 1].base.C <= 4) h->wide_rows = 2048;
  *out = h;
  return EVO_OK;
}

}  // extern "C"

namespace {

// The observation tokens' keys/values of a call: the spread-out bf16 kernels
// for a few tokens, else the general ones.
cudaError_t obs_cond(evo_handle* h, const float* obs, int N, float* scratch, float* kv_obs, cudaStream_t st) {
  h->last_cond_kernels = 4;
  if (h->cond_w16 && cond_fast_ok(h->E, h->L, (long long)N * h->cfg.n_obs)) {
    h->last_cond_kernels = 3;
    return launch_obs_cond_fast(h->wf32, h->woff, h->cond_w16, h->cond_bkv, obs, N, h->cfg.n_obs, h->cfg.obs_dim,
                                h->L, h->E, scratch, h->cond_part, h->cond_count, kv_obs, st);
  }
  return launch_obs_cond(h->wf32, h->woff_d, h->woff, obs, N, h->cfg.n_obs, h->cfg.obs_dim, h->L, h->E, scratch,
                         kv_obs, st);
}

// Copy n_sched lattices (+ optionally an all-ones reference lattice) into the
// handle's device buffer.  Host lattices are validated here; device lattices
// are checked by a kernel that sets status[1].
evo_status stage_schedules(evo_handle* h, const uint8_t* S, int n_sched, int rows, bool add_ones, cudaStream_t st,
                           const int** err_out) {
  const size_t one = (size_t)rows * h->T;
  const size_t bytes = one * n_sched;
  const size_t total = bytes + (add_ones ? one : 0);
  if (total > h->sched_cap) return EVO_ERR_SHAPE;
  *err_out = nullptr;
  if (!is_device_ptr(S)) {
    if (!lattice_ok(S, bytes)) return EVO_ERR_SCHEDULE;
    const bool same = h->last_valid && h->last_rows == rows && h->last_sched.size() == total &&
                      std::memcmp(h->last_sched.data(), S, bytes) == 0;
    if (same) return EVO_OK;
    EVO_CUDA(cudaEventSynchronize(h->stage_ev));
    std::memcpy(h->stage, S, bytes);
    if (add_ones) std::memset(h->stage + bytes, 1, one);
    EVO_CUDA(cudaMemcpyAsync(h->sched, h->stage, total, cudaMemcpyHostToDevice, st));
    EVO_CUDA(cudaEventRecord(h->stage_ev, st));
    h->last_sched.assign(h->stage, h->stage + total);
    h->last_rows = rows;
    h->last_valid = true;
    return EVO_OK;
  }
  h->last_valid = false;
  EVO_CUDA(cudaMemcpyAsync(h->sched, S, bytes, cudaMemcpyDeviceToDevice, st));
  if (add_ones) EVO_CUDA(cudaMemsetAsync(h->sched + bytes, 1, one, st));
  EVO_CUDA(cudaMemsetAsync(h->status + 1, 0, sizeof(int), st));
  EVO_CUDA(launch_validate(h->sched, (long long)bytes, h->status + 1, st));
  *err_out = h->status + 1;
  return EVO_OK;
}


// The decomposition a cluster-path call of `samples` samples takes: the fewest
// estimated job rounds, weighting a round of a smaller cluster by (C_max/C)^0.4
// (per-job time measured at n_emb 256: 1.0 / 1.23 / 2.0 for C = 16 / 8 / 4 at
// refresh fraction 0.125, 1.0 / 1.15 / 1.41 at 1.0).
struct Pick {
  const JobParams* base;
  int shape, max_clusters;
};

Pick pick_decomposition(const evo_handle* h, long long samples) {
  Pick best{&h->base, h->shape, h->max_clusters};
  auto cost = [&](const JobParams& b, int mc) {
    const long long jobs = (samples + b.g - 1) / b.g;
    const long long rounds = (jobs + mc - 1) / mc;
    return (double)rounds * std::pow((double)h->base.C / (double)b.C, 0.4);
  };
  double bc = cost(h->base, h->max_clusters);
  for (int i = 0; i < h->n_alt; ++i) {
    const double c = cost(h->alt[i].base, h->alt[i].max_clusters);
    if (c < bc) {
      bc = c;
      best = {&h->alt[i].base, h->alt[i].shape, h->alt[i].max_clusters};
    }
  }
  return best;
}

cudaError_t launch_loop(evo_handle* h, const JobParams& p, cudaStream_t st, const Pick& pk) {
  if (h->prof_start && h->prof_stop) {
    cudaError_t e = cudaEventRecord(h->prof_start, st);
    if (e != cudaSuccess) return e;
  }
  cudaError_t e = launch_job(pk.shape, p, std::min(p.n_jobs, pk.max_clusters), st);
  if (e != cudaSuccess) return e;
  h->last_base = pk.base;
  h->last_mc = pk.max_clusters;
  h->last_path = 0;
  h->last_kernels = h->last_cond_kernels + 1 + (p.sched_err ? 1 : 0);
  if (h->prof_start && h->prof_stop) return cudaEventRecord(h->prof_stop, st);
  return cudaSuccess;
}

evo_status finish(evo_handle* h, cudaStream_t st) {
  h->last_stream = st;
  EVO_CUDA(cudaGetLastError());
  if (h->cfg.debug_sync) return evo_get_status(h);
  return EVO_OK;
}

// Stage n_sched lattices for the batch-wide path, which needs them on the host
// as well: a device lattice is copied back (one synchronisation) and checked there.
evo_status stage_wide(evo_handle* h, const uint8_t* S, int n_sched, int rows, bool add_ones, cudaStream_t st) {
  const size_t bytes = (size_t)rows * h->T * n_sched;
  std::vector<uint8_t> host;
  if (is_device_ptr(S)) {
    host.resize(bytes);
    EVO_CUDA(cudaMemcpyAsync(host.data(), S, bytes, cudaMemcpyDeviceToHost, st));
    EVO_CUDA(cudaStreamSynchronize(st));
    S = host.data();
  }
  const int* err = nullptr;
  return stage_schedules(h, S, n_sched, rows, add_ones, st, &err);   // host lattice: validated, cached
}

cudaError_t launch_wide(evo_handle* h, const float* obs, const float* noise, float* out, int samples, int per_sched,
                        int n_sched, int S_rows, cudaStream_t st, float* trace = nullptr) {
  WideCall c{};
  c.obs = obs;
  c.noise = noise;
  c.out = out;
  c.kv_obs = h->kv_obs;
  c.kv_time = h->kv_time;
  c.stab = h->stab;
  c.samples = samples;
  c.per_sched = per_sched;
  c.obs_mod = per_sched;
  c.S_host = h->last_sched.data();
  c.S_dev = h->sched;
  c.n_sched = n_sched;
  c.S_rows = S_rows;
  c.trace = trace;
  c.status = h->status;
  c.st = st;
  if (h->prof_start && h->prof_stop) {
    const cudaError_t e = cudaEventRecord(h->prof_start, st);
    if (e != cudaSuccess) return e;
  }
  const cudaError_t e = wide_run(h->wide, c);
  if (e != cudaSuccess) return e;
  h->last_path = 1;
  h->last_kernels = h->last_cond_kernels + wide_last_launches(h->wide);
  if (h->prof_start && h->prof_stop) return cudaEventRecord(h->prof_stop, st);
  return cudaSuccess;
}

bool use_wide(const evo_handle* h, long long samples) {
  return h->wide && samples * h->H >= h->wide_rows && samples * h->H <= wide_rows_capacity(h->wide);
}

evo_status run(evo_handle* h, const float* obs, const float* noise, const uint8_t* S, int S_rows, int N, float* out,
               float* trace, void* stream) {
  if (!h || !obs || !noise || !S || !out) return EVO_ERR_ARG;
  if (N <= 0 || N > h->max_batch) return EVO_ERR_SHAPE;
  if (S_rows != h->U && S_rows != h->L) return EVO_ERR_SCHEDULE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (use_wide(h, N)) {
    const evo_status s = stage_wide(h, S, 1, S_rows, false, st);
    if (s != EVO_OK) return s;
    h->last_cond_kernels = 0;                  // the batch-wide sequence computes kv_obs itself
    EVO_CUDA(launch_wide(h, obs, noise, out, N, N, 1, S_rows, st, trace));
    return finish(h, st);
  }
  const int* err = nullptr;
  evo_status s = stage_schedules(h, S, 1, S_rows, false, st, &err);
  if (s != EVO_OK) return s;
  EVO_CUDA(obs_cond(h, obs, N, h->cond_scratch, h->kv_obs, st));
  const Pick pk = pick_decomposition(h, N);
  JobParams p = *pk.base;
  p.samples = N;
  p.per_sched = N;
  p.obs_mod = N;
  p.n_jobs = (N + p.g - 1) / p.g;
  p.S = h->sched;
  p.S_rows = S_rows;
  p.S_stride = (long long)S_rows * h->T;
  p.sched_err = err;
  p.noise = noise;
  p.out = out;
  p.trace = trace;
  EVO_CUDA(launch_loop(h, p, st, pk));
  return finish(h, st);
}

}  // namespace

extern "C" {

evo_status evo_denoise(evo_handle* h, const float* obs, const float* noise, const uint8_t* S, int32_t S_rows,
                       int32_t N, float* out_actions, void* stream) {
  NvtxRange range("evo_denoise");
  return run(h, obs, noise, S, S_rows, N, out_actions, nullptr, stream);
}

evo_status evo_denoise_trace(evo_handle* h, const float* obs, const float* noise, const uint8_t* S, int32_t S_rows,
                             int32_t N, float* out_actions, float* trace, void* stream) {
  if (!trace) return EVO_ERR_ARG;
  NvtxRange range("evo_denoise_trace");
  return run(h, obs, noise, S, S_rows, N, out_actions, trace, stream);
}

}  // extern "C"

namespace {

// Scratch of evo_denoise_noalloc: a file-scope device array (no allocation at
// call time).  Host code may not use the symbol as a device address; its
// address is looked up once per device with cudaGetSymbolAddress.
constexpr size_t NOALLOC_SCRATCH_BYTES = size_t(8) << 20;
__device__ __align__(256) unsigned char g_noalloc_scratch[NOALLOC_SCRATCH_BYTES];

std::mutex g_noalloc_mu;
void* g_noalloc_addr[256] = {};

evo_status noalloc_scratch(int dev, float** out) {
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (dev < 0 || dev >= 256) return EVO_ERR_UNSUPPORTED;
  if (!g_noalloc_addr[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || !ptr) return EVO_ERR_CUDA;
    g_noalloc_addr[dev] = ptr;
  }
  *out = static_cast<float*>(g_noalloc_addr[dev]);
  return EVO_OK;
}

}  // namespace

extern "C" {

evo_status evo_denoise_noalloc(evo_handle* h, const float* obs, const float* noise, const uint8_t* S, int32_t S_rows,
                               int32_t N, float* out_actions, void* stream) {
  NvtxRange range("evo_denoise_noalloc");
  if (!h || !obs || !noise || !S || !out_actions) return EVO_ERR_ARG;
  if (N <= 0 || N > h->max_batch) return EVO_ERR_SHAPE;
  if (S_rows != h->U && S_rows != h->L) return EVO_ERR_SCHEDULE;
  // observation keys/values, then the condition MLP's intermediates (6E floats per token)
  const size_t kv_floats = (size_t)N * h->cfg.n_obs * h->L * 2 * h->E;
  const size_t need = (kv_floats + (size_t)N * h->cfg.n_obs * 6 * h->E) * sizeof(float);
  if (need > NOALLOC_SCRATCH_BYTES) return EVO_ERR_SHAPE;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return EVO_ERR_CUDA;
  if (dev != h->device) return EVO_ERR_ARG;
  float* kv = nullptr;
  const evo_status ss = noalloc_scratch(dev, &kv);
  if (ss != EVO_OK) return ss;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int* err = nullptr;
  evo_status s = stage_schedules(h, S, 1, S_rows, false, st, &err);
  if (s != EVO_OK) return s;
  EVO_CUDA(obs_cond(h, obs, N, kv + kv_floats, kv, st));
  const Pick pk = pick_decomposition(h, N);
  JobParams p = *pk.base;
  p.kv_obs = kv;
  p.samples = N;
  p.per_sched = N;
  p.obs_mod = N;
  p.n_jobs = (N + p.g - 1) / p.g;
  p.S = h->sched;
  p.S_rows = S_rows;
  p.S_stride = (long long)S_rows * h->T;
  p.sched_err = err;
  p.noise = noise;
  p.out = out_actions;
  p.trace = nullptr;
  EVO_CUDA(launch_loop(h, p, st, pk));
  return finish(h, st);
}

evo_status evo_denoise_population(evo_handle* h, const float* obs, const float* noise, const uint8_t* S_pop,
                                  int32_t P, int32_t S_rows, int32_t N_obs, float* out_actions, float* dev_l2,
                                  void* stream) {
  NvtxRange range("evo_denoise_population");
  if (!h || !obs || !noise || !S_pop || !dev_l2) return EVO_ERR_ARG;
  if (P <= 0 || N_obs <= 0) return EVO_ERR_SHAPE;
  const long long samples = (long long)(P + 1) * N_obs;
  if (samples > h->max_batch) return EVO_ERR_SHAPE;
  if (S_rows != h->U && S_rows != h->L) return EVO_ERR_SCHEDULE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int HA = h->H * h->A;
  if (use_wide(h, samples)) {
    const evo_status s = stage_wide(h, S_pop, P, S_rows, true, st);
    if (s != EVO_OK) return s;
    h->last_cond_kernels = 0;                  // the batch-wide sequence computes kv_obs itself
    EVO_CUDA(launch_wide(h, obs, noise, h->pop_x, (int)samples, N_obs, P + 1, S_rows, st));
    EVO_CUDA(launch_pop_dev(h->pop_x, P, N_obs, HA, dev_l2, st));
    h->last_kernels += 1;
    if (out_actions)
      EVO_CUDA(cudaMemcpyAsync(out_actions, h->pop_x, (size_t)P * N_obs * HA * 4, cudaMemcpyDeviceToDevice, st));
    return finish(h, st);
  }
  const int* err = nullptr;
  evo_status s = stage_schedules(h, S_pop, P, S_rows, true, st, &err);
  if (s != EVO_OK) return s;
  EVO_CUDA(obs_cond(h, obs, N_obs, h->cond_scratch, h->kv_obs, st));
  Pick pk = pick_decomposition(h, samples);
  JobParams p = *pk.base;
  // samples of one job must share a schedule: g divides N_obs
  int g = p.g;
  while (g > 1 && N_obs % g) g >>= 1;
  if (g != p.g) {
    // fewer samples per job: the compiled shape for g, with its own ring geometry
    int slot = 0, nslot = 0;
    pk.shape = shape_find(h->cfg.dtype, h->E, h->cfg.n_head, h->H, p.C, g, &slot, &nslot);
    if (pk.shape < 0) return EVO_ERR_UNSUPPORTED;
    const int smem = plan(&h->cfg, p.C, g, slot, nslot, h->smem_limit, p);
    if (smem < 0) return EVO_ERR_UNSUPPORTED;
    EVO_CUDA(job_kernel_prepare(pk.shape, smem, &pk.max_clusters));
    p.stab = h->stab;
    p.kv_time = h->kv_time;
    p.kv_obs = h->kv_obs;
    p.wpack = h->wpack;
    p.vec = h->vec;
    p.cache = h->cache;
    p.status = h->status;
    h->replan = p;
    pk.base = &h->replan;
  }
  p.samples = (int)samples;
  p.per_sched = N_obs;
  p.obs_mod = N_obs;
  p.n_jobs = (int)((samples + p.g - 1) / p.g);
  p.S = h->sched;
  p.S_rows = S_rows;
  p.S_stride = (long long)S_rows * h->T;
  p.sched_err = err;
  p.noise = noise;
  p.out = h->pop_x;
  p.trace = nullptr;
  EVO_CUDA(launch_loop(h, p, st, pk));
  EVO_CUDA(launch_pop_dev(h->pop_x, P, N_obs, HA, dev_l2, st));
  h->last_kernels += 1;
  if (out_actions)
    EVO_CUDA(cudaMemcpyAsync(out_actions, h->pop_x, (size_t)P * N_obs * HA * 4, cudaMemcpyDeviceToDevice, st));
  return finish(h, st);
}

evo_status evo_check_guards(evo_handle* h) {
  if (!h) return EVO_ERR_ARG;
  if (cudaStreamSynchronize(h->last_stream) != cudaSuccess) return EVO_ERR_CUDA;
  int r = guards_check(h->guards);
  if (r == 0 && h->wide) r = guards_check(*wide_guards(h->wide));
  return r == 0 ? EVO_OK : (r > 0 ? EVO_ERR_CORRUPT : EVO_ERR_CUDA);
}

evo_status evo_test_wait_timeout(evo_handle* h, int32_t helper, int64_t limit, void* stream) {
  if (!h || (helper != 0 && helper != 1)) return EVO_ERR_ARG;
  // bounded so that the probe ends within milliseconds: 10^7 cycles or 10^5 polls
  if (limit < 1 || limit > (helper == 0 ? 10000000 : 100000)) return EVO_ERR_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  EVO_CUDA(launch_wait_probe(helper, limit, h->status, st));
  h->last_stream = st;
  return EVO_OK;
}

evo_status evo_test_gelu(const float* x, float* y, int64_t n, int32_t packed, void* stream) {
  if (n < 0 || (packed != 0 && packed != 1) || (n > 0 && (!x || !y))) return EVO_ERR_ARG;
  if (n > 0 && (!is_device_ptr(x) || !is_device_ptr(y))) return EVO_ERR_ARG;
  EVO_CUDA(launch_gelu_probe(x, y, n, packed, reinterpret_cast<cudaStream_t>(stream)));
  return EVO_OK;
}

evo_status evo_set_profile_events(evo_handle* h, void* start, void* stop) {
  if (!h || (start == nullptr) != (stop == nullptr)) return EVO_ERR_ARG;
  h->prof_start = reinterpret_cast<cudaEvent_t>(start);
  h->prof_stop = reinterpret_cast<cudaEvent_t>(stop);
  return EVO_OK;
}

int32_t evo_last_cuda_error(void) { return g_last_cuda_error; }

size_t evo_redundancy_scratch_bytes(int32_t T, int32_t U, int32_t N, int32_t n, int32_t metric) {
  if (!redundancy_shape_ok(T, U, N, n, metric)) return 0;
  return redundancy_scratch_bytes(T, U, N, n, metric);
}

evo_status evo_redundancy_map(const float* trace, int32_t T, int32_t U, int32_t N, int32_t n, int32_t metric,
                              float* d, void* scratch, void* stream) {
  if (!trace || !d || !scratch) return EVO_ERR_ARG;
  if (!redundancy_shape_ok(T, U, N, n, metric)) return EVO_ERR_SHAPE;
  EVO_CUDA(launch_redundancy(trace, T, U, N, n, metric, d, scratch, reinterpret_cast<cudaStream_t>(stream)));
  return EVO_OK;
}

evo_status evo_guided_schedules(const float* d, int32_t U, int32_t T, int32_t K, float eps, int32_t gamma,
                                const uint64_t* rnd, int32_t P, uint8_t* S, void* stream) {
  if (!d || !rnd || !S || !(eps >= 0.f)) return EVO_ERR_ARG;
  if (!guided_shape_ok(U, T, K, gamma, P)) return EVO_ERR_SHAPE;
  EVO_CUDA(launch_guided(d, U, T, K, eps, gamma, rnd, P, S, reinterpret_cast<cudaStream_t>(stream)));
  return EVO_OK;
}

evo_status evo_get_last_call(const evo_handle* h, int32_t* path, int64_t* kernels) {
  if (!h) return EVO_ERR_ARG;
  if (path) *path = h->last_path;
  if (kernels) *kernels = h->last_kernels;
  return EVO_OK;
}

evo_status evo_get_status(evo_handle* h) {
  if (!h) return EVO_ERR_ARG;
  if (cudaStreamSynchronize(h->last_stream) != cudaSuccess) return EVO_ERR_CUDA;
  int st[2] = {0, 0};
  if (cudaMemcpy(st, h->status, sizeof(st), cudaMemcpyDeviceToHost) != cudaSuccess) return EVO_ERR_CUDA;
  if (st[0] || st[1]) cudaMemset(h->status, 0, sizeof(st));
  if (st[1]) return EVO_ERR_SCHEDULE;
  if (st[0] & ST_INDEX) return EVO_ERR_CORRUPT;
  if (st[0] & ST_TIMEOUT) return EVO_ERR_TIMEOUT;
  if (st[0] & ST_SCHEDULE) return EVO_ERR_SCHEDULE;
  return EVO_OK;
}

}  // extern "C"
