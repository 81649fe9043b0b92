// Host implementation of the C ABI declared in include/lrqat.h: argument
// validation, workspace carving, TMA tensor-map encoding and kernel launches.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "kernels.h"
#include "merge.h"
#include "lrqat.h"

namespace lrqat {
namespace {

// Device status word: kernels OR a bit into it when a bounded wait gives up.
__device__ int g_device_status;

constexpr uint64_t kWaitTimeoutNs = 2000000000ull;   // 2 s per wait

thread_local std::string t_last_error;

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  t_last_error = buf;
  return code;
}

int cuda_fail(cudaError_t e, const char* what) {
  return fail(LRQAT_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

struct DeviceInfo {
  bool ready = false;
  int sms = 0;
  int* status = nullptr;
};
DeviceInfo g_dev[kMaxDevices];
std::mutex g_dev_mu;

int device_info(DeviceInfo** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return fail(LRQAT_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
  std::lock_guard<std::mutex> lock(g_dev_mu);
  DeviceInfo& d = g_dev[dev];
  if (!d.ready) {
    e = cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_device_status);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(status)");
    d.status = static_cast<int*>(p);
    d.ready = true;
  }
  *out = &d;
  return LRQAT_OK;
}

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
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

// Row-major 2-D tensor [outer][inner] with rows of `row_bytes` bytes.
int encode_2d(CUtensorMap* map, CUtensorMapDataType dt, const void* ptr, uint64_t inner, uint64_t outer,
              uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swz, const char* what) {
  auto fn = tensor_map_encoder();
  if (!fn) return fail(LRQAT_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  CUresult r = fn(map, dt, 2, const_cast<void*>(ptr), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(LRQAT_ERR_CUDA, "tensor map for %s failed (CUresult %d)", what, (int)r);
  return LRQAT_OK;
}

// The fused GEMMs load only the first r16 columns of the second low-rank factor per
// stage, as rows of 32, 64 or 128 bytes with the matching swizzle (rank 33..48 keeps
// 64 columns: no swizzle mode has 96-byte rows).
int sf_cols(int r16) { return r16 == 48 ? 64 : r16; }
CUtensorMapSwizzle sf_swizzle(int r16) {
  const int c = sf_cols(r16);
  return c == 16 ? CU_TENSOR_MAP_SWIZZLE_32B : c == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// The fused GEMMs read the factors straight from the caller's A [m, r] and B [r, k] when
// TMA can address them (16-byte aligned rows: r a multiple of 8, aligned bases): A as
// 64-column K-major boxes whose columns past r read as zeros (the same tile as the padded
// copy), B as MN-major boxes of r16 rank rows whose rows past r read as zeros.
bool direct_factors(const lrqat_layer& L, const void* A, const void* B) {
  return L.r % 8 == 0 && aligned16(A) && aligned16(B);
}

int frac_bits(const lrqat_layer& L) { return L.phi_format == LRQAT_PHI_QFIXED ? 8 - L.bits : 0; }

// Where the forward and dX GEMMs take the low-rank term from (lrqat_set_lowrank_path):
// 1 = the tile that each GEMM stage computes next to the main product (ranks up to 64);
// 2 = the codes pass: one tensor-core pass per call writes the unclipped codes round(u) of every
// weight (int8, saturated) into the workspace, and the GEMMs read them as their base with the
// low-rank term switched off.  In the pair GEMM the in-stage tile is a chain of small MMAs
// whose TMEM buffer holds one stage, so it paces the stage (measured on a 4096 x 4096 layer at
// T = 8192: forward 218 -> 191 us, dX 254 -> 210 us with the codes, for a pass of 18 us), while
// the pass moves ~2 bytes per weight through HBM whatever T is.  Measured fwd + bwd per call,
// tile against codes: 4096 x 4096 at T = 2048 353 / 355 us, at T = 4096 511 / 500 us;
// 5120 x 13824 at T = 2048 1017 / 1044 us, at T = 4096 1657 / 1625 us.  So 0 (auto) takes the
// codes from kCodesMinTokens tokens on.  Ranks above 64 always take the codes: their factor slices do not
// fit next to the GEMMs' token ring, and recomputing A B per 448-token tile would cost r/448 of
// the GEMM's own tensor work.  The same holds for dW, which otherwise computes its own tile.
int lowrank_path_from_env() {
  const char* v = std::getenv("LRQAT_LOWRANK_PATH");
  if (v && std::strcmp(v, "tile") == 0) return 1;
  if (v && std::strcmp(v, "codes") == 0) return 2;
  return 0;
}
std::atomic<int> g_lowrank_path{lowrank_path_from_env()};
constexpr int64_t kCodesMinTokens = 3072;
bool codes_dw(const lrqat_layer& L) { return L.r > 64; }
bool codes_gemm(const lrqat_layer& L, int64_t T) {
  if (L.r > 64) return true;
  const int v = g_lowrank_path.load(std::memory_order_relaxed);
  return v == 2 || (v == 0 && T >= kCodesMinTokens);
}
bool phi_16bit(const lrqat_layer& L) { return L.phi_format == LRQAT_PHI_BF16 || L.phi_format == LRQAT_PHI_FP16; }
int round16(int r) { return (r + 15) / 16 * 16; }

int validate_layer(const lrqat_layer* L) {
  if (!L) return fail(LRQAT_ERR_INVALID_ARG, "layer is NULL");
  if (L->m <= 0 || L->k <= 0) return fail(LRQAT_ERR_INVALID_ARG, "m and k must be positive (m=%lld k=%lld)",
                                          (long long)L->m, (long long)L->k);
  if (L->m % 128 || L->k % 128)
    return fail(LRQAT_ERR_UNSUPPORTED, "m and k must be multiples of 128 (m=%lld k=%lld)", (long long)L->m,
                (long long)L->k);
  if (L->m > (int64_t)1 << 30 || L->k > (int64_t)1 << 30) return fail(LRQAT_ERR_UNSUPPORTED, "m or k too large");
  if (L->r < 1) return fail(LRQAT_ERR_INVALID_ARG, "rank r must be >= 1 (r=%d)", L->r);
  if (L->r > 256) return fail(LRQAT_ERR_UNSUPPORTED, "rank r=%d > 256 is not supported", L->r);
  if (!std::isfinite(L->alpha)) return fail(LRQAT_ERR_INVALID_ARG, "alpha must be finite");
  if (L->phi_format == LRQAT_PHI_QFIXED) {
    if (L->bits < 2 || L->bits > 7) return fail(LRQAT_ERR_INVALID_ARG, "QFIXED needs 2 <= bits <= 7 (bits=%d)", L->bits);
  } else if (L->phi_format == LRQAT_PHI_INT_PACKED) {
    if (L->bits < 2 || L->bits > 4)
      return fail(LRQAT_ERR_INVALID_ARG, "INT_PACKED needs 2 <= bits <= 4 (bits=%d)", L->bits);
  } else if (L->phi_format >= LRQAT_PHI_BF16 && L->phi_format <= LRQAT_PHI_FP8_E5M2) {
    if (L->bits < 2 || L->bits > 8)
      return fail(LRQAT_ERR_INVALID_ARG, "floating-point phi needs 2 <= bits <= 8 (bits=%d)", L->bits);
    if (L->zero)
      return fail(LRQAT_ERR_UNSUPPORTED, "zero offsets are implemented for the integer phi formats only");
  } else {
    return fail(LRQAT_ERR_INVALID_ARG, "unknown phi_format %d", L->phi_format);
  }
  if (L->group_size < 0) return fail(LRQAT_ERR_INVALID_ARG, "group_size must be >= 0");
  if (L->group_size > 0 && (L->group_size % 128 || L->k % L->group_size))
    return fail(LRQAT_ERR_UNSUPPORTED, "group_size %d must be a multiple of 128 dividing k", L->group_size);
  if (L->r > 64 && L->bits > 7)
    return fail(LRQAT_ERR_UNSUPPORTED, "ranks above 64 need bits <= 7 (the unclipped codes are kept as int8)");
  if (L->act_bits != 0 && L->act_bits != 8)
    return fail(LRQAT_ERR_UNSUPPORTED, "act_bits must be 0 or 8 (got %d)", L->act_bits);
  if (L->zero && !aligned16(L->zero)) return fail(LRQAT_ERR_ALIGNMENT, "zero (offsets) is not 16-byte aligned");
  if (L->act_per_token != 0 && (L->act_per_token != 1 || L->act_bits != 8))
    return fail(LRQAT_ERR_INVALID_ARG, "act_per_token must be 0, or 1 with act_bits == 8");
  if (L->u_bf16 != 0) {
    if (L->u_bf16 != 1) return fail(LRQAT_ERR_INVALID_ARG, "u_bf16 must be 0 or 1");
    if (L->phi_format == LRQAT_PHI_FP16)
      return fail(LRQAT_ERR_UNSUPPORTED, "u_bf16 needs a base exact in bf16 (not FP16)");
    if (L->zero) return fail(LRQAT_ERR_UNSUPPORTED, "u_bf16 is implemented for symmetric grids only");
    int e = 0;
    if (!(L->alpha > 0.0f) || std::frexp(static_cast<double>(L->alpha) / L->r, &e) != 0.5)
      return fail(LRQAT_ERR_UNSUPPORTED, "u_bf16 needs alpha / r to be a power of two");
  }
  return LRQAT_OK;
}

#define LRQAT_CHECK_PTR(p, name)                                                       \
  do {                                                                                 \
    if (!(p)) return fail(LRQAT_ERR_INVALID_ARG, "%s is NULL", name);                  \
    if (!aligned16(p)) return fail(LRQAT_ERR_ALIGNMENT, "%s is not 16-byte aligned", name); \
  } while (0)

#define LRQAT_CUDA(expr, what)                          \
  do {                                                  \
    cudaError_t e_ = (expr);                            \
    if (e_ != cudaSuccess) return cuda_fail(e_, what);  \
  } while (0)

#define LRQAT_TRY(expr)          \
  do {                           \
    int st_ = (expr);            \
    if (st_ != LRQAT_OK) return st_; \
  } while (0)

// ------------------------------------------------------------------ tracing --
struct TraceRec {
  const char* name;
  int kernels;
  cudaEvent_t start, stop;
};
std::mutex g_trace_mu;
bool g_trace_on = false;
std::vector<TraceRec> g_trace;
std::vector<cudaEvent_t> g_event_pool;

cudaEvent_t trace_event() {
  if (!g_event_pool.empty()) {
    cudaEvent_t e = g_event_pool.back();
    g_event_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

void trace_clear_locked() {
  for (auto& r : g_trace) {
    if (r.start) g_event_pool.push_back(r.start);
    if (r.stop) g_event_pool.push_back(r.stop);
  }
  g_trace.clear();
}

// Brackets the kernels enqueued in its scope with events on `stream` while tracing is on.
class TraceScope {
 public:
  TraceScope(const char* name, int kernels, cudaStream_t stream) : stream_(stream) {
    std::lock_guard<std::mutex> lock(g_trace_mu);
    if (!g_trace_on) return;
    rec_.name = name;
    rec_.kernels = kernels;
    rec_.start = trace_event();
    rec_.stop = trace_event();
    if (rec_.start && rec_.stop && cudaEventRecord(rec_.start, stream) == cudaSuccess) active_ = true;
  }
  ~TraceScope() {
    if (!active_) return;
    std::lock_guard<std::mutex> lock(g_trace_mu);
    if (cudaEventRecord(rec_.stop, stream_) == cudaSuccess) g_trace.push_back(rec_);
  }

 private:
  cudaStream_t stream_;
  TraceRec rec_{};
  bool active_ = false;
};

#define LRQAT_LAUNCH(name, nkernels, stream, expr, what)        \
  do {                                                          \
    TraceScope ts_(name, nkernels, stream);                     \
    cudaError_t e_ = (expr);                                    \
    if (e_ != cudaSuccess) return cuda_fail(e_, what);          \
  } while (0)

// Carves aligned sub-buffers out of a caller-provided workspace.
struct Carver {
  uintptr_t base;
  size_t used = 0;
  explicit Carver(void* p) : base(reinterpret_cast<uintptr_t>(p)) {}
  void* take(size_t bytes) {
    used = (used + 255) & ~size_t(255);
    void* p = reinterpret_cast<void*>(base + used);
    used += bytes;
    return p;
  }
};

// ----------------------------------------------------------------- planning --
// Schedule of the weight-gradient work: 0 = chosen per call by the cost model below,
// 1 = equal token splits, 2 = whole tiles and a tail.  The environment variable
// LRQAT_DW_SCHEDULE ("split" / "tail") sets the start value once, when the library is
// loaded; lrqat_set_dw_schedule changes it explicitly.
int dw_schedule_from_env() {
  const char* v = std::getenv("LRQAT_DW_SCHEDULE");
  if (v && std::strcmp(v, "split") == 0) return 1;
  if (v && std::strcmp(v, "tail") == 0) return 2;
  return 0;
}
std::atomic<int> g_dw_schedule{dw_schedule_from_env()};

// Kernel of the forward and dX GEMMs (lrqat_set_gemm_variant): 0 = CTA pairs (fused_pair.cu)
// wherever they were measured faster, which is every GEMM whose produced weight operand has a
// multiple of 256 rows (with the dX scales read as bf16 rows, group-wise dX too: 916 -> 730 us on
// the 14336 x 4096 g128 projection at T = 8192); 1 = the one-SM kernel (fused_gemm.cu) always;
// 2 = pairs wherever the rows allow.  LRQAT_GEMM_VARIANT ("auto" / "single" / "pair") sets the
// start value once, when the library is loaded.
int gemm_variant_from_env() {
  const char* v = std::getenv("LRQAT_GEMM_VARIANT");
  if (v && std::strcmp(v, "single") == 0) return 1;
  if (v && std::strcmp(v, "pair") == 0) return 2;
  return 0;
}
std::atomic<int> g_gemm_variant{gemm_variant_from_env()};
bool use_pair(int64_t rows) {
  const int v = g_gemm_variant.load(std::memory_order_relaxed);
  return rows % 256 == 0 && v != 1;
}
constexpr int kPairTokens = 448;   // tokens per pair tile (two accumulators of 224)

constexpr int kDwPairTokensPerStage = 64;   // the pair dW kernel's stage (dw_pair.cu)
// dW on CTA pairs (dw_pair.cu): 256 x 256 tiles, ranks up to 64, by the same setting as the
// forward and dX GEMMs (lrqat_set_gemm_variant: not with 1, the one-SM kernels).
bool use_pair_dw(const lrqat_layer& L) {
  return L.m % 256 == 0 && L.k % 256 == 0 && !codes_dw(L) && g_gemm_variant.load(std::memory_order_relaxed) != 1;
}

struct DwPlan {
  int nchunks, ni, nj, nsplit, tchunk, units;
  DwSched sched;
  bool pair;   // the pair kernel: ni counts 256-row tiles and sched.grid pairs
  int ni128;   // 128-row blocks (the partial outputs)
  int bkt;     // tokens per pipeline stage
};

// sms: the work slots of the persistent grid (SMs for the one-SM kernel, resident pairs for
// the pair kernel).
DwPlan plan_dw(const lrqat_layer& L, int64_t T, int sms, bool pair) {
  DwPlan p;
  p.pair = pair;
  p.nchunks = (L.k % 256 == 0 && !codes_dw(L)) ? 2 : 1;
  p.ni128 = static_cast<int>(L.m / 128);
  p.ni = static_cast<int>(pair ? L.m / 256 : L.m / 128);
  p.nj = static_cast<int>(L.k / (128 * p.nchunks));
  const int tiles = p.ni * p.nj;
  p.bkt = pair ? kDwPairTokensPerStage : 32;   // tokens per pipeline stage
  const int64_t tsteps = (T + p.bkt - 1) / p.bkt;
  // Pick the token split that fills the SMs best; keep >= 256 tokens per split.
  int best = 1;
  double best_eff = 0.0;
  for (int s = 1; s <= 8; ++s) {
    if (s > 1 && tsteps / s < 8) break;
    const int64_t units = static_cast<int64_t>(tiles) * s;
    const int64_t waves = (units + sms - 1) / sms;
    const double eff = static_cast<double>(units) / static_cast<double>(waves * sms) * (1.0 - 0.01 * (s - 1));
    if (eff > best_eff + 1e-9) {
      best_eff = eff;
      best = s;
    }
  }
  p.nsplit = best;
  p.tchunk = static_cast<int>((tsteps + best - 1) / best) * p.bkt;
  p.nsplit = static_cast<int>((T + p.tchunk - 1) / p.tchunk);   // no empty splits
  p.units = tiles * p.nsplit;
  const int grid_eq = p.units < sms ? p.units : sms;
  p.sched = DwSched{0, grid_eq, tsteps, 0, 0, 0};
  // Against whole tiles for the full waves of every SM and the remaining tiles cut into equal
  // token parts, one per CTA (at most 8 parts a tile, none shorter than a stage), by the
  // slowest CTA's cost in stage units: its stages plus kEpilogueStages for each unit it
  // finishes (the part of the epilogue that the next main loop waits for).
  const int64_t kEpilogueStages = 32 * 32 / p.bkt;
  const int64_t waves = (p.units + grid_eq - 1) / grid_eq;
  const int64_t cost_eq = waves * (p.tchunk / p.bkt + kEpilogueStages);
  const int64_t full_tiles = tiles / sms * sms;
  const int64_t tail_tiles = tiles - full_tiles;
  const int64_t q_cap = tsteps < 8 ? tsteps : 8;
  const int64_t tail_grid = tail_tiles * q_cap < sms ? tail_tiles * q_cap : sms;
  const DwSched tl{1, sms, tsteps, full_tiles, tail_tiles, tail_grid};
  const bool tail_ok = tail_tiles > 0;
  int64_t cost_tail = 0;
  if (tail_ok) {
    const int64_t q_min = tail_grid / tail_tiles;   // the longest parts
    cost_tail = full_tiles / sms * (tsteps + kEpilogueStages) + (tsteps + q_min - 1) / q_min + kEpilogueStages;
  }
  // a forced schedule (lrqat_set_dw_schedule) overrides the choice; the tail needs tail tiles
  const int force = g_dw_schedule.load(std::memory_order_relaxed);
  const bool use_tail = !tail_ok ? false : force == 2 ? true : force == 1 ? false : cost_tail < cost_eq;
  if (use_tail) {
    p.sched = tl;
    p.nsplit = dw_tile_segments(full_tiles, tl);   // the first tail tile has the most parts
    p.tchunk = 0;                                  // not used
    p.units = sms;
  }
  return p;
}

struct FwdWs {
  uint16_t* a_pad;
  uint16_t* bt_pad;
  uint16_t* x_codes;   // int8 codes (per tensor) or X_hat (per token), bf16
  uint16_t* at;        // codes path: A^T [r16, m] and B [r16, k] zero-padded, codes [m, k]
  uint16_t* b_pad;
  int8_t* codes;
  uint16_t* s_bf16;    // group-wise: the scales (and zero offsets) as bf16 rows [groups][m]
  uint16_t* z_bf16;
};

// with_codes: carve the buffers of the codes path too (ranks above 64 always have them).
size_t fwd_ws_layout(const lrqat_layer& L, int64_t T, bool with_codes, void* base, FwdWs* ws) {
  Carver c(base);
  FwdWs w{};
  if (L.r <= 64) {
    w.a_pad = static_cast<uint16_t*>(c.take(static_cast<size_t>(L.m) * 64 * 2));
    w.bt_pad = static_cast<uint16_t*>(c.take(static_cast<size_t>(L.k) * 64 * 2));
  }
  if (with_codes || L.r > 64) {
    const size_t r16 = static_cast<size_t>(round16(L.r));
    w.at = static_cast<uint16_t*>(c.take(r16 * L.m * 2));
    w.b_pad = static_cast<uint16_t*>(c.take(r16 * L.k * 2));
    w.codes = static_cast<int8_t*>(c.take(static_cast<size_t>(L.m) * L.k));
  }
  if (L.act_bits == 8) w.x_codes = static_cast<uint16_t*>(c.take(static_cast<size_t>(T) * L.k * 2));
  if (L.group_size) {
    const size_t groups = static_cast<size_t>(L.k / L.group_size);
    w.s_bf16 = static_cast<uint16_t*>(c.take(groups * L.m * 2));
    if (L.zero) w.z_bf16 = static_cast<uint16_t*>(c.take(groups * L.m * 2));
  }
  if (ws) *ws = w;
  return (c.used + 255) & ~size_t(255);
}

struct BwdWs {
  uint16_t* a_pad;
  uint16_t* bt_pad;
  uint16_t* at;
  uint16_t* b_pad;
  int8_t* phit;
  uint16_t* x_codes;
  uint32_t* xmask;
  float* dA_part;
  float* dB_part;
  float* ds_part;
  int32_t* tile_segs;
  int8_t* codes;       // codes path: the unclipped codes [m, k] (phit then holds their transpose)
  uint16_t* s_bf16;    // dX: the scales (and zero offsets) as bf16 rows [groups][m]
  uint16_t* z_bf16;
};

size_t bwd_ws_layout(const lrqat_layer& L, int64_t T, const DwPlan& p, void* base, BwdWs* ws) {
  Carver c(base);
  BwdWs w{};
  const int r16 = round16(L.r);
  // the buffers of both low-rank paths (lrqat_set_lowrank_path), so the size is the same for every setting
  w.codes = static_cast<int8_t*>(c.take(static_cast<size_t>(L.m) * L.k));
  if (L.r <= 64) {
    w.a_pad = static_cast<uint16_t*>(c.take(static_cast<size_t>(L.m) * 64 * 2));
    w.bt_pad = static_cast<uint16_t*>(c.take(static_cast<size_t>(L.k) * 64 * 2));
  }
  w.at = static_cast<uint16_t*>(c.take(static_cast<size_t>(r16) * L.m * 2));
  w.b_pad = static_cast<uint16_t*>(c.take(static_cast<size_t>(r16) * L.k * 2));
  // the transposed base of the dX GEMM: 16-bit for a 16-bit base on the tile path, else int8
  w.phit = static_cast<int8_t*>(c.take(static_cast<size_t>(L.m) * L.k * (phi_16bit(L) && L.r <= 64 ? 2 : 1)));
  if (L.act_bits == 8) {
    w.x_codes = static_cast<uint16_t*>(c.take(static_cast<size_t>(T) * L.k * 2));
    w.xmask = static_cast<uint32_t*>(c.take(static_cast<size_t>(L.k) * ((T + 31) / 32) * 4));
  }
  w.dA_part = static_cast<float*>(c.take(static_cast<size_t>(p.nj) * p.nsplit * L.m * L.r * 4));
  w.dB_part = static_cast<float*>(c.take(static_cast<size_t>(p.ni128) * p.nsplit * L.r * L.k * 4));
  w.ds_part = static_cast<float*>(c.take(static_cast<size_t>(2) * p.nsplit * L.m * (L.k / 128) * 4));
  w.tile_segs = static_cast<int32_t*>(c.take(static_cast<size_t>(p.ni128) * p.nj * 4));
  const size_t groups = L.group_size ? static_cast<size_t>(L.k / L.group_size) : 1;
  w.s_bf16 = static_cast<uint16_t*>(c.take(groups * L.m * 2));
  if (L.zero) w.z_bf16 = static_cast<uint16_t*>(c.take(groups * L.m * 2));
  if (ws) *ws = w;
  return (c.used + 255) & ~size_t(255);
}

int phi_map(CUtensorMap* map, const lrqat_layer& L, const void* phi0, uint32_t box_cols_elems, bool dw) {
  // Forward: slices of 64 columns (64 B rows of 8-bit values, SW64; packed 32 B rows,
  // SW32; 16-bit values 128 B rows, SW128).
  // dW: chunks of 128 columns (128 B rows, SW128; packed 64 B rows, SW64); 16-bit
  // bases are read by the dW epilogue without the map (a 64-column box is encoded).
  if (phi_16bit(L))
    return encode_2d(map, CU_TENSOR_MAP_DATA_TYPE_UINT16, phi0, L.k, L.m, L.k * 2, 64, 128,
                     CU_TENSOR_MAP_SWIZZLE_128B, "Phi0 (16-bit)");
  if (L.phi_format != LRQAT_PHI_INT_PACKED)
    return encode_2d(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, phi0, L.k, L.m, L.k, box_cols_elems, 128,
                     dw ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B, "Phi0");
  return encode_2d(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, phi0, L.k / 2, L.m, L.k / 2, box_cols_elems / 2, 128,
                   dw ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B, "Phi0 (packed)");
}

// Quantizer constants of the codes written for ranks above 64: the clamp bounds are the int8
// range instead of [n, p] (the GEMMs clip and mask from the unclipped code).
// The bias of the clipped codes the GEMMs read (merge.h, FusedArgs::codes_bias): c + 64 fits a
// byte's low seven bits for b <= 7 (the GEMM producers then turn four codes into bf16 with two
// byte permutes and two bf16 subtractions), c + 128 for b = 8.
uint32_t codes_bias(const lrqat_layer& L) { return L.bits <= 7 ? 64u : 128u; }

QuantParams saturating_params(const lrqat_layer& L) {
  QuantParams q = make_quant_params(L.bits, frac_bits(L), L.alpha, L.r);
  const QuantParams wide = make_quant_params(8, frac_bits(L), L.alpha, L.r);
  q.lo = wide.lo;
  q.hi = wide.hi;
  return q;
}

// The codes pass: codes[i, j] = sat8(round(phi^{-1}(Phi0[i, j]) + (alpha/r) (A B)[i, j])) on the
// tensor cores (any rank up to 256), from A [m, r] and B [r, k] themselves when the factors are
// direct (rank a multiple of 8, 16-byte aligned: TMA boxes past r read as zeros), else from the
// zero-padded A^T [r16, m] and B [r16, k].  clipped: the codes clip(round(u), n, p) plus the bias
// (codes_bias) instead, for when only the forward and dX GEMMs read them (dW of ranks above 64
// needs the unclipped codes for its mask).
int run_codes_pass(const lrqat_layer& L, const void* Phi0, const uint16_t* A, const uint16_t* B, const uint16_t* At,
                   const uint16_t* B_pad, int8_t* codes, bool clipped, const DeviceInfo* dev, cudaStream_t stream);

}  // namespace
}  // namespace lrqat

// Scratch of lrqat_linear_fwd_noalloc, for callers that cannot allocate device
// memory (runtimes that own all device memory and give an operator only its
// inputs and outputs, or that forbid allocation after start-up because
// cudaMalloc can synchronize the device).  It is part of the library image, so
// every device that loads the library holds these bytes until the process exits.
static __device__ __align__(256) unsigned char g_fwd_noalloc_scratch[LRQAT_FWD_NOALLOC_SCRATCH_BYTES];

namespace lrqat {
namespace {

std::mutex g_noalloc_mu;
void* g_noalloc_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device.  In host code the
// array's name is only a host-side stand-in, so the address is looked up once per
// device (with that device current) and cached.
int noalloc_scratch(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return fail(LRQAT_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (g_noalloc_addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_fwd_noalloc_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(forward scratch)");
    g_noalloc_addr[dev] = p;
  }
  *out = g_noalloc_addr[dev];
  return LRQAT_OK;
}

}  // namespace

namespace {
int run_codes_pass(const lrqat_layer& L, const void* Phi0, const uint16_t* A, const uint16_t* B, const uint16_t* At,
                   const uint16_t* B_pad, int8_t* codes, bool clipped, const DeviceInfo* dev, cudaStream_t stream) {
  const int r16 = round16(L.r);
  const bool direct = direct_factors(L, A, B);
  CUtensorMap tm_a, tm_b;
  if (direct) {
    LRQAT_TRY(encode_2d(&tm_a, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, A, L.r, L.m, L.r * 2, 64, 128,
                        CU_TENSOR_MAP_SWIZZLE_128B, "A"));
    LRQAT_TRY(encode_2d(&tm_b, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, B, L.k, L.r, L.k * 2, 64,
                        static_cast<uint32_t>(r16), CU_TENSOR_MAP_SWIZZLE_128B, "B"));
  } else {
    LRQAT_TRY(encode_2d(&tm_a, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, At, L.m, r16, L.m * 2, 64,
                        static_cast<uint32_t>(r16), CU_TENSOR_MAP_SWIZZLE_128B, "A^T (padded)"));
    LRQAT_TRY(encode_2d(&tm_b, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, B_pad, L.k, r16, L.k * 2, 64,
                        static_cast<uint32_t>(r16), CU_TENSOR_MAP_SWIZZLE_128B, "B (padded)"));
  }
  CUtensorMap tm_phi;
  LRQAT_TRY(phi_map(&tm_phi, L, Phi0, 128, true));
  MergeArgs a{};
  a.wz = codes;
  a.m = L.m;
  a.k = L.k;
  a.r16 = r16;
  a.q = clipped ? make_quant_params(L.bits, frac_bits(L), L.alpha, L.r) : saturating_params(L);
  a.code_bias = clipped ? codes_bias(L) : 0u;
  a.status = dev->status;
  a.timeout_ns = kWaitTimeoutNs;
  LRQAT_LAUNCH("lowrank_codes", 1, stream,
               launch_merge_tc(L.phi_format, L.u_bf16, direct ? 0 : 1, tm_a, tm_b, tm_phi, a, stream),
               "low-rank code pass");
  return LRQAT_OK;
}
}  // namespace
}  // namespace lrqat

using namespace lrqat;

extern "C" {

const char* lrqat_last_error(void) { return t_last_error.c_str(); }

static int linear_fwd_impl(const lrqat_layer* layer, int64_t T, const uint16_t* X, bool quantized, const void* Phi0,
                           const float* s, const uint16_t* A, const uint16_t* B, const float* s_x, uint16_t* Y,
                           void* workspace, size_t workspace_bytes, bool allow_codes, lrqat_stream_t stream);

// The forward of lrqat_linear_fwd with its scratch taken from the fixed array
// above instead of a caller workspace.  The first call on a device performs the
// address look-up.  Calls share the array, so calls that overlap on the GPU
// race; each call rewrites every scratch byte it later reads (padded adapter
// copies, activation codes), so nothing needs clearing between calls.  Nothing
// is allocated or freed here or in lrqat_linear_fwd.
int lrqat_linear_fwd_noalloc(const lrqat_layer* layer, int64_t T, const uint16_t* X, const void* Phi0,
                             const float* s, const uint16_t* A, const uint16_t* B, const float* s_x, uint16_t* Y,
                             lrqat_stream_t stream) {
  LRQAT_TRY(validate_layer(layer));
  if (T < 1) return fail(LRQAT_ERR_INVALID_ARG, "T must be >= 1 (T=%lld)", (long long)T);
  if (T > (int64_t)1 << 30) return fail(LRQAT_ERR_UNSUPPORTED, "T too large");
  // ranks up to 64 take the in-GEMM low-rank tile here: the codes of m x k weights would not fit
  const size_t need = fwd_ws_layout(*layer, T, false, nullptr, nullptr);
  if (need > LRQAT_FWD_NOALLOC_SCRATCH_BYTES)
    return fail(LRQAT_ERR_WORKSPACE,
                "lrqat_linear_fwd_noalloc: this layer and T need %zu bytes of scratch but the fixed scratch holds "
                "%zu bytes; use lrqat_linear_fwd with a workspace",
                need, (size_t)LRQAT_FWD_NOALLOC_SCRATCH_BYTES);
  void* scratch = nullptr;
  LRQAT_TRY(noalloc_scratch(&scratch));
  return linear_fwd_impl(layer, T, X, false, Phi0, s, A, B, s_x, Y, scratch, LRQAT_FWD_NOALLOC_SCRATCH_BYTES, false,
                         stream);
}

int lrqat_range_minmax(const lrqat_layer* layer, const float* W0, float* s0, lrqat_stream_t stream) {
  LRQAT_TRY(validate_layer(layer));
  LRQAT_CHECK_PTR(W0, "W0");
  LRQAT_CHECK_PTR(s0, "s0");
  const lrqat_layer& L = *layer;
  LRQAT_LAUNCH("range_minmax", 1, stream,
               launch_range_minmax(W0, L.m, L.k, L.group_size, L.bits, s0, L.zero, stream),
               "range_minmax launch");
  return LRQAT_OK;
}

int lrqat_range_lp(const lrqat_layer* layer, const float* W0, float p_norm, int32_t n_candidates, float* s0,
                   lrqat_stream_t stream) {
  LRQAT_TRY(validate_layer(layer));
  LRQAT_CHECK_PTR(W0, "W0");
  LRQAT_CHECK_PTR(s0, "s0");
  const lrqat_layer& L = *layer;
  if (L.zero) return fail(LRQAT_ERR_UNSUPPORTED, "L^p range setting is implemented for symmetric grids only");
  if (!(p_norm > 0.0f) || !std::isfinite(p_norm)) return fail(LRQAT_ERR_INVALID_ARG, "p_norm must be positive");
  if (n_candidates < 1 || n_candidates > 256)
    return fail(LRQAT_ERR_INVALID_ARG, "n_candidates must be in [1, 256] (got %d)", n_candidates);
  const int64_t seg = L.group_size ? L.group_size : L.k;
  if (seg * 4 > 200 * 1024) return fail(LRQAT_ERR_UNSUPPORTED, "row or group of %lld values too long", (long long)seg);
  LRQAT_LAUNCH("range_lp", 1, stream,
               launch_range_lp(W0, L.m, L.k, L.group_size, L.bits, p_norm, n_candidates, s0, stream),
               "range_lp launch");
  return LRQAT_OK;
}

int lrqat_act_quant(const lrqat_layer* layer, int64_t T, const uint16_t* X, const float* s_x, uint16_t* X_out,
                    uint32_t* mask, lrqat_stream_t stream) {
  LRQAT_TRY(validate_layer(layer));
  const lrqat_layer& L = *layer;
  if (L.act_bits != 8) return fail(LRQAT_ERR_INVALID_ARG, "lrqat_act_quant needs act_bits == 8");
  if (T < 1) return fail(LRQAT_ERR_INVALID_ARG, "T must be >= 1 (T=%lld)", (long long)T);
  if (T > (int64_t)1 << 30) return fail(LRQAT_ERR_UNSUPPORTED, "T too large");
  LRQAT_CHECK_PTR(X, "X");
  LRQAT_CHECK_PTR(X_out, "X_out");
  if (L.act_per_token) {
    LRQAT_LAUNCH("act_quant", 1, stream, launch_act_quant_token(X, T, L.k, X_out, stream), "activation quantizer");
    return LRQAT_OK;
  }
  if (!s_x) return fail(LRQAT_ERR_INVALID_ARG, "s_x is required for the per-tensor quantizer");
  if (mask && (reinterpret_cast<uintptr_t>(mask) & 3u)) return fail(LRQAT_ERR_ALIGNMENT, "mask is not 4-byte aligned");
  LRQAT_LAUNCH("act_quant", 1, stream, launch_act_quant(X, T, L.k, s_x, X_out, mask, stream), "activation quantizer");
  return LRQAT_OK;
}

int lrqat_downcast(const lrqat_layer* layer, const float* W0, const float* s0, void* Phi0, lrqat_stream_t stream) {
  LRQAT_TRY(validate_layer(layer));
  LRQAT_CHECK_PTR(W0, "W0");
  LRQAT_CHECK_PTR(s0, "s0");
  LRQAT_CHECK_PTR(Phi0, "Phi0");
  const lrqat_layer& L = *layer;
  LRQAT_LAUNCH("downcast", 1, stream,
               launch_downcast(W0, s0, L.zero, L.m, L.k, L.group_size, L.bits, L.phi_format, Phi0, stream),
               "downcast launch");
  return LRQAT_OK;
}

size_t lrqat_fwd_workspace_bytes(const lrqat_layer* layer, int64_t T) {
  if (validate_layer(layer) != LRQAT_OK || T < 1) return 0;
  return fwd_ws_layout(*layer, T, true, nullptr, nullptr);
}

// quantized: X is already the activation quantizer's output for this layer (per tensor: the
// codes; per token: X_hat), so no quantizer runs.  allow_codes: the workspace has the buffers
// of the codes path (false for the allocation-free forward, whose scratch is sized without them).
static int linear_fwd_impl(const lrqat_layer* layer, int64_t T, const uint16_t* X, bool quantized, const void* Phi0,
                           const float* s, const uint16_t* A, const uint16_t* B, const float* s_x, uint16_t* Y,
                           void* workspace, size_t workspace_bytes, bool allow_codes, lrqat_stream_t stream) {
  LRQAT_TRY(validate_layer(layer));
  const lrqat_layer& L = *layer;
  if (quantized && L.act_bits != 8)
    return fail(LRQAT_ERR_INVALID_ARG, "quantized activations need act_bits == 8 (got %d)", L.act_bits);
  if (T < 1) return fail(LRQAT_ERR_INVALID_ARG, "T must be >= 1 (T=%lld)", (long long)T);
  if (T > (int64_t)1 << 30) return fail(LRQAT_ERR_UNSUPPORTED, "T too large");
  LRQAT_CHECK_PTR(X, "X");
  LRQAT_CHECK_PTR(Phi0, "Phi0");
  LRQAT_CHECK_PTR(s, "s");
  if (!A) return fail(LRQAT_ERR_INVALID_ARG, "A is NULL");
  if (!B) return fail(LRQAT_ERR_INVALID_ARG, "B is NULL");
  LRQAT_CHECK_PTR(Y, "Y");
  if (L.act_bits == 8 && !L.act_per_token && !s_x)
    return fail(LRQAT_ERR_INVALID_ARG, "s_x is required when act_bits == 8 (per-tensor scale)");
  const size_t need = fwd_ws_layout(L, T, allow_codes, nullptr, nullptr);
  if (!workspace || workspace_bytes < need)
    return fail(LRQAT_ERR_WORKSPACE, "forward workspace of %zu bytes required, %zu given", need,
                workspace ? workspace_bytes : (size_t)0);
  if (!aligned16(workspace)) return fail(LRQAT_ERR_ALIGNMENT, "workspace is not 16-byte aligned");
  DeviceInfo* dev = nullptr;
  LRQAT_TRY(device_info(&dev));

  FwdWs ws;
  fwd_ws_layout(L, T, allow_codes, workspace, &ws);
  const int r16 = round16(L.r);
  const bool cb = L.r > 64 || (allow_codes && codes_gemm(L, T));
  const bool pair = use_pair(L.m);
  // the pair kernel reads K-major factor slices, so it takes B^T from the padded copy
  const bool direct = !cb && !pair && direct_factors(L, A, B);
  if (cb) {
    // the codes of every weight, once per call (from A and B themselves when the factors are direct)
    if (!direct_factors(L, A, B))
      LRQAT_LAUNCH("adapter_layouts", 1, stream,
                   launch_adapter_layouts(A, B, L.m, L.k, L.r, r16, nullptr, nullptr, ws.at, ws.b_pad, stream),
                   "adapter layouts");
    LRQAT_TRY(run_codes_pass(L, Phi0, A, B, ws.at, ws.b_pad, ws.codes, true, dev, stream));
  } else if (!direct) {
    LRQAT_LAUNCH("adapter_layouts", 1, stream,
                 launch_adapter_layouts(A, B, L.m, L.k, L.r, r16, ws.a_pad, ws.bt_pad, nullptr, nullptr, stream),
                 "adapter layouts");
  }
  const uint16_t* tok = X;
  if (quantized) {
    // the caller ran lrqat_act_quant on this X
  } else if (L.act_bits == 8 && L.act_per_token) {
    // X_hat = bf16(s_x[t] X_Z): the per-token scales are folded into the token operand
    LRQAT_LAUNCH("act_quant", 1, stream, launch_act_quant_token(X, T, L.k, ws.x_codes, stream),
                 "activation quantizer");
    tok = ws.x_codes;
  } else if (L.act_bits == 8) {
    LRQAT_LAUNCH("act_quant", 1, stream, launch_act_quant(X, T, L.k, s_x, ws.x_codes, nullptr, stream),
                 "activation quantizer");
    tok = ws.x_codes;
  }
  CUtensorMap tm_tok, tm_phi, tm_rf, tm_sf;
  LRQAT_TRY(encode_2d(&tm_tok, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, tok, L.k, T, L.k * 2, 64, pair ? 112 : 224,
                      CU_TENSOR_MAP_SWIZZLE_128B, "X"));
  if (cb) {
    // the codes as an 8-bit base; the factor maps are not read
    LRQAT_TRY(encode_2d(&tm_phi, CU_TENSOR_MAP_DATA_TYPE_UINT8, ws.codes, L.k, L.m, L.k, 64, 128,
                        CU_TENSOR_MAP_SWIZZLE_64B, "codes"));
    tm_rf = tm_phi;
    tm_sf = tm_phi;
  } else {
    LRQAT_TRY(phi_map(&tm_phi, L, Phi0, 64, false));
  }
  if (cb) {
  } else if (direct) {
    LRQAT_TRY(encode_2d(&tm_rf, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, A, L.r, L.m, L.r * 2, 64, 128,
                        CU_TENSOR_MAP_SWIZZLE_128B, "A"));
    LRQAT_TRY(encode_2d(&tm_sf, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, B, L.k, L.r, L.k * 2, 64,
                        static_cast<uint32_t>(r16), CU_TENSOR_MAP_SWIZZLE_128B, "B"));
  } else {
    LRQAT_TRY(encode_2d(&tm_rf, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, ws.a_pad, 64, L.m, 128, 64, 128,
                        CU_TENSOR_MAP_SWIZZLE_128B, "A (padded)"));
    LRQAT_TRY(encode_2d(&tm_sf, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, ws.bt_pad, 64, L.k, 128, sf_cols(r16),
                        pair ? 32 : 64, sf_swizzle(r16), "B^T (padded)"));
  }
  FusedArgs a{};
  a.rows = static_cast<int32_t>(L.m);
  a.kdim = static_cast<int32_t>(L.k);
  a.T = static_cast<int32_t>(T);
  a.r16 = cb ? 0 : r16;
  a.sf_cols = cb ? 0 : sf_cols(r16);
  a.num_rb = static_cast<int32_t>(L.m / 128);
  a.num_tb = static_cast<int32_t>((T + 447) / 448);
  a.num_tiles = a.num_rb * a.num_tb;
  a.q = make_quant_params(L.bits, cb ? 0 : frac_bits(L), L.alpha, L.r);
  a.s = s;
  a.zero = L.zero;
  a.u_bf16 = cb ? 0 : L.u_bf16;
  a.sf_mn = direct ? 1 : 0;
  a.codes_bias = cb ? static_cast<int32_t>(codes_bias(L)) : 0;
  a.s_ld = L.group_size ? static_cast<int32_t>(L.k / L.group_size) : 0;
  a.group_size = L.group_size;
  a.s_x = L.act_bits == 8 && !L.act_per_token ? s_x : nullptr;
  a.xmask = nullptr;
  a.xmask_ld = 0;
  a.out = Y;
  a.out_ld = L.m;
  a.status = dev->status;
  a.timeout_ns = kWaitTimeoutNs;
  const int fmode = L.group_size ? FUSED_FWD_GROUP : FUSED_FWD_PC;
  const int ffmt = cb ? LRQAT_PHI_QFIXED : L.phi_format;
  if (pair && L.group_size) {
    // the pair kernel's producers read the group scales as bf16 rows [groups][m], staged per stage
    const int groups = static_cast<int>(L.k / L.group_size);
    LRQAT_LAUNCH("scale_rows", 1, stream,
                 launch_dx_scales(s, L.zero, L.m, groups, groups, ws.s_bf16, ws.z_bf16, stream), "scale rows");
    a.s_bf16 = ws.s_bf16;
    a.z_bf16 = ws.z_bf16;
  }
  if (pair) {
    const int64_t tiles = (L.m / 256) * ((T + kPairTokens - 1) / kPairTokens);
    const int npairs = static_cast<int>(tiles < dev->sms / 2 ? tiles : dev->sms / 2);
    LRQAT_LAUNCH("fused_fwd", 1, stream, launch_fused_pair(fmode, ffmt, tm_tok, tm_phi, tm_rf, tm_sf, a, npairs, stream),
                 "fused forward launch (CTA pairs)");
  } else {
    const int grid = a.num_tiles < dev->sms ? a.num_tiles : dev->sms;
    LRQAT_LAUNCH("fused_fwd", 1, stream, launch_fused(fmode, ffmt, tm_tok, tm_phi, tm_rf, tm_sf, a, grid, stream),
                 "fused forward launch");
  }
  return LRQAT_OK;
}

int lrqat_linear_fwd(const lrqat_layer* layer, int64_t T, const uint16_t* X, const void* Phi0, const float* s,
                     const uint16_t* A, const uint16_t* B, const float* s_x, uint16_t* Y, void* workspace,
                     size_t workspace_bytes, lrqat_stream_t stream) {
  return linear_fwd_impl(layer, T, X, false, Phi0, s, A, B, s_x, Y, workspace, workspace_bytes, true, stream);
}

int lrqat_linear_fwd_quantized(const lrqat_layer* layer, int64_t T, const uint16_t* X_q, const void* Phi0,
                               const float* s, const uint16_t* A, const uint16_t* B, const float* s_x, uint16_t* Y,
                               void* workspace, size_t workspace_bytes, lrqat_stream_t stream) {
  return linear_fwd_impl(layer, T, X_q, true, Phi0, s, A, B, s_x, Y, workspace, workspace_bytes, true, stream);
}

size_t lrqat_bwd_workspace_bytes(const lrqat_layer* layer, int64_t T) {
  if (validate_layer(layer) != LRQAT_OK || T < 1) return 0;
  DeviceInfo* dev = nullptr;
  int sms = 152;
  if (device_info(&dev) == LRQAT_OK) sms = dev->sms;
  const bool pair = use_pair_dw(*layer);
  int pairs = sms / 2;
  if (pair && dev) pairs = dw_pair_max_pairs();
  if (pair && pairs < 1) return 0;
  return bwd_ws_layout(*layer, T, plan_dw(*layer, T, pair ? pairs : sms, pair), nullptr, nullptr);
}

// quantized: X is already the activation quantizer's output (as for linear_fwd_impl) and
// x_mask its clip mask (per tensor).
static int linear_bwd_impl(const lrqat_layer* layer, int64_t T, const uint16_t* dY, const uint16_t* X, bool quantized,
                           const uint32_t* x_mask, const void* Phi0, const float* s, const uint16_t* A,
                           const uint16_t* B, const float* s_x, uint16_t* dX, float* dA, float* dB, float* ds,
                           int accumulate, void* workspace, size_t workspace_bytes, lrqat_stream_t stream) {
  LRQAT_TRY(validate_layer(layer));
  const lrqat_layer& L = *layer;
  if (quantized) {
    if (L.act_bits != 8)
      return fail(LRQAT_ERR_INVALID_ARG, "quantized activations need act_bits == 8 (got %d)", L.act_bits);
    if (!L.act_per_token && !x_mask)
      return fail(LRQAT_ERR_INVALID_ARG, "the clip mask is required for per-tensor quantized activations");
    if (x_mask && (reinterpret_cast<uintptr_t>(x_mask) & 3u))
      return fail(LRQAT_ERR_ALIGNMENT, "mask is not 4-byte aligned");
  }
  if (T < 1) return fail(LRQAT_ERR_INVALID_ARG, "T must be >= 1 (T=%lld)", (long long)T);
  if (T > (int64_t)1 << 30) return fail(LRQAT_ERR_UNSUPPORTED, "T too large");
  LRQAT_CHECK_PTR(dY, "dY");
  LRQAT_CHECK_PTR(X, "X");
  LRQAT_CHECK_PTR(Phi0, "Phi0");
  LRQAT_CHECK_PTR(s, "s");
  if (!A) return fail(LRQAT_ERR_INVALID_ARG, "A is NULL");
  if (!B) return fail(LRQAT_ERR_INVALID_ARG, "B is NULL");
  LRQAT_CHECK_PTR(dX, "dX");
  // the gradient reduction reads and writes dA and dB with 16-byte accesses; ds is written
  // as scalars
  LRQAT_CHECK_PTR(dA, "dA");
  LRQAT_CHECK_PTR(dB, "dB");
  if (!ds) return fail(LRQAT_ERR_INVALID_ARG, "ds is NULL");
  if (L.act_bits == 8 && !L.act_per_token && !s_x)
    return fail(LRQAT_ERR_INVALID_ARG, "s_x is required when act_bits == 8 (per-tensor scale)");
  DeviceInfo* dev = nullptr;
  LRQAT_TRY(device_info(&dev));
  const bool dw_pair = use_pair_dw(L);
  const int dw_pairs = dw_pair ? dw_pair_max_pairs() : 0;
  if (dw_pair && dw_pairs < 1) return fail(LRQAT_ERR_CUDA, "no cluster of two fits the dW kernel");
  const DwPlan plan = plan_dw(L, T, dw_pair ? dw_pairs : dev->sms, dw_pair);
  const size_t need = bwd_ws_layout(L, T, plan, nullptr, nullptr);
  if (!workspace || workspace_bytes < need)
    return fail(LRQAT_ERR_WORKSPACE, "backward workspace of %zu bytes required, %zu given", need,
                workspace ? workspace_bytes : (size_t)0);
  if (!aligned16(workspace)) return fail(LRQAT_ERR_ALIGNMENT, "workspace is not 16-byte aligned");

  BwdWs ws;
  bwd_ws_layout(L, T, plan, workspace, &ws);
  const int r16 = round16(L.r);
  // the transposed base of a packed layer holds one int8 code per byte
  const int fmt_t = L.phi_format == LRQAT_PHI_INT_PACKED ? LRQAT_PHI_QFIXED : L.phi_format;
  // with direct factors the dX GEMM reads its A slices from A itself; its row factor stays the
  // padded B^T, and dW takes A^T and B padded
  // cb: the dX GEMM reads the codes (lrqat_set_lowrank_path); cbw: so does dW (ranks above 64)
  const bool cb = codes_gemm(L, T);
  const bool cbw = codes_dw(L);
  const bool direct = !cb && direct_factors(L, A, B);
  if (cb && direct_factors(L, A, B)) {
    // the codes of every weight from A and B themselves, then one launch for A^T and B padded
    // (dW's operands) and the transposed codes (the dX GEMM's base)
    LRQAT_TRY(run_codes_pass(L, Phi0, A, B, ws.at, ws.b_pad, ws.codes, !cbw, dev, stream));
    LRQAT_LAUNCH("bwd_prep", 1, stream,
                 launch_bwd_prep(A, B, L.m, L.k, L.r, r16, nullptr, nullptr, ws.at, ws.b_pad, ws.codes,
                                 LRQAT_PHI_QFIXED, ws.phit, stream, cbw ? L.bits : 0),
                 "adapter layouts and transposed codes");
  } else if (cb) {
    // the codes of every weight, then their transpose for the dX GEMM; A^T and B padded serve
    // the code pass and dW
    LRQAT_LAUNCH("adapter_layouts", 1, stream,
                 launch_adapter_layouts(A, B, L.m, L.k, L.r, r16, nullptr, nullptr, ws.at, ws.b_pad, stream),
                 "adapter layouts");
    LRQAT_TRY(run_codes_pass(L, Phi0, A, B, ws.at, ws.b_pad, ws.codes, !cbw, dev, stream));
    LRQAT_LAUNCH("bwd_prep", 1, stream,
                 launch_bwd_prep(A, B, L.m, L.k, L.r, r16, nullptr, nullptr, nullptr, nullptr, ws.codes,
                                 LRQAT_PHI_QFIXED, ws.phit, stream, cbw ? L.bits : 0),
                 "transposed codes");
  } else {
    LRQAT_LAUNCH("bwd_prep", 1, stream,
                 launch_bwd_prep(A, B, L.m, L.k, L.r, r16, direct ? nullptr : ws.a_pad, ws.bt_pad, ws.at, ws.b_pad,
                                 Phi0, L.phi_format, ws.phit, stream),
                 "adapter layouts and transposed base");
  }
  const uint16_t* xop = X;
  const uint32_t* xmask = nullptr;
  if (quantized) {
    xmask = L.act_per_token ? nullptr : x_mask;
  } else if (L.act_bits == 8 && L.act_per_token) {
    // dW takes X_hat = bf16(s_x[t] X_Z); absmax scaling never clips, so dX needs no mask
    LRQAT_LAUNCH("act_quant", 1, stream, launch_act_quant_token(X, T, L.k, ws.x_codes, stream),
                 "activation quantizer");
    xop = ws.x_codes;
  } else if (L.act_bits == 8) {
    LRQAT_LAUNCH("act_quant", 1, stream, launch_act_quant(X, T, L.k, s_x, ws.x_codes, ws.xmask, stream),
                 "activation quantizer");
    xop = ws.x_codes;
    xmask = ws.xmask;
  }
  // the codes base has no fraction bits
  const QuantParams q = make_quant_params(L.bits, cb ? 0 : frac_bits(L), L.alpha, L.r);
  const QuantParams qw = make_quant_params(L.bits, cbw ? 0 : frac_bits(L), L.alpha, L.r);

  // dX = dY W_hat (W_hat^T produced on chip from Phi0^T, B^T and A).
  {
    const int groups = L.group_size ? static_cast<int>(L.k / L.group_size) : 1;
    LRQAT_LAUNCH("dx_scales", 1, stream,
                 launch_dx_scales(s, L.zero, L.m, groups, L.group_size ? groups : 0, ws.s_bf16, ws.z_bf16, stream),
                 "dX scale rows");
    const bool pair = use_pair(L.k);
    CUtensorMap tm_tok, tm_phi, tm_rf, tm_sf;
    LRQAT_TRY(encode_2d(&tm_tok, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, dY, L.m, T, L.m * 2, 64, pair ? 112 : 224,
                        CU_TENSOR_MAP_SWIZZLE_128B, "dY"));
    if (phi_16bit(L) && !cb)
      LRQAT_TRY(encode_2d(&tm_phi, CU_TENSOR_MAP_DATA_TYPE_UINT16, ws.phit, L.m, L.k, L.m * 2, 64, 128,
                          CU_TENSOR_MAP_SWIZZLE_128B, "Phi0^T (16-bit)"));
    else
      LRQAT_TRY(encode_2d(&tm_phi, CU_TENSOR_MAP_DATA_TYPE_UINT8, ws.phit, L.m, L.k, L.m, 64, 128,
                          CU_TENSOR_MAP_SWIZZLE_64B, "Phi0^T"));
    if (cb) {   // no factors are read
      tm_rf = tm_phi;
      tm_sf = tm_phi;
    } else {
    LRQAT_TRY(encode_2d(&tm_rf, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, ws.bt_pad, 64, L.k, 128, 64, 128,
                        CU_TENSOR_MAP_SWIZZLE_128B, "B^T (padded)"));
    if (direct)
      LRQAT_TRY(encode_2d(&tm_sf, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, A, L.r, L.m, L.r * 2, sf_cols(r16),
                          pair ? 32 : 64, sf_swizzle(r16), "A"));
    else
      LRQAT_TRY(encode_2d(&tm_sf, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, ws.a_pad, 64, L.m, 128, sf_cols(r16),
                          pair ? 32 : 64, sf_swizzle(r16), "A (padded)"));
    }
    FusedArgs a{};
    a.rows = static_cast<int32_t>(L.k);
    a.kdim = static_cast<int32_t>(L.m);
    a.T = static_cast<int32_t>(T);
    a.r16 = cb ? 0 : r16;
    a.sf_cols = cb ? 0 : sf_cols(r16);
    a.num_rb = static_cast<int32_t>(L.k / 128);
    a.num_tb = static_cast<int32_t>((T + 447) / 448);
    a.num_tiles = a.num_rb * a.num_tb;
    a.q = q;
    a.s = s;
    a.zero = L.zero;
    a.u_bf16 = cb ? 0 : L.u_bf16;
    a.sf_mn = 0;
    a.codes_bias = cb ? static_cast<int32_t>(codes_bias(L)) : 0;   // ranks above 64: clipped and biased in the transpose
    a.s_bf16 = ws.s_bf16;
    a.z_bf16 = ws.z_bf16;
    a.s_ld = L.group_size ? static_cast<int32_t>(L.k / L.group_size) : 0;
    a.group_size = L.group_size;
    a.s_x = nullptr;
    a.xmask = L.act_bits == 8 && !L.act_per_token ? xmask : nullptr;
    a.xmask_ld = static_cast<int32_t>((T + 31) / 32);
    a.out = dX;
    a.out_ld = L.k;
    a.status = dev->status;
    a.timeout_ns = kWaitTimeoutNs;
    const int dfmt = cb ? LRQAT_PHI_QFIXED : fmt_t;
    if (pair) {
      const int64_t tiles = (L.k / 256) * ((T + kPairTokens - 1) / kPairTokens);
      const int npairs = static_cast<int>(tiles < dev->sms / 2 ? tiles : dev->sms / 2);
      LRQAT_LAUNCH("fused_dx", 1, stream,
                   launch_fused_pair(FUSED_DX, dfmt, tm_tok, tm_phi, tm_rf, tm_sf, a, npairs, stream),
                   "fused dX launch (CTA pairs)");
    } else {
      const int grid = a.num_tiles < dev->sms ? a.num_tiles : dev->sms;
      LRQAT_LAUNCH("fused_dx", 1, stream, launch_fused(FUSED_DX, dfmt, tm_tok, tm_phi, tm_rf, tm_sf, a, grid, stream),
                   "fused dX launch");
    }
  }
  // G = dY^T X_hat in TMEM, STE epilogue -> partials of dA, dB, ds.
  {
    CUtensorMap tm_dy, tm_x, tm_at, tm_phi, tm_b;
    LRQAT_TRY(encode_2d(&tm_dy, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, dY, L.m, T, L.m * 2, 64,
                        static_cast<uint32_t>(plan.bkt), CU_TENSOR_MAP_SWIZZLE_128B, "dY (dW)"));
    LRQAT_TRY(encode_2d(&tm_x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, xop, L.k, T, L.k * 2, 64,
                        static_cast<uint32_t>(plan.bkt), CU_TENSOR_MAP_SWIZZLE_128B, "X (dW)"));
    // the codes base: boxes of 64 rank rows (one round of the adapter contractions)
    const uint32_t rbox_rows = cbw ? 64u : static_cast<uint32_t>(r16);
    LRQAT_TRY(encode_2d(&tm_at, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, ws.at, L.m, r16, L.m * 2, 64, rbox_rows,
                        CU_TENSOR_MAP_SWIZZLE_128B, "A^T"));
    if (cbw)
      LRQAT_TRY(encode_2d(&tm_phi, CU_TENSOR_MAP_DATA_TYPE_UINT8, ws.codes, L.k, L.m, L.k, 128, 128,
                          CU_TENSOR_MAP_SWIZZLE_128B, "codes"));
    else
      LRQAT_TRY(phi_map(&tm_phi, L, Phi0, 128, true));
    LRQAT_TRY(encode_2d(&tm_b, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, ws.b_pad, L.k, r16, L.k * 2, 64, rbox_rows,
                        CU_TENSOR_MAP_SWIZZLE_128B, "B (padded)"));
    DwArgs a{};
    a.m = static_cast<int32_t>(L.m);
    a.k = static_cast<int32_t>(L.k);
    a.T = static_cast<int32_t>(T);
    a.r = L.r;
    a.r16 = r16;
    a.nchunks = plan.nchunks;
    a.ni = plan.ni;
    a.nj = plan.nj;
    a.nsplit = plan.nsplit;
    a.tchunk = plan.tchunk;
    a.num_units = plan.units;
    a.q = qw;
    a.s = s;
    a.zero = L.zero;
    a.u_bf16 = cbw ? 0 : L.u_bf16;
    a.s_ld = L.group_size ? static_cast<int32_t>(L.k / L.group_size) : 0;
    a.group_size = L.group_size;
    a.s_x = L.act_bits == 8 && !L.act_per_token ? s_x : nullptr;   // per token: folded into X_hat
    a.dA_part = ws.dA_part;
    a.dB_part = ws.dB_part;
    a.ds_part = ws.ds_part;
    a.status = dev->status;
    a.timeout_ns = kWaitTimeoutNs;
    a.phi = cbw ? static_cast<const void*>(ws.codes) : Phi0;
    a.sched = plan.sched;
    a.tile_segs = ws.tile_segs;
    a.codes_base = cbw ? 1 : 0;
    const int grid = plan.sched.grid;
    if (plan.pair) {
      // each CTA of a pair loads half of the ranks of the slices that serve as N-split B operands
      CUtensorMap tm_ath, tm_bh;
      LRQAT_TRY(encode_2d(&tm_ath, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, ws.at, L.m, r16, L.m * 2, 64,
                          static_cast<uint32_t>(r16 / 2), CU_TENSOR_MAP_SWIZZLE_128B, "A^T (rank halves)"));
      LRQAT_TRY(encode_2d(&tm_bh, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, ws.b_pad, L.k, r16, L.k * 2, 64,
                          static_cast<uint32_t>(r16 / 2), CU_TENSOR_MAP_SWIZZLE_128B, "B (rank halves)"));
      LRQAT_LAUNCH("fused_dw", 1, stream,
                   launch_dw_pair(L.phi_format, tm_dy, tm_x, tm_at, tm_ath, tm_phi, tm_b, tm_bh, a, grid, stream),
                   "fused dW launch (CTA pairs)");
    } else {
      LRQAT_LAUNCH("fused_dw", 1, stream,
                   launch_dw(cbw ? LRQAT_PHI_QFIXED : L.phi_format, tm_dy, tm_x, tm_at, tm_phi, tm_b, a, grid, stream),
                   "fused dW launch");
    }
  }
  ReduceArgs ra{};
  ra.dA_part = ws.dA_part;
  ra.nA = plan.nj * plan.nsplit;
  ra.dB_part = ws.dB_part;
  ra.nB = plan.ni128 * plan.nsplit;
  ra.ds_part = ws.ds_part;
  ra.nS = 2 * plan.nsplit;
  ra.dA = dA;
  ra.dB = dB;
  ra.ds = ds;
  ra.m = L.m;
  ra.k = L.k;
  ra.r = L.r;
  ra.group_size = L.group_size;
  ra.lr = static_cast<float>(static_cast<double>(L.alpha) / L.r);
  ra.accumulate = accumulate ? 1 : 0;
  ra.sched = plan.sched;
  // the reduction counts 128-row tiles: a whole pair tile is two whole 128-row tiles
  if (plan.pair) ra.sched.full_tiles *= 2;
  ra.ni = plan.ni128;
  ra.nsplit = plan.nsplit;
  ra.bn = 128 * plan.nchunks;
  ra.tile_segs = ws.tile_segs;
  LRQAT_LAUNCH("reduce_grads", 1, stream, launch_reduce(ra, stream), "gradient reduction");
  return LRQAT_OK;
}

int lrqat_linear_bwd(const lrqat_layer* layer, int64_t T, const uint16_t* dY, const uint16_t* X, const void* Phi0,
                     const float* s, const uint16_t* A, const uint16_t* B, const float* s_x, uint16_t* dX, float* dA,
                     float* dB, float* ds, int accumulate, void* workspace, size_t workspace_bytes,
                     lrqat_stream_t stream) {
  return linear_bwd_impl(layer, T, dY, X, false, nullptr, Phi0, s, A, B, s_x, dX, dA, dB, ds, accumulate, workspace,
                         workspace_bytes, stream);
}

int lrqat_linear_bwd_quantized(const lrqat_layer* layer, int64_t T, const uint16_t* dY, const uint16_t* X_q,
                               const uint32_t* mask, const void* Phi0, const float* s, const uint16_t* A,
                               const uint16_t* B, const float* s_x, uint16_t* dX, float* dA, float* dB, float* ds,
                               int accumulate, void* workspace, size_t workspace_bytes, lrqat_stream_t stream) {
  return linear_bwd_impl(layer, T, dY, X_q, true, mask, Phi0, s, A, B, s_x, dX, dA, dB, ds, accumulate, workspace,
                         workspace_bytes, stream);
}

int lrqat_merge(const lrqat_layer* layer, const void* Phi0, const uint16_t* A, const uint16_t* B, int8_t* W_Z,
                lrqat_stream_t stream) {
  LRQAT_TRY(validate_layer(layer));
  const lrqat_layer& L = *layer;
  LRQAT_CHECK_PTR(Phi0, "Phi0");
  if (!A) return fail(LRQAT_ERR_INVALID_ARG, "A is NULL");
  if (!B) return fail(LRQAT_ERR_INVALID_ARG, "B is NULL");
  LRQAT_CHECK_PTR(W_Z, "W_Z");
  const QuantParams q = make_quant_params(L.bits, frac_bits(L), L.alpha, L.r);
  if (direct_factors(L, A, B) && aligned16(Phi0) && aligned16(W_Z)) {
    DeviceInfo* dev = nullptr;
    LRQAT_TRY(device_info(&dev));
    const int r16 = round16(L.r);
    CUtensorMap tm_a, tm_b;
    LRQAT_TRY(encode_2d(&tm_a, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, A, L.r, L.m, L.r * 2, 64, 128,
                        CU_TENSOR_MAP_SWIZZLE_128B, "A"));
    LRQAT_TRY(encode_2d(&tm_b, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, B, L.k, L.r, L.k * 2, 64,
                        static_cast<uint32_t>(r16), CU_TENSOR_MAP_SWIZZLE_128B, "B"));
    CUtensorMap tm_phi;
    LRQAT_TRY(phi_map(&tm_phi, L, Phi0, 128, true));
    MergeArgs a{};
    a.wz = W_Z;
    a.m = L.m;
    a.k = L.k;
    a.r16 = r16;
    a.q = q;
    a.status = dev->status;
    a.timeout_ns = kWaitTimeoutNs;
    LRQAT_LAUNCH("merge", 1, stream, launch_merge_tc(L.phi_format, L.u_bf16, 0, tm_a, tm_b, tm_phi, a, stream),
                 "merge launch");
    return LRQAT_OK;
  }
  LRQAT_LAUNCH("merge", 1, stream,
               launch_merge(Phi0, A, B, L.m, L.k, L.r, L.phi_format, L.u_bf16, q, W_Z, stream),
               "merge launch");
  return LRQAT_OK;
}

int lrqat_grad_sqnorm(const lrqat_layer* layer, const float* dA, const float* dB, const float* ds, float* sqnorm,
                      lrqat_stream_t stream) {
  LRQAT_TRY(validate_layer(layer));
  const lrqat_layer& L = *layer;
  if (!dA || !dB || !ds || !sqnorm) return fail(LRQAT_ERR_INVALID_ARG, "dA, dB, ds and sqnorm must be non-NULL");
  const int64_t ns = L.group_size ? L.m * (L.k / L.group_size) : L.m;
  LRQAT_LAUNCH("grad_sqnorm", 1, stream,
               launch_grad_sqnorm(dA, L.m * L.r, dB, static_cast<int64_t>(L.r) * L.k, ds, ns, sqnorm, stream),
               "gradient norm launch");
  return LRQAT_OK;
}

int lrqat_adamw_step(const lrqat_layer* layer, const lrqat_adamw* opt, const float* sqnorm, const float* dA,
                     const float* dB, const float* ds, const lrqat_adamw_state* state, float* s, uint16_t* A,
                     uint16_t* B, lrqat_stream_t stream) {
  LRQAT_TRY(validate_layer(layer));
  if (!opt || !state) return fail(LRQAT_ERR_INVALID_ARG, "opt and state must be non-NULL");
  if (opt->step < 1) return fail(LRQAT_ERR_INVALID_ARG, "step must be >= 1 (step=%d)", opt->step);
  if (!(opt->beta1 >= 0.0f && opt->beta1 < 1.0f && opt->beta2 >= 0.0f && opt->beta2 < 1.0f))
    return fail(LRQAT_ERR_INVALID_ARG, "betas must lie in [0, 1)");
  if (!(opt->eps > 0.0f)) return fail(LRQAT_ERR_INVALID_ARG, "eps must be positive");
  if (!dA || !dB || !ds || !sqnorm || !s || !A || !B || !state->A32 || !state->B32 || !state->mA || !state->vA ||
      !state->mB || !state->vB || !state->ms || !state->vs)
    return fail(LRQAT_ERR_INVALID_ARG, "gradients, parameters, state arrays and sqnorm must be non-NULL");
  const lrqat_layer& L = *layer;
  AdamwArgs a{};
  a.dA = dA;
  a.dB = dB;
  a.ds = ds;
  a.A32 = state->A32;
  a.B32 = state->B32;
  a.s = s;
  a.mA = state->mA;
  a.vA = state->vA;
  a.mB = state->mB;
  a.vB = state->vB;
  a.ms = state->ms;
  a.vs = state->vs;
  a.A = A;
  a.B = B;
  a.nA = L.m * L.r;
  a.nB = static_cast<int64_t>(L.r) * L.k;
  a.ns = L.group_size ? L.m * (L.k / L.group_size) : L.m;
  a.lr_ab = opt->lr_ab;
  a.lr_s = opt->lr_s;
  a.wd_ab = opt->weight_decay_ab;
  a.wd_s = opt->weight_decay_s;
  a.beta1 = opt->beta1;
  a.beta2 = opt->beta2;
  a.eps = opt->eps;
  a.bc1 = static_cast<float>(1.0 - std::pow(static_cast<double>(opt->beta1), opt->step));
  a.bc2 = static_cast<float>(1.0 - std::pow(static_cast<double>(opt->beta2), opt->step));
  a.max_norm = opt->max_grad_norm;
  a.sqnorm = sqnorm;
  LRQAT_LAUNCH("adamw", 1, stream, launch_adamw(a, stream), "AdamW launch");
  return LRQAT_OK;
}

int lrqat_get_gemm_variant(void) { return g_gemm_variant.load(std::memory_order_relaxed); }
int lrqat_get_lowrank_path(void) { return g_lowrank_path.load(std::memory_order_relaxed); }
int lrqat_get_dw_schedule(void) { return g_dw_schedule.load(std::memory_order_relaxed); }

int lrqat_set_gemm_variant(int variant) {
  if (variant < 0 || variant > 2)
    return fail(LRQAT_ERR_INVALID_ARG, "GEMM variant must be 0, 1 or 2 (got %d)", variant);
  g_gemm_variant.store(variant, std::memory_order_relaxed);
  return LRQAT_OK;
}

int lrqat_set_lowrank_path(int path) {
  if (path < 0 || path > 2) return fail(LRQAT_ERR_INVALID_ARG, "low-rank path must be 0, 1 or 2 (got %d)", path);
  g_lowrank_path.store(path, std::memory_order_relaxed);
  return LRQAT_OK;
}

int lrqat_set_dw_schedule(int schedule) {
  if (schedule < 0 || schedule > 2) return fail(LRQAT_ERR_INVALID_ARG, "dW schedule must be 0, 1 or 2 (got %d)", schedule);
  g_dw_schedule.store(schedule, std::memory_order_relaxed);
  return LRQAT_OK;
}

int lrqat_get_device_status(lrqat_stream_t stream) {
  DeviceInfo* dev = nullptr;
  LRQAT_TRY(device_info(&dev));
  LRQAT_CUDA(cudaStreamSynchronize(stream), "cudaStreamSynchronize");
  int h = 0;
  LRQAT_CUDA(cudaMemcpy(&h, dev->status, sizeof(int), cudaMemcpyDeviceToHost), "read device status");
  if (h != 0) {
    LRQAT_CUDA(cudaMemset(dev->status, 0, sizeof(int)), "clear device status");
    return fail(LRQAT_ERR_TIMEOUT, "a kernel's bounded wait gave up (status word 0x%x)", h);
  }
  return LRQAT_OK;
}

int lrqat_trace_enable(int enable) {
  std::lock_guard<std::mutex> lock(g_trace_mu);
  if (enable) trace_clear_locked();
  g_trace_on = enable != 0;
  return LRQAT_OK;
}

int lrqat_trace_read(int max_entries, const char** names, int64_t* launches, double* total_ms, int* count) {
  if (max_entries < 0 || (max_entries > 0 && (!names || !launches || !total_ms)) || !count)
    return fail(LRQAT_ERR_INVALID_ARG, "trace_read: bad output arrays");
  std::lock_guard<std::mutex> lock(g_trace_mu);
  std::vector<const char*> keys;
  std::vector<int64_t> n;
  std::vector<double> ms;
  for (auto& r : g_trace) {
    cudaError_t e = cudaEventSynchronize(r.stop);
    if (e != cudaSuccess) return cuda_fail(e, "trace_read: cudaEventSynchronize");
    float t = 0.0f;
    e = cudaEventElapsedTime(&t, r.start, r.stop);
    if (e != cudaSuccess) return cuda_fail(e, "trace_read: cudaEventElapsedTime");
    size_t i = 0;
    while (i < keys.size() && std::strcmp(keys[i], r.name) != 0) ++i;
    if (i == keys.size()) {
      keys.push_back(r.name);
      n.push_back(0);
      ms.push_back(0.0);
    }
    n[i] += r.kernels;
    ms[i] += t;
  }
  *count = static_cast<int>(keys.size());
  for (int i = 0; i < max_entries && i < static_cast<int>(keys.size()); ++i) {
    names[i] = keys[i];
    launches[i] = n[i];
    total_ms[i] = ms[i];
  }
  return LRQAT_OK;
}

}  // extern "C"
