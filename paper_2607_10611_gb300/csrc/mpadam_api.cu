// mpadam_api.cu -- host side of the C ABI declared in include/mpadam.h, plus
// the small auxiliary kernels (E4M3 scale-state seeding, random-lane dump,
// table fills of the allocation-free step).  The fused step kernel itself
// lives in step_kernel.cuh.
#include <cuda_runtime.h>
#include <sys/mman.h>
#include <sys/syscall.h>
#include <unistd.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <vector>

#include "mpadam.h"
#include "step_args.h"
#include "step_kernel.cuh"
#include "toy.h"

using mpadam::StepArgs;
using mpadam::StepScalars;
using mpadam::TensorAux;
using mpadam::TensorDesc;

namespace {

thread_local std::string g_last_error;

// Allocation-failure injection for the tests (mpadam_debug_fail_allocation):
// the allocation after `countdown` more successful ones fails, once.
std::atomic<int32_t> g_fail_countdown{-1};

bool injected_failure() {
  int32_t c = g_fail_countdown.load();
  while (c >= 0) {
    if (g_fail_countdown.compare_exchange_weak(c, c - 1)) return c == 0;
  }
  return false;
}

// Every device and pinned allocation of the library goes through these.
cudaError_t dev_malloc(void** p, size_t bytes) {
  if (injected_failure()) { *p = nullptr; return cudaErrorMemoryAllocation; }
  return cudaMalloc(p, bytes);
}
template <typename T>
cudaError_t dev_malloc(T** p, size_t bytes) {
  return dev_malloc(reinterpret_cast<void**>(p), bytes);
}
cudaError_t host_malloc(void** p, size_t bytes) {
  if (injected_failure()) { *p = nullptr; return cudaErrorMemoryAllocation; }
  return cudaMallocHost(p, bytes);
}

int32_t fail(int32_t code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return code;
}

int32_t cuda_fail(cudaError_t e, const char* what) {
  return fail(MPADAM_ECUDA, "%s: %s (%s)", what, cudaGetErrorString(e), cudaGetErrorName(e));
}

size_t elem_size(int32_t dt) { return dt == MPADAM_F32 ? 4 : (dt == MPADAM_BF16 ? 2 : 1); }

// Bytes of n stored weights (NVFP4: two per byte).
size_t weight_bytes(int32_t wd, int64_t n) {
  return wd == MPADAM_NVFP4 ? (size_t)((n + 1) / 2) : (size_t)n * elem_size(wd);
}

bool is_aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Per-step binary32 scalars of the canonical update, from binary64.
float toward_zero(double x) {
  float f = static_cast<float>(x);
  if (x > 0.0 && static_cast<double>(f) > x) f = std::nextafter(f, 0.0f);
  if (x < 0.0 && static_cast<double>(f) < x) f = std::nextafter(f, 0.0f);
  return f;
}

void make_scalars(const mpadam_config& c, int64_t t, StepScalars* s) {
  double bc1 = 1.0, bc2 = 1.0;
  if (c.bias_correction) {
    bc1 = 1.0 - std::pow(static_cast<double>(c.beta1), static_cast<double>(t));
    bc2 = 1.0 - std::pow(static_cast<double>(c.beta2), static_cast<double>(t));
  }
  s->b1 = c.beta1;
  s->b2 = c.beta2;
  s->omb1 = static_cast<float>(1.0 - static_cast<double>(c.beta1));
  s->omb2 = static_cast<float>(1.0 - static_cast<double>(c.beta2));
  s->ka = static_cast<float>(-static_cast<double>(c.lr_add) / bc1);
  s->c2 = static_cast<float>(1.0 / std::sqrt(bc2));
  s->km = -c.lr_mul;
  s->ln2 = static_cast<float>(0.693147180559945309417232121458);
  s->eps = c.eps;
  s->tau = c.tau;
  const double d = static_cast<double>(c.dmult_max);
  s->hi = toward_zero(std::fmin(static_cast<double>(c.rmax_pos), std::exp2(d) - 1.0));
  s->lo = toward_zero(std::fmax(-static_cast<double>(c.rmax_neg), std::exp2(-d) - 1.0));
  s->gmax_on = std::isfinite(c.g_max) ? 1 : 0;
  s->gmax = s->gmax_on ? c.g_max : 0.0f;
  s->wmax_on = std::isfinite(c.w_max) ? 1 : 0;
  s->wmax = s->wmax_on ? c.w_max : 0.0f;
  s->wd_on = c.wd_add != 0.0f ? 1 : 0;
  s->kwd = static_cast<float>(static_cast<double>(c.lr_add) * static_cast<double>(c.wd_add));
  s->cert_ok = (c.eps >= 0x1p-28f && c.tau >= 0x1p-125f && s->c2 <= 0x1p14f && c.lr_mul <= 4.0f) ? 1 : 0;
}

// Philox4x32-10 round keys: key + r * (0x9E3779B9, 0xBB67AE85), r = 0..9.
void round_keys(uint64_t seed, uint32_t* rk0, uint32_t* rk1) {
  uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
  for (int r = 0; r < mpadam::kPhiloxRounds; ++r) {
    rk0[r] = k0;
    rk1[r] = k1;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
}

// Shared-memory ring of the step kernel: one stage holds one tile of every
// array (w | g | mu | nu | nu_e | block scales); as many stages as fit, 2 to
// kMaxStages.
struct Geometry {
  int32_t stages = 0, stage_bytes = 0, off_g = 0, off_m = 0, off_v = 0, off_ve = 0, off_s = 0, dyn_smem = 0;
};

int32_t make_geometry(const mpadam_config& c, int32_t wd, int dev, Geometry* g);

bool kernel_options(const mpadam_config& c) {
  return std::isfinite(c.g_max) || std::isfinite(c.w_max) || c.wd_add != 0.0f;
}

// per_tensor_weights: the weight formats come with the tensors
// (mpadam_create_ex) and cfg->weight_dtype is not used.
int32_t check_config(const mpadam_config* c, bool per_tensor_weights = false) {
  if (!c) return fail(MPADAM_EINVAL, "config is NULL");
  if (!per_tensor_weights && (c->weight_dtype == MPADAM_E4M3_B32 || c->weight_dtype == MPADAM_NVFP4))
    return fail(MPADAM_EINVAL, "block-scaled weights need their scale arrays: use mpadam_create_ex");
  if (!per_tensor_weights && c->weight_dtype != MPADAM_BF16 && c->weight_dtype != MPADAM_E4M3)
    return fail(MPADAM_EINVAL, "weight_dtype must be MPADAM_BF16 or MPADAM_E4M3 (got %d)", c->weight_dtype);
  if (c->grad_dtype != MPADAM_F32 && c->grad_dtype != MPADAM_BF16)
    return fail(MPADAM_EINVAL, "grad_dtype must be MPADAM_F32 or MPADAM_BF16 (got %d)", c->grad_dtype);
  if (c->moment_dtype != MPADAM_F32 && c->moment_dtype != MPADAM_BF16)
    return fail(MPADAM_EINVAL, "moment_dtype must be MPADAM_F32 or MPADAM_BF16 (got %d)", c->moment_dtype);
  if (c->rounding != MPADAM_ROUND_NEAREST && c->rounding != MPADAM_ROUND_STOCHASTIC)
    return fail(MPADAM_EINVAL, "rounding must be nearest (0) or stochastic (1) (got %d)", c->rounding);
  if (c->bias_correction != 0 && c->bias_correction != 1)
    return fail(MPADAM_EINVAL, "bias_correction must be 0 or 1");
  if (c->reserved != 0) return fail(MPADAM_EINVAL, "reserved must be 0");
  auto fin_nonneg = [](float x) { return std::isfinite(x) && x >= 0.0f; };
  auto fin_pos = [](float x) { return std::isfinite(x) && x > 0.0f; };
  if (!fin_nonneg(c->lr_add)) return fail(MPADAM_EINVAL, "lr_add must be finite and >= 0");
  if (!fin_nonneg(c->lr_mul)) return fail(MPADAM_EINVAL, "lr_mul must be finite and >= 0");
  if (!(c->beta1 >= 0.0f && c->beta1 < 1.0f)) return fail(MPADAM_EINVAL, "beta1 must be in [0, 1)");
  if (!(c->beta2 >= 0.0f && c->beta2 < 1.0f)) return fail(MPADAM_EINVAL, "beta2 must be in [0, 1)");
  if (!fin_pos(c->eps)) return fail(MPADAM_EINVAL, "eps must be finite and > 0");
  if (!fin_pos(c->tau)) return fail(MPADAM_EINVAL, "tau must be finite and > 0");
  if (!fin_pos(c->rmax_pos)) return fail(MPADAM_EINVAL, "rmax_pos must be finite and > 0");
  if (!(fin_pos(c->rmax_neg) && c->rmax_neg < 1.0f)) return fail(MPADAM_EINVAL, "rmax_neg must be in (0, 1)");
  if (!(c->g_max > 0.0f)) return fail(MPADAM_EINVAL, "g_max must be > 0 (+inf = off)");
  if (!(c->dmult_max > 0.0f)) return fail(MPADAM_EINVAL, "dmult_max must be > 0 (+inf = off)");
  if (!(c->w_max > 0.0f)) return fail(MPADAM_EINVAL, "w_max must be > 0 (+inf = off)");
  if (!fin_nonneg(c->wd_add)) return fail(MPADAM_EINVAL, "wd_add must be finite and >= 0");
  return MPADAM_OK;
}

int32_t make_geometry(const mpadam_config& c, int32_t wd, int dev, Geometry* g) {
  const int32_t rw = (int32_t)weight_bytes(wd, mpadam::kTile);
  const int32_t rg = mpadam::kTile * (int32_t)elem_size(c.grad_dtype);
  const int32_t rm = mpadam::kTile * (int32_t)elem_size(c.moment_dtype);
  const int32_t rs = wd == MPADAM_E4M3_B32 ? mpadam::kTileBlocks * 2           // 240 bytes, a 16-byte multiple
                   : wd == MPADAM_NVFP4    ? mpadam::kTileFp4Blocks               // 240 bytes
                                           : 0;
  g->off_g = rw;
  g->off_m = rw + rg;
  g->off_v = g->off_m + rm;
  g->off_ve = g->off_v + rm;
  g->off_s = g->off_ve + rm;
  g->stage_bytes = g->off_s + rs;
  int optin = 0;
  cudaError_t e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute(MaxSharedMemoryPerBlockOptin)");
  const int32_t budget = optin - 1024;  // static barriers (128 bytes) and slack
  g->stages = std::min<int32_t>(mpadam::kMaxStages, budget / g->stage_bytes);
  if (g->stages < 2) return fail(MPADAM_EUNSUPPORTED, "device shared memory too small for the step pipeline");
  g->dyn_smem = g->stages * g->stage_bytes;
  return MPADAM_OK;
}

// ---------------------------------------------------------------------------
// Auxiliary kernels
// ---------------------------------------------------------------------------

// Largest |decoded stored E4M3 weight| of each tensor -> fp8_amax[slot], over
// the same per-CTA tile ranges as the step kernel (kConsumers threads; thread
// c reads the 8 codes [8c, 8c + 8) of each tile).  Launched over the
// per-tensor-scaled E4M3 tensors only; rings are indexed by list position.
__global__ void __launch_bounds__(mpadam::kConsumers) fp8_amax_kernel(const __grid_constant__ StepArgs a,
                                                                      int32_t exp_slot, int32_t amax_slot) {
  const int64_t T = a.total_tiles;
  const int64_t tb = a.tile_base + (int64_t)blockIdx.x * T / gridDim.x;
  const int64_t te = a.tile_base + ((int64_t)blockIdx.x + 1) * T / gridDim.x;
  if (tb >= te) return;
  const int n = a.n_tensors;
  int k = a.cta_first[blockIdx.x];
  TensorDesc d = a.desc[k];
  int64_t tiles = (d.numel + mpadam::kTile - 1) / mpadam::kTile;
  uint32_t mag = 0;
  for (int64_t t = tb; t < te; ++t) {
    if (t >= d.tile_off + tiles) {
      const uint32_t wmag = __reduce_max_sync(0xFFFFFFFFu, mag);
      if ((threadIdx.x & 31) == 0 && wmag != 0u) {
        const int32_t e = a.fp8_exp[(int64_t)exp_slot * n + d.ring];
        const float v = __fmul_rn(mpadam::e4m3_value(wmag), mpadam::pow2f(e));
        atomicMax(&a.fp8_amax[(int64_t)amax_slot * n + d.ring], __float_as_uint(v));
      }
      mag = 0;
      do {
        ++k;
        d = a.desc[k];
        tiles = (d.numel + mpadam::kTile - 1) / mpadam::kTile;
      } while (t >= d.tile_off + tiles);
    }
    const int64_t e0 = (t - d.tile_off) * mpadam::kTile + mpadam::kGroup * (int64_t)threadIdx.x;
    const uint8_t* q = static_cast<const uint8_t*>(d.w);
    for (int j = 0; j < mpadam::kGroup; ++j) {
      if (e0 + j < d.numel) {
        const uint32_t c = q[e0 + j] & 0x7Fu;
        if (c != 0x7Fu) mag = max(mag, c);  // E4M3 magnitude order = code order
      }
    }
  }
  const uint32_t wmag = __reduce_max_sync(0xFFFFFFFFu, mag);
  if ((threadIdx.x & 31) == 0 && wmag != 0u) {
    const int32_t e = a.fp8_exp[(int64_t)exp_slot * n + d.ring];
    const float v = __fmul_rn(mpadam::e4m3_value(wmag), mpadam::pow2f(e));
    atomicMax(&a.fp8_amax[(int64_t)amax_slot * n + d.ring], __float_as_uint(v));
  }
}

struct RngArgs {
  uint32_t rk0[mpadam::kPhiloxRounds], rk1[mpadam::kPhiloxRounds];
  uint32_t t_lo, t_hi;
  int32_t bf16;
  uint64_t first;
  int64_t n;
  uint32_t* out;
};

__global__ void rng_lanes_kernel(const __grid_constant__ RngArgs a) {
  for (int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; k < a.n;
       k += (int64_t)gridDim.x * blockDim.x) {
    const uint64_t i = a.first + (uint64_t)k;
    const uint64_t blk = a.bf16 ? (i >> 3) : (i >> 2);
    const uint4 r = mpadam::philox4x32_10((uint32_t)blk, (uint32_t)(blk >> 32), a.t_lo, a.t_hi, a.rk0, a.rk1);
    const uint32_t lane = a.bf16 ? (uint32_t)(i & 7) : (uint32_t)(i & 3);
    const uint32_t word_idx = a.bf16 ? (lane >> 1) : lane;
    const uint32_t word = word_idx == 0 ? r.x : (word_idx == 1 ? r.y : (word_idx == 2 ? r.z : r.w));
    a.out[k] = a.bf16 ? ((lane & 1) ? (word >> 16) : (word & 0xFFFFu)) : word;
  }
}

}  // namespace

// ---------------------------------------------------------------------------
// State
//
// A tensor list is stepped by one kernel launch per weight format present
// (a "group"): the descriptor, aux and gradient tables are stored in group
// order (group 0's tensors first, each group in list order), every group
// numbers its own tiles from 0 and has its own per-CTA start table.  Global
// element indices and the E4M3 scale rings follow list positions.
// ---------------------------------------------------------------------------
struct Group {
  int32_t wd = 0;                 // weight format of the launch
  int32_t first = 0, count = 0;   // positions [first, first + count) of the group-ordered tables
  int64_t tiles = 0;
  std::vector<int64_t> numel;     // of its tensors, in order
  bool aux = false;               // the launch reads the aux table
  const void* kernel = nullptr;
  Geometry geo;
  int32_t default_grid = 0, grid = 0;
  int32_t* d_cta_first = nullptr;
  int32_t cta_cap = 0;
  mpadam::PoolChunk* d_pool = nullptr;  // tail pool of the current grid (none when static_q is 1024)
  int32_t pool_chunks = 0, pool_cap = 0;
  std::vector<TensorDesc> h_desc;       // host copies of its table entries (inline in short launches)
  std::vector<TensorAux> h_aux;
};

struct mpadam_state {
  int32_t n = 0;
  mpadam_config cfg{};
  std::vector<int32_t> wdt;                    // weight format of each tensor (list order)
  std::vector<int64_t> numel, goff, tile_off;  // list order; tile_off in its group's numbering
  std::vector<void*> w;
  std::vector<int32_t> order;                  // group-ordered position -> list position
  std::vector<Group> groups;
  int64_t length = 0;  // padded global index space
  int device = 0;
  int sm_count = 0;
  TensorDesc* d_desc = nullptr;
  TensorAux* d_aux = nullptr;
  const void** d_grads = nullptr;
  int32_t* d_err = nullptr;        // device error bits of the step kernel
  const void** h_grads = nullptr;  // pinned staging of the grad pointer table (group order)
  std::vector<const void*> last_grads;
  bool grads_uploaded = false;
  cudaEvent_t upload_done = nullptr;
  bool upload_pending = false;
  int32_t* fp8_exp = nullptr;
  uint32_t* fp8_amax = nullptr;
  char* d_gstage = nullptr;  // mpadam_step_host gradient staging (global-index layout)
  std::vector<const void*> stage_ptrs;
  // mpadam_step_host pipeline (single-group states): chunks of whole tiles, copied and stepped in turn
  cudaStream_t s_h2d = nullptr, s_d2h = nullptr;
  std::vector<cudaEvent_t> ev;                // per chunk: h2d done, kernel done; plus start / end
  std::vector<int64_t> chunk_tile;            // chunk c covers tiles [chunk_tile[c], chunk_tile[c+1])
  std::vector<int64_t> chunk_elem;            // and global elements [chunk_elem[2c], chunk_elem[2c+1])
  int32_t* d_chunk_first = nullptr;           // [chunks][grid] CTA start tensors
  // tail pool of mpadam_step's launches: static prefix of each CTA's range (1/1024) and chunk length;
  // until set_tail_pool is called, groups of fewer than kPoolMinTilesPerCta tiles per CTA keep
  // static runs (with a tile or two per CTA, greedy claims would pile chunks on a few CTAs)
  int32_t pool_q = 768, pool_chunk = 4;
  bool pool_set = false;
  uint32_t* d_pool_next = nullptr;            // [groups] claim counters, zeroed before each step
};

namespace {

void release_pipeline(mpadam_state* s) {
  if (s->d_chunk_first) cudaFree(s->d_chunk_first);
  s->d_chunk_first = nullptr;
  for (cudaEvent_t e : s->ev) cudaEventDestroy(e);
  s->ev.clear();
  if (s->s_h2d) cudaStreamDestroy(s->s_h2d);
  if (s->s_d2h) cudaStreamDestroy(s->s_d2h);
  s->s_h2d = s->s_d2h = nullptr;
  s->chunk_tile.clear();
  s->chunk_elem.clear();
}

void release(mpadam_state* s) {
  if (!s) return;
  if (s->d_desc) cudaFree(s->d_desc);
  if (s->d_aux) cudaFree(s->d_aux);
  if (s->d_grads) cudaFree(const_cast<void**>(s->d_grads));
  for (auto& g : s->groups) {
    if (g.d_cta_first) cudaFree(g.d_cta_first);
    if (g.d_pool) cudaFree(g.d_pool);
  }
  if (s->d_pool_next) cudaFree(s->d_pool_next);
  if (s->d_err) cudaFree(s->d_err);
  if (s->d_gstage) cudaFree(s->d_gstage);
  release_pipeline(s);
  if (s->h_grads) cudaFreeHost(const_cast<void**>(s->h_grads));
  if (s->upload_done) cudaEventDestroy(s->upload_done);
  delete s;
}

int64_t tiles_of(int64_t numel) { return (numel + mpadam::kTile - 1) / mpadam::kTile; }

// Tensor holding each CTA's first tile of the range [tile_base, tile_base +
// total_tiles) (n when the CTA has no tiles).
void cta_first_table(const int64_t* numel, int32_t n, int64_t total_tiles, int32_t grid, int32_t* first,
                     int64_t tile_base = 0) {
  int32_t k = 0;
  int64_t tile_off = 0;
  for (int32_t b = 0; b < grid; ++b) {
    const int64_t tb = tile_base + (int64_t)b * total_tiles / grid;
    while (k < n && tile_off + tiles_of(numel[k]) <= tb) {
      tile_off += tiles_of(numel[k]);
      ++k;
    }
    first[b] = k;
  }
}

int32_t upload_cta_table(Group& g, int32_t grid) {
  if (grid > g.cta_cap) {
    if (g.d_cta_first) cudaFree(g.d_cta_first);
    g.d_cta_first = nullptr;
    g.cta_cap = 0;
    if (dev_malloc(&g.d_cta_first, sizeof(int32_t) * grid) != cudaSuccess)
      return fail(MPADAM_EALLOC, "cudaMalloc of %d CTA entries failed", grid);
    g.cta_cap = grid;
  }
  std::vector<int32_t> first(grid);
  cta_first_table(g.numel.data(), g.count, g.tiles, grid, first.data());
  cudaError_t e = cudaMemcpy(g.d_cta_first, first.data(), sizeof(int32_t) * grid, cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(e, "upload of the CTA table");
  g.grid = grid;
  return MPADAM_OK;
}

// The tail pool of `grid` CTAs over a list of `count` tensors (numel) with
// `tiles` tiles in all: CTA b keeps the first (te - tb) * q / 1024 tiles of
// its range [tb, te) (the kernel computes the same split) and the rest of
// every range becomes chunks of at most `chunk` tiles, in tile order, each
// with the tensor holding its first tile.  Host only.
void pool_host(const int64_t* numel, int32_t count, int64_t tiles, int32_t grid, int32_t q, int32_t chunk,
               std::vector<mpadam::PoolChunk>& pool) {
  pool.clear();
  if (q >= 1024 || tiles == 0) return;
  int32_t k = 0;
  int64_t tile_off = 0;
  auto tensor_of = [&](int64_t t) {  // t never decreases across calls
    while (k < count && tile_off + tiles_of(numel[k]) <= t) {
      tile_off += tiles_of(numel[k]);
      ++k;
    }
    return k;
  };
  for (int32_t b = 0; b < grid; ++b) {
    const int64_t tb = (int64_t)b * tiles / grid, te = ((int64_t)b + 1) * tiles / grid;
    for (int64_t t = tb + (te - tb) * q / 1024; t < te; t += chunk) {
      mpadam::PoolChunk pc;
      pc.start = t;
      pc.count = (int32_t)std::min<int64_t>(chunk, te - t);
      pc.first = tensor_of(t);
      pool.push_back(pc);
    }
  }
}

// The group's tail pool for `grid` CTAs, uploaded (none when q is 1024).
int32_t upload_pool(Group& g, int32_t grid, int32_t q, int32_t chunk) {
  g.pool_chunks = 0;
  std::vector<mpadam::PoolChunk> pool;
  pool_host(g.numel.data(), g.count, g.tiles, grid, q, chunk, pool);
  if (pool.empty()) return MPADAM_OK;
  if (pool.size() > (size_t)INT32_MAX) return fail(MPADAM_EINVAL, "tail pool too large");
  if ((int32_t)pool.size() > g.pool_cap) {
    if (g.d_pool) cudaFree(g.d_pool);
    g.d_pool = nullptr;
    g.pool_cap = 0;
    if (dev_malloc(&g.d_pool, sizeof(mpadam::PoolChunk) * pool.size()) != cudaSuccess)
      return fail(MPADAM_EALLOC, "cudaMalloc of %zu tail-pool chunks failed", pool.size());
    g.pool_cap = (int32_t)pool.size();
  }
  cudaError_t e = cudaMemcpy(g.d_pool, pool.data(), sizeof(mpadam::PoolChunk) * pool.size(), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(e, "upload of the tail pool");
  g.pool_chunks = (int32_t)pool.size();
  return MPADAM_OK;
}

// The static share a group's launches use: every format (per-tensor E4M3
// too, whose consumers seed the exact-maximum threshold from the amax ring
// after each tensor change), but by default only groups with at least
// kPoolMinTilesPerCta tiles per CTA.  A producer claims chunks while its ring
// has free stages, so with a tile or two per CTA the first CTAs to reach the
// pool take several chunks each and the launch waits on them (measured on a
// 1 Mi-element list: 16.2 us pooled, 14.5 us static).
constexpr int64_t kPoolMinTilesPerCta = 8;
int32_t pool_q_of(const mpadam_state* s, const Group& g) {
  if (!s->pool_set && g.tiles < kPoolMinTilesPerCta * g.grid) return 1024;
  return s->pool_q;
}

void fill_common(StepArgs& a, const mpadam_config& cfg, const Geometry& geo, int64_t total_tiles, int32_t n,
                 int32_t* fp8_exp, uint32_t* fp8_amax) {
  std::memset(&a, 0, sizeof a);
  a.total_tiles = total_tiles;
  a.n_tensors = n;
  a.stages = geo.stages;
  a.stage_bytes = geo.stage_bytes;
  a.off_g = geo.off_g;
  a.off_m = geo.off_m;
  a.off_v = geo.off_v;
  a.off_ve = geo.off_ve;
  a.off_s = geo.off_s;
  round_keys(cfg.seed, a.rk0, a.rk1);
  a.fp8_exp = fp8_exp;
  a.fp8_amax = fp8_amax;
  a.static_q = 1024;  // static ranges only unless a launch brings a tail pool
}

void fill_step(StepArgs& a, const mpadam_config& cfg, int64_t step) {
  make_scalars(cfg, step, &a.s);
  a.t_lo = (uint32_t)(uint64_t)step;
  a.t_hi = (uint32_t)((uint64_t)step >> 32);
  a.e_cur_slot = (int32_t)(step % 2);
  a.e_next_slot = (int32_t)((step + 1) % 2);
  a.a_cur_slot = (int32_t)(step % 3);
  a.a_next_slot = (int32_t)((step + 1) % 3);
  a.a_zero_slot = (int32_t)((step + 2) % 3);
}

StepArgs base_args(const mpadam_state* s, const Group& g) {
  StepArgs a;
  fill_common(a, s->cfg, g.geo, g.tiles, s->n, s->fp8_exp, s->fp8_amax);
  a.desc = s->d_desc + g.first;
  a.aux = g.aux ? s->d_aux + g.first : nullptr;
  a.grads = s->d_grads + g.first;
  a.cta_first = g.d_cta_first;
  a.err = s->d_err;
  return a;
}

const void* select_kernel(const mpadam_config& c, int32_t wd) {
  const int opt = kernel_options(c) ? 1 : 0;
  if (wd == MPADAM_BF16) return mpadam::step_kernel_bf16(c.grad_dtype, c.moment_dtype, c.rounding, opt);
  if (wd == MPADAM_E4M3) return mpadam::step_kernel_e4m3(c.grad_dtype, c.moment_dtype, c.rounding, opt);
  if (wd == MPADAM_E4M3_B32) return mpadam::step_kernel_e4m3b(c.grad_dtype, c.moment_dtype, c.rounding, opt);
  if (wd == MPADAM_NVFP4) return mpadam::step_kernel_nvfp4(c.grad_dtype, c.moment_dtype, c.rounding, opt);
  return nullptr;
}

// Opt the kernel into the ring's shared memory and size one full wave.
int32_t prepare_kernel(const void* kernel, const Geometry& geo, int sms, int32_t* grid) {
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, geo.dyn_smem);
  if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(MaxDynamicSharedMemorySize)");
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, mpadam::kThreads, geo.dyn_smem);
  if (e != cudaSuccess) return cuda_fail(e, "occupancy query");
  if (per_sm < 1) return fail(MPADAM_ECUDA, "step kernel cannot be resident");
  *grid = per_sm * sms;
  return MPADAM_OK;
}

int32_t check_device(const mpadam_state* s) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev != s->device)
    return fail(MPADAM_EINVAL, "current device %d differs from the state's device %d", dev, s->device);
  return MPADAM_OK;
}

// One tensor of either creation call, with its format resolved.
struct TensorIn {
  void *w, *m, *v, *ve;
  int64_t numel;
  int32_t wd;
  void* scale;
  uint16_t* compute;
  float gscale;
};

// Validate a tensor list, lay out its global index and format groups, and
// allocate and upload the device tables.  `fallback_wd` is the format of the
// single (empty) group of an empty list.
int32_t create_state(const std::vector<TensorIn>& t, const mpadam_config* cfg, int32_t fallback_wd,
                     int32_t* fp8_exp, uint32_t* fp8_amax, mpadam_state** out) {
  const int32_t n = (int32_t)t.size();
  const size_t msz = elem_size(cfg->moment_dtype);
  bool any_e4m3 = false;
  int64_t off = 0;
  for (int32_t k = 0; k < n; ++k) {
    const TensorIn& x = t[k];
    if (x.wd != MPADAM_BF16 && x.wd != MPADAM_E4M3 && x.wd != MPADAM_E4M3_B32 && x.wd != MPADAM_NVFP4)
      return fail(MPADAM_EINVAL, "tensor %d: weight_dtype must be BF16, E4M3, E4M3_B32 or NVFP4 (got %d)", k, x.wd);
    if (x.wd == MPADAM_NVFP4 && !(std::isfinite(x.gscale) && x.gscale > 0.0f))
      return fail(MPADAM_EINVAL, "tensor %d: NVFP4 weights need a finite global_scale > 0", k);
    if (x.wd != MPADAM_NVFP4 && x.gscale != 0.0f)
      return fail(MPADAM_EINVAL, "tensor %d: global_scale is only for NVFP4 weights (must be 0)", k);
    if (x.numel < 0) return fail(MPADAM_EINVAL, "tensor %d: numel < 0", k);
    any_e4m3 = any_e4m3 || x.wd == MPADAM_E4M3;
    if (x.numel > 0) {
      if (!x.w || !x.m || !x.v || !x.ve) return fail(MPADAM_EINVAL, "tensor %d: NULL pointer", k);
      if (!is_aligned(x.w, elem_size(x.wd)) || !is_aligned(x.m, msz) || !is_aligned(x.v, msz) ||
          !is_aligned(x.ve, msz))
        return fail(MPADAM_EINVAL, "tensor %d: pointer not aligned to its element size", k);
      if (x.wd == MPADAM_E4M3_B32 && (!x.scale || !is_aligned(x.scale, 2)))
        return fail(MPADAM_EINVAL, "tensor %d: block-scaled weights need a 2-byte aligned block_scale array", k);
      if (x.wd == MPADAM_NVFP4 && !x.scale)
        return fail(MPADAM_EINVAL, "tensor %d: NVFP4 weights need their block_scale array", k);
      if (x.compute && !is_aligned(x.compute, 2))
        return fail(MPADAM_EINVAL, "tensor %d: compute copy not 2-byte aligned", k);
    }
    if (x.wd != MPADAM_E4M3_B32 && x.wd != MPADAM_NVFP4 && x.scale)
      return fail(MPADAM_EINVAL, "tensor %d: block_scale is only for E4M3_B32 and NVFP4 weights", k);
    if (x.wd == MPADAM_BF16 && x.compute)
      return fail(MPADAM_EINVAL, "tensor %d: BF16 weights are their own compute copy (compute must be NULL)", k);
    if (x.numel > (int64_t(1) << 56) || off > (int64_t(1) << 58))
      return fail(MPADAM_EINVAL, "tensor %d: element index space too large", k);
    off = (off + x.numel + 7) / 8 * 8;
  }
  if (any_e4m3) {
    if (!fp8_exp || !fp8_amax) return fail(MPADAM_EINVAL, "E4M3 weights need the fp8_exp and fp8_amax rings");
    if (!is_aligned(fp8_exp, 4) || !is_aligned(fp8_amax, 4))
      return fail(MPADAM_EINVAL, "fp8_exp / fp8_amax must be 4-byte aligned");
  }

  mpadam_state* s = new (std::nothrow) mpadam_state();
  if (!s) return fail(MPADAM_EALLOC, "host allocation failed");
  try {
    s->n = n;
    s->cfg = *cfg;
    s->wdt.resize(n);
    s->numel.resize(n);
    s->goff.resize(n);
    s->tile_off.resize(n);
    s->w.resize(n);
    s->last_grads.assign(n, nullptr);
    int64_t o = 0;
    for (int32_t k = 0; k < n; ++k) {
      s->wdt[k] = t[k].wd;
      s->numel[k] = t[k].numel;
      s->goff[k] = o;
      s->w[k] = t[k].w;
      o = (o + t[k].numel + 7) / 8 * 8;
    }
    s->length = o;
    s->fp8_exp = fp8_exp;
    s->fp8_amax = fp8_amax;

    // format groups, in the fixed order BF16, E4M3, E4M3_B32, NVFP4
    std::vector<TensorDesc> desc;
    std::vector<TensorAux> aux;
    bool any_aux = false;
    for (int32_t wd : {MPADAM_BF16, MPADAM_E4M3, MPADAM_E4M3_B32, MPADAM_NVFP4}) {
      Group g;
      g.wd = wd;
      g.first = (int32_t)s->order.size();
      for (int32_t k = 0; k < n; ++k) {
        if (t[k].wd != wd) continue;
        s->tile_off[k] = g.tiles;
        desc.push_back(TensorDesc{t[k].w, t[k].m, t[k].v, t[k].ve, t[k].numel, s->goff[k], g.tiles, k, 0});
        aux.push_back(TensorAux{t[k].scale, t[k].compute, t[k].gscale, 0});
        g.h_desc.push_back(desc.back());
        g.h_aux.push_back(aux.back());
        g.aux = g.aux || t[k].scale != nullptr || t[k].compute != nullptr;
        g.numel.push_back(t[k].numel);
        g.tiles += tiles_of(t[k].numel);
        s->order.push_back(k);
      }
      g.count = (int32_t)s->order.size() - g.first;
      any_aux = any_aux || g.aux;
      if (g.count > 0 || (n == 0 && wd == fallback_wd)) s->groups.push_back(std::move(g));
    }

    cudaError_t e = cudaGetDevice(&s->device);
    if (e != cudaSuccess) { release(s); return cuda_fail(e, "cudaGetDevice"); }
    e = cudaDeviceGetAttribute(&s->sm_count, cudaDevAttrMultiProcessorCount, s->device);
    if (e != cudaSuccess) { release(s); return cuda_fail(e, "cudaDeviceGetAttribute"); }
    int32_t rc;
    for (auto& g : s->groups) {
      g.kernel = select_kernel(*cfg, g.wd);
      if (!g.kernel) { release(s); return fail(MPADAM_EUNSUPPORTED, "no kernel for these formats"); }
      rc = make_geometry(*cfg, g.wd, s->device, &g.geo);
      if (rc) { release(s); return rc; }
      rc = prepare_kernel(g.kernel, g.geo, s->sm_count, &g.default_grid);
      if (rc) { release(s); return rc; }
    }

    const size_t nn = n > 0 ? (size_t)n : 1;
    if (dev_malloc(&s->d_desc, sizeof(TensorDesc) * nn) != cudaSuccess ||
        dev_malloc(reinterpret_cast<void**>(&s->d_grads), sizeof(void*) * nn) != cudaSuccess ||
        (any_aux && dev_malloc(&s->d_aux, sizeof(TensorAux) * nn) != cudaSuccess) ||
        dev_malloc(&s->d_err, sizeof(int32_t)) != cudaSuccess ||
        dev_malloc(&s->d_pool_next, sizeof(uint32_t) * std::max<size_t>(1, s->groups.size())) != cudaSuccess ||
        host_malloc(reinterpret_cast<void**>(&s->h_grads), sizeof(void*) * nn) != cudaSuccess) {
      release(s);
      return fail(MPADAM_EALLOC, "allocation of the tensor tables failed");
    }
    e = cudaMemset(s->d_err, 0, sizeof(int32_t));
    if (e != cudaSuccess) { release(s); return cuda_fail(e, "clearing the error word"); }
    e = cudaEventCreateWithFlags(&s->upload_done, cudaEventDisableTiming);
    if (e != cudaSuccess) { release(s); return cuda_fail(e, "cudaEventCreate"); }
    if (n > 0) {
      e = cudaMemcpy(s->d_desc, desc.data(), sizeof(TensorDesc) * n, cudaMemcpyHostToDevice);
      if (e != cudaSuccess) { release(s); return cuda_fail(e, "upload of the tensor table"); }
      if (any_aux) {
        e = cudaMemcpy(s->d_aux, aux.data(), sizeof(TensorAux) * n, cudaMemcpyHostToDevice);
        if (e != cudaSuccess) { release(s); return cuda_fail(e, "upload of the aux table"); }
      }
    }
    for (auto& g : s->groups) {
      rc = upload_cta_table(g, g.default_grid);
      if (!rc) rc = upload_pool(g, g.grid, pool_q_of(s, g), s->pool_chunk);
      if (rc) { release(s); return rc; }
    }
  } catch (const std::bad_alloc&) {
    release(s);
    return fail(MPADAM_EALLOC, "host allocation failed");
  }
  *out = s;
  return MPADAM_OK;
}

// Re-upload the gradient pointer table (in group order) when it differs from
// the last one.
int32_t upload_grad_table(mpadam_state* s, const void* const* grads, cudaStream_t stream) {
  cudaError_t e;
  if (s->grads_uploaded && std::memcmp(s->last_grads.data(), grads, sizeof(void*) * s->n) == 0) return MPADAM_OK;
  if (s->upload_pending) {  // the pinned table may still be read by the last copy
    e = cudaEventSynchronize(s->upload_done);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventSynchronize");
  }
  for (int32_t p = 0; p < s->n; ++p) s->h_grads[p] = grads[s->order[p]];
  e = cudaMemcpyAsync(s->d_grads, s->h_grads, sizeof(void*) * s->n, cudaMemcpyHostToDevice, stream);
  if (e != cudaSuccess) return cuda_fail(e, "upload of the gradient table");
  e = cudaEventRecord(s->upload_done, stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
  s->upload_pending = true;
  std::memcpy(s->last_grads.data(), grads, sizeof(void*) * s->n);
  s->grads_uploaded = true;
  return MPADAM_OK;
}

// One launch of a group's step kernel over its tiles [tile_base, tile_base + count).
int32_t launch_step(mpadam_state* s, const Group& g, int64_t step, cudaStream_t stream, int64_t tile_base,
                    int64_t count, const int32_t* cta_first, int32_t grid, uint32_t* pool_next = nullptr) {
  StepArgs a = base_args(s, g);
  a.cta_first = cta_first;
  a.tile_base = tile_base;
  a.total_tiles = count;
  if (pool_next && g.pool_chunks > 0) {  // whole-group launches only: the pool covers all of its tiles
    a.pool = g.d_pool;
    a.pool_next = pool_next;
    a.pool_chunks = g.pool_chunks;
    a.static_q = pool_q_of(s, g);
  }
  if (tile_base == 0 && count == g.tiles && g.count <= mpadam::kInlineTensors) {
    // a short whole-group launch carries its tables (the gradient pointers as
    // staged for this step's upload, in group order)
    a.n_inline = g.count;
    for (int32_t i = 0; i < g.count; ++i) {
      a.inl_desc[i] = g.h_desc[i];
      a.inl_aux[i] = g.h_aux[i];
      a.inl_grads[i] = s->h_grads[g.first + i];
    }
  }
  fill_step(a, s->cfg, step);
  void* params[] = {&a};
  cudaError_t e = cudaLaunchKernel(g.kernel, dim3(grid), dim3(mpadam::kThreads), params, (size_t)g.geo.dyn_smem,
                                   stream);
  if (e != cudaSuccess) return cuda_fail(e, "launch of the step kernel");
  return MPADAM_OK;
}

// Global element index of a tile's first element, and one past its last
// (single-group states: tile numbering follows the list).
void tile_elements(const mpadam_state* s, int64_t t, int64_t* first, int64_t* end) {
  const auto it = std::upper_bound(s->tile_off.begin(), s->tile_off.end(), t);
  int32_t k = (int32_t)(it - s->tile_off.begin()) - 1;
  while (tiles_of(s->numel[k]) == 0 || t >= s->tile_off[k] + tiles_of(s->numel[k])) ++k;
  const int64_t j = t - s->tile_off[k];
  *first = s->goff[k] + j * mpadam::kTile;
  *end = s->goff[k] + std::min<int64_t>((j + 1) * mpadam::kTile, s->numel[k]);
}

// The host-buffer pipeline: chunks of whole tiles, their CTA tables, two
// copy streams and the events that order them (created on first use).
int32_t prepare_pipeline(mpadam_state* s) {
  if (!s->chunk_tile.empty()) return MPADAM_OK;
  release_pipeline(s);  // whatever a failed earlier attempt left
  const Group& g = s->groups[0];
  const int32_t chunks = (int32_t)std::max<int64_t>(1, std::min<int64_t>(8, g.tiles / 256));  // 8: best measured
  std::vector<int64_t> ct(chunks + 1), ce(2 * (size_t)chunks);
  for (int32_t c = 0; c <= chunks; ++c) ct[c] = (int64_t)c * g.tiles / chunks;
  for (int32_t c = 0; c < chunks; ++c) {
    int64_t f0, e0, f1, e1;
    tile_elements(s, ct[c], &f0, &e0);
    tile_elements(s, ct[c + 1] - 1, &f1, &e1);
    ce[2 * c] = f0;
    ce[2 * c + 1] = e1;
  }
  std::vector<int32_t> first((size_t)chunks * g.grid);
  for (int32_t c = 0; c < chunks; ++c)
    cta_first_table(s->numel.data(), s->n, ct[c + 1] - ct[c], g.grid, first.data() + (size_t)c * g.grid, ct[c]);
  if (dev_malloc(&s->d_chunk_first, sizeof(int32_t) * first.size()) != cudaSuccess)
    return fail(MPADAM_EALLOC, "cudaMalloc of the chunk tables failed");
  cudaError_t e = cudaMemcpy(s->d_chunk_first, first.data(), sizeof(int32_t) * first.size(), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(e, "upload of the chunk tables");
  e = cudaStreamCreateWithFlags(&s->s_h2d, cudaStreamNonBlocking);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamCreate");
  e = cudaStreamCreateWithFlags(&s->s_d2h, cudaStreamNonBlocking);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamCreate");
  s->ev.resize(2 * (size_t)chunks + 2);
  for (auto& ev : s->ev) {
    e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventCreate");
  }
  s->chunk_tile = ct;
  s->chunk_elem = ce;
  return MPADAM_OK;
}

}  // namespace

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------
extern "C" {

const char* mpadam_last_error(void) { return g_last_error.c_str(); }

int32_t mpadam_create(const mpadam_tensor* tensors, int32_t n, const mpadam_config* cfg,
                      int32_t* fp8_exp, uint32_t* fp8_amax, mpadam_state** out) {
  if (!out) return fail(MPADAM_EINVAL, "out is NULL");
  *out = nullptr;
  if (n < 0) return fail(MPADAM_EINVAL, "n must be >= 0 (got %d)", n);
  if (n > 0 && !tensors) return fail(MPADAM_EINVAL, "tensors is NULL");
  int32_t rc = check_config(cfg);
  if (rc) return rc;
  if (cfg->weight_dtype == MPADAM_E4M3 && (!fp8_exp || !fp8_amax))
    return fail(MPADAM_EINVAL, "E4M3 weights need the fp8_exp and fp8_amax rings");
  try {
    std::vector<TensorIn> t(n);
    for (int32_t k = 0; k < n; ++k)
      t[k] = TensorIn{tensors[k].w, tensors[k].m, tensors[k].v, tensors[k].ve, tensors[k].numel, cfg->weight_dtype,
                      nullptr, nullptr, 0.0f};
    return create_state(t, cfg, cfg->weight_dtype, fp8_exp, fp8_amax, out);
  } catch (const std::bad_alloc&) {
    return fail(MPADAM_EALLOC, "host allocation failed");
  }
}

int32_t mpadam_create_ex(const mpadam_tensor_ex* tensors, int32_t n, const mpadam_config* cfg,
                         int32_t* fp8_exp, uint32_t* fp8_amax, mpadam_state** out) {
  if (!out) return fail(MPADAM_EINVAL, "out is NULL");
  *out = nullptr;
  if (n < 0) return fail(MPADAM_EINVAL, "n must be >= 0 (got %d)", n);
  if (n > 0 && !tensors) return fail(MPADAM_EINVAL, "tensors is NULL");
  int32_t rc = check_config(cfg, true);
  if (rc) return rc;
  try {
    std::vector<TensorIn> t(n);
    for (int32_t k = 0; k < n; ++k) {
      const mpadam_tensor_ex& x = tensors[k];
      t[k] = TensorIn{x.w, x.m, x.v, x.ve, x.numel, x.weight_dtype, x.block_scale, x.compute, x.global_scale};
    }
    return create_state(t, cfg, MPADAM_BF16, fp8_exp, fp8_amax, out);
  } catch (const std::bad_alloc&) {
    return fail(MPADAM_EALLOC, "host allocation failed");
  }
}

int32_t mpadam_destroy(mpadam_state* s) {
  if (!s) return MPADAM_OK;
  release(s);
  return MPADAM_OK;
}

int32_t mpadam_global_offset(const mpadam_state* s, int32_t k, int64_t* offset) {
  if (!s || !offset) return fail(MPADAM_EINVAL, "NULL argument");
  if (k < 0 || k >= s->n) return fail(MPADAM_EINVAL, "tensor index %d out of range [0, %d)", k, s->n);
  *offset = s->goff[k];
  return MPADAM_OK;
}

int32_t mpadam_global_length(const mpadam_state* s, int64_t* length) {
  if (!s || !length) return fail(MPADAM_EINVAL, "NULL argument");
  *length = s->length;
  return MPADAM_OK;
}

int32_t mpadam_set_grid(mpadam_state* s, int32_t ctas) {
  if (!s) return fail(MPADAM_EINVAL, "state is NULL");
  if (ctas < 0 || ctas > (1 << 20)) return fail(MPADAM_EINVAL, "ctas must be in [0, 2^20]");
  int32_t rc = check_device(s);
  if (rc) return rc;
  cudaError_t e = cudaDeviceSynchronize();  // the old table may be in use
  if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
  release_pipeline(s);  // the host-buffer pipeline's per-chunk tables follow the grid: rebuilt on next use
  for (auto& g : s->groups) {
    rc = upload_cta_table(g, ctas == 0 ? g.default_grid : ctas);
    if (!rc) rc = upload_pool(g, g.grid, pool_q_of(s, g), s->pool_chunk);
    if (rc) return rc;
  }
  return MPADAM_OK;
}

int32_t mpadam_set_tail_pool(mpadam_state* s, int32_t static_q, int32_t chunk_tiles) {
  if (!s) return fail(MPADAM_EINVAL, "state is NULL");
  if (static_q < 0 || static_q > 1024) return fail(MPADAM_EINVAL, "static_q must be in [0, 1024]");
  if (chunk_tiles < 1 || chunk_tiles > (1 << 20)) return fail(MPADAM_EINVAL, "chunk_tiles must be in [1, 2^20]");
  int32_t rc = check_device(s);
  if (rc) return rc;
  cudaError_t e = cudaDeviceSynchronize();  // the old pool may be in use
  if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
  s->pool_q = static_q;
  s->pool_chunk = chunk_tiles;
  s->pool_set = true;
  for (auto& g : s->groups) {
    rc = upload_pool(g, g.grid, pool_q_of(s, g), s->pool_chunk);
    if (rc) return rc;
  }
  return MPADAM_OK;
}

int32_t mpadam_launch_info(const mpadam_state* s, int32_t* ctas, int32_t* threads) {
  if (!s || !ctas || !threads) return fail(MPADAM_EINVAL, "NULL argument");
  *ctas = s->groups.empty() ? 0 : s->groups[0].grid;
  *threads = mpadam::kThreads;
  return MPADAM_OK;
}

int32_t mpadam_device_status(mpadam_state* s, int32_t* code) {
  if (!s || !code) return fail(MPADAM_EINVAL, "NULL argument");
  int32_t rc = check_device(s);
  if (rc) return rc;
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
  e = cudaMemcpy(code, s->d_err, sizeof(int32_t), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "reading the error word");
  e = cudaMemset(s->d_err, 0, sizeof(int32_t));
  if (e != cudaSuccess) return cuda_fail(e, "clearing the error word");
  return MPADAM_OK;
}

int32_t mpadam_step(mpadam_state* s, const void* const* grads, int64_t step, cudaStream_t stream) {
  if (!s) return fail(MPADAM_EINVAL, "state is NULL");
  if (step < 1) return fail(MPADAM_EINVAL, "step must be >= 1 (got %lld)", (long long)step);
  int64_t tiles = 0;
  for (const auto& g : s->groups) tiles += g.tiles;
  if (s->n == 0 || tiles == 0) return MPADAM_OK;
  if (!grads) return fail(MPADAM_EINVAL, "grads is NULL");
  const size_t gsz = elem_size(s->cfg.grad_dtype);
  for (int32_t k = 0; k < s->n; ++k) {
    if (s->numel[k] == 0) continue;
    if (!grads[k]) return fail(MPADAM_EINVAL, "grads[%d] is NULL", k);
    if (!is_aligned(grads[k], gsz)) return fail(MPADAM_EINVAL, "grads[%d] not aligned to its element size", k);
  }
  int32_t rc = check_device(s);
  if (rc) return rc;
  rc = upload_grad_table(s, grads, stream);
  if (rc) return rc;
  bool pooled = false;
  for (const auto& g : s->groups) pooled = pooled || g.pool_chunks > 0;
  if (pooled) {  // the pools' claim counters start at zero
    cudaError_t e = cudaMemsetAsync(s->d_pool_next, 0, sizeof(uint32_t) * s->groups.size(), stream);
    if (e != cudaSuccess) return cuda_fail(e, "clearing the tail-pool counters");
  }
  for (size_t i = 0; i < s->groups.size(); ++i) {
    const Group& g = s->groups[i];
    if (g.tiles == 0) continue;
    rc = launch_step(s, g, step, stream, 0, g.tiles, g.d_cta_first, g.grid, s->d_pool_next + i);
    if (rc) return rc;
  }
  return MPADAM_OK;
}

int32_t mpadam_fp8_init(mpadam_state* s, const int32_t* init_exp, int64_t first_step, cudaStream_t stream) {
  if (!s) return fail(MPADAM_EINVAL, "state is NULL");
  const Group* g = nullptr;
  for (const auto& x : s->groups)
    if (x.wd == MPADAM_E4M3) g = &x;
  if (!g) return fail(MPADAM_EINVAL, "fp8_init needs E4M3 weights");
  if (first_step < 1) return fail(MPADAM_EINVAL, "first_step must be >= 1");
  if (s->n == 0) return MPADAM_OK;
  if (!init_exp) return fail(MPADAM_EINVAL, "init_exp is NULL");
  for (int32_t k = 0; k < s->n; ++k)
    if (s->wdt[k] == MPADAM_E4M3 && (init_exp[k] < -100 || init_exp[k] > 100))
      return fail(MPADAM_EINVAL, "init_exp[%d] = %d outside [-100, 100]", k, init_exp[k]);
  int32_t rc = check_device(s);
  if (rc) return rc;
  std::vector<int32_t> both(2 * (size_t)s->n, 0);
  for (int32_t k = 0; k < s->n; ++k)
    if (s->wdt[k] == MPADAM_E4M3) both[k] = both[s->n + k] = init_exp[k];
  cudaError_t e = cudaMemcpyAsync(s->fp8_exp, both.data(), sizeof(int32_t) * both.size(),
                                  cudaMemcpyHostToDevice, stream);
  if (e != cudaSuccess) return cuda_fail(e, "upload of the initial exponents");
  e = cudaStreamSynchronize(stream);  // `both` is pageable and about to go away
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  e = cudaMemsetAsync(s->fp8_amax, 0, sizeof(uint32_t) * 3 * (size_t)s->n, stream);
  if (e != cudaSuccess) return cuda_fail(e, "clearing fp8_amax");
  if (g->tiles == 0) return MPADAM_OK;
  StepArgs a = base_args(s, *g);
  int32_t exp_slot = (int32_t)(first_step % 2), amax_slot = (int32_t)(first_step % 3);
  void* params[] = {&a, &exp_slot, &amax_slot};
  e = cudaLaunchKernel(reinterpret_cast<const void*>(&fp8_amax_kernel), dim3(g->grid), dim3(mpadam::kConsumers),
                       params, 0, stream);
  if (e != cudaSuccess) return cuda_fail(e, "launch of the amax kernel");
  return MPADAM_OK;
}

int32_t mpadam_rng_lanes(uint64_t seed, int64_t step, int32_t weight_dtype, int64_t first, int64_t n,
                         uint32_t* out, cudaStream_t stream) {
  if (step < 0) return fail(MPADAM_EINVAL, "step must be >= 0");
  if (weight_dtype != MPADAM_BF16 && weight_dtype != MPADAM_E4M3 && weight_dtype != MPADAM_E4M3_B32 &&
      weight_dtype != MPADAM_NVFP4)
    return fail(MPADAM_EINVAL, "weight_dtype must be MPADAM_BF16, MPADAM_E4M3, MPADAM_E4M3_B32 or MPADAM_NVFP4");
  if (first < 0 || n < 0) return fail(MPADAM_EINVAL, "first and n must be >= 0");
  if (n == 0) return MPADAM_OK;
  if (!out || !is_aligned(out, 4)) return fail(MPADAM_EINVAL, "out is NULL or misaligned");
  RngArgs a;
  round_keys(seed, a.rk0, a.rk1);
  a.t_lo = (uint32_t)(uint64_t)step;
  a.t_hi = (uint32_t)((uint64_t)step >> 32);
  a.bf16 = weight_dtype == MPADAM_BF16 ? 1 : 0;
  a.first = (uint64_t)first;
  a.n = n;
  a.out = out;
  const int64_t blocks = std::min<int64_t>((n + 255) / 256, 4096);
  rng_lanes_kernel<<<(unsigned)blocks, 256, 0, stream>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "launch of the rng kernel");
  return MPADAM_OK;
}

int32_t mpadam_step_host(mpadam_state* s, const void* const* host_grads, void* const* host_w_out,
                         int64_t step, cudaStream_t stream) {
  if (!s) return fail(MPADAM_EINVAL, "state is NULL");
  if (step < 1) return fail(MPADAM_EINVAL, "step must be >= 1");
  int64_t tiles = 0;
  for (const auto& g : s->groups) tiles += g.tiles;
  if (s->n == 0 || tiles == 0) return MPADAM_OK;
  if (!host_grads || !host_w_out) return fail(MPADAM_EINVAL, "host_grads / host_w_out is NULL");
  for (int32_t k = 0; k < s->n; ++k)
    if (s->numel[k] > 0 && (!host_grads[k] || !host_w_out[k]))
      return fail(MPADAM_EINVAL, "host buffer %d is NULL", k);
  int32_t rc = check_device(s);
  if (rc) return rc;
  const size_t gsz = elem_size(s->cfg.grad_dtype);
  cudaError_t e;
  if (!s->d_gstage) {
    if (dev_malloc(&s->d_gstage, (size_t)s->length * gsz) != cudaSuccess)
      return fail(MPADAM_EALLOC, "cudaMalloc of %lld bytes of gradient staging failed",
                  (long long)((size_t)s->length * gsz));
    s->stage_ptrs.resize(s->n);
    for (int32_t k = 0; k < s->n; ++k) s->stage_ptrs[k] = s->d_gstage + (size_t)s->goff[k] * gsz;
  }
  // Does a set of per-tensor pointers follow one flat buffer in global-index layout?
  auto flat_base = [&](const void* const* p, size_t esz, const char** base) {
    const char* b = nullptr;
    for (int32_t k = 0; k < s->n; ++k) {
      if (s->numel[k] == 0) continue;
      const char* c = static_cast<const char*>(p[k]) - (size_t)s->goff[k] * esz;
      if (!b) b = c;
      else if (c != b) return false;
    }
    *base = b;
    return b != nullptr;
  };
  int32_t first = 0, last = s->n - 1;
  while (first < s->n && s->numel[first] == 0) ++first;
  while (last >= 0 && s->numel[last] == 0) --last;
  if (first > last) return MPADAM_OK;
  const size_t lo_e = (size_t)s->goff[first], hi_e = (size_t)(s->goff[last] + s->numel[last]);
  // one weight format for the whole list?  (then wsz is its element size)
  const bool single = s->groups.size() == 1 && s->groups[0].wd != MPADAM_NVFP4;
  const size_t wsz = elem_size(s->groups[0].wd);

  const char* hb = nullptr;
  const char* dw0 = nullptr;
  const char* hw0 = nullptr;
  if (single && flat_base(host_grads, gsz, &hb) && flat_base(s->w.data(), wsz, &dw0) &&
      flat_base(host_w_out, wsz, &hw0)) {
    // Pipelined: chunk c's gradients upload on s_h2d, its step runs on
    // `stream` after them, its weights download on s_d2h after the step.
    const Group& g = s->groups[0];
    rc = prepare_pipeline(s);
    if (rc) return rc;
    rc = upload_grad_table(s, s->stage_ptrs.data(), stream);
    if (rc) return rc;
    const int32_t chunks = (int32_t)s->chunk_tile.size() - 1;
    cudaEvent_t ev_start = s->ev[2 * chunks], ev_end = s->ev[2 * chunks + 1];
    // the copies must not overtake earlier work on `stream` (a previous step
    // still reading the staging buffer or writing the weights)
    if ((e = cudaEventRecord(ev_start, stream)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
    if ((e = cudaStreamWaitEvent(s->s_h2d, ev_start, 0)) != cudaSuccess) return cuda_fail(e, "cudaStreamWaitEvent");
    if ((e = cudaStreamWaitEvent(s->s_d2h, ev_start, 0)) != cudaSuccess) return cuda_fail(e, "cudaStreamWaitEvent");
    for (int32_t c = 0; c < chunks; ++c) {
      const size_t a0 = (size_t)s->chunk_elem[2 * c], a1 = (size_t)s->chunk_elem[2 * c + 1];
      e = cudaMemcpyAsync(s->d_gstage + a0 * gsz, hb + a0 * gsz, (a1 - a0) * gsz, cudaMemcpyHostToDevice, s->s_h2d);
      if (e != cudaSuccess) return cuda_fail(e, "gradient upload");
      if ((e = cudaEventRecord(s->ev[2 * c], s->s_h2d)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
      if ((e = cudaStreamWaitEvent(stream, s->ev[2 * c], 0)) != cudaSuccess) return cuda_fail(e, "cudaStreamWaitEvent");
      rc = launch_step(s, g, step, stream, s->chunk_tile[c], s->chunk_tile[c + 1] - s->chunk_tile[c],
                       s->d_chunk_first + (size_t)c * g.grid, g.grid);
      if (rc) return rc;
      if ((e = cudaEventRecord(s->ev[2 * c + 1], stream)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
      if ((e = cudaStreamWaitEvent(s->s_d2h, s->ev[2 * c + 1], 0)) != cudaSuccess)
        return cuda_fail(e, "cudaStreamWaitEvent");
      e = cudaMemcpyAsync(const_cast<char*>(hw0) + a0 * wsz, dw0 + a0 * wsz, (a1 - a0) * wsz, cudaMemcpyDeviceToHost,
                          s->s_d2h);
      if (e != cudaSuccess) return cuda_fail(e, "weight download");
    }
    // `stream` completes only after every download
    if ((e = cudaEventRecord(ev_end, s->s_d2h)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
    if ((e = cudaStreamWaitEvent(stream, ev_end, 0)) != cudaSuccess) return cuda_fail(e, "cudaStreamWaitEvent");
    return MPADAM_OK;
  }
  if (flat_base(host_grads, gsz, &hb)) {
    e = cudaMemcpyAsync(s->d_gstage + lo_e * gsz, hb + lo_e * gsz, (hi_e - lo_e) * gsz,
                        cudaMemcpyHostToDevice, stream);
    if (e != cudaSuccess) return cuda_fail(e, "gradient upload");
  } else {
    for (int32_t k = 0; k < s->n; ++k) {
      if (s->numel[k] == 0) continue;
      e = cudaMemcpyAsync(const_cast<void*>(s->stage_ptrs[k]), host_grads[k], (size_t)s->numel[k] * gsz,
                          cudaMemcpyHostToDevice, stream);
      if (e != cudaSuccess) return cuda_fail(e, "gradient upload");
    }
  }
  rc = mpadam_step(s, s->stage_ptrs.data(), step, stream);
  if (rc) return rc;
  const char* dw = nullptr;
  const char* hw = nullptr;
  if (single && flat_base(const_cast<const void* const*>(reinterpret_cast<void* const*>(s->w.data())), wsz, &dw) &&
      flat_base(const_cast<const void* const*>(host_w_out), wsz, &hw)) {
    e = cudaMemcpyAsync(const_cast<char*>(hw) + lo_e * wsz, dw + lo_e * wsz, (hi_e - lo_e) * wsz,
                        cudaMemcpyDeviceToHost, stream);
    if (e != cudaSuccess) return cuda_fail(e, "weight download");
  } else {
    for (int32_t k = 0; k < s->n; ++k) {
      if (s->numel[k] == 0) continue;
      e = cudaMemcpyAsync(host_w_out[k], s->w[k], weight_bytes(s->wdt[k], s->numel[k]), cudaMemcpyDeviceToHost,
                          stream);
      if (e != cudaSuccess) return cuda_fail(e, "weight download");
    }
  }
  return MPADAM_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free step (mpadam_step_noalloc)
//
// For callers that must not call cudaMalloc -- for example a runtime whose
// device memory all belongs to its own caching allocator or memory pool, or
// a service that fixes its device-memory budget at start-up.  The metadata
// the step kernel reads (tensor descriptors, gradient pointers, per-CTA start
// tensors) goes into one file-scope device array instead of memory the
// library allocates.  Every GPU that loads the library holds the array until
// the process exits.  The tables are written by small kernels that receive
// them as kernel parameters, so no host staging buffer is needed either.
// ---------------------------------------------------------------------------
namespace {

constexpr int32_t kNoAllocMaxTensors = 8192;
constexpr int32_t kNoAllocMaxCtas = 4096;
constexpr size_t kNoAllocTableBytes =
    sizeof(TensorDesc) * kNoAllocMaxTensors + sizeof(void*) * kNoAllocMaxTensors +
    sizeof(int32_t) * kNoAllocMaxCtas;  // 606,208 bytes
// The step kernel's device error word (a bounded wait that gave up) sits in
// its own 256-byte slot after the tables.  It is sticky: every call ORs into
// it, and only mpadam_noalloc_status reads and clears it.  The array starts
// zeroed when the library's module loads.
constexpr size_t kNoAllocErrOffset = kNoAllocTableBytes;
constexpr size_t kNoAllocScratchBytes = kNoAllocTableBytes + 256;  // 606,464 bytes
static_assert(kNoAllocErrOffset % 256 == 0, "the error word keeps the array's alignment");

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int32_t kFillChunk = 384;  // table entries per fill launch (27.7 KB of parameters)

struct FillTensorArgs {
  TensorDesc desc[kFillChunk];
  const void* grads[kFillChunk];
  TensorDesc* dst_desc;
  const void** dst_grads;
  int32_t count;
};

struct FillCtaArgs {
  int32_t first[kNoAllocMaxCtas];
  int32_t* dst;
  int32_t count;
};

__global__ void noalloc_fill_tensors(const __grid_constant__ FillTensorArgs a) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < a.count) {
    a.dst_desc[i] = a.desc[i];
    a.dst_grads[i] = a.grads[i];
  }
}

__global__ void noalloc_fill_ctas(const __grid_constant__ FillCtaArgs a) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < a.count; i += gridDim.x * blockDim.x)
    a.dst[i] = a.first[i];
}

// Per-device set-up: the scratch array's device address and the SM count.
constexpr int kNoAllocMaxDevices = 64;
std::mutex g_noalloc_mutex;
unsigned char* g_noalloc_ptr[kNoAllocMaxDevices] = {};
int g_noalloc_sms[kNoAllocMaxDevices] = {};

int32_t noalloc_setup(int dev, unsigned char** scratch, int* sms) {
  if (dev < 0 || dev >= kNoAllocMaxDevices) return fail(MPADAM_EUNSUPPORTED, "device %d beyond the set-up table", dev);
  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);  // with `dev` current
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress of the scratch array");
    int n_sm = 0;
    e = cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
    g_noalloc_sms[dev] = n_sm;
    g_noalloc_ptr[dev] = static_cast<unsigned char*>(p);
  }
  *scratch = g_noalloc_ptr[dev];
  *sms = g_noalloc_sms[dev];
  return MPADAM_OK;
}

}  // namespace

extern "C" int32_t mpadam_step_noalloc(const mpadam_tensor* tensors, int32_t n, const void* const* grads,
                                       const mpadam_config* cfg, int32_t* fp8_exp, uint32_t* fp8_amax,
                                       int64_t step, cudaStream_t stream) {
  if (n < 0) return fail(MPADAM_EINVAL, "n must be >= 0 (got %d)", n);
  if (n > kNoAllocMaxTensors)
    return fail(MPADAM_EINVAL, "mpadam_step_noalloc takes at most %d tensors (got %d); use mpadam_create",
                kNoAllocMaxTensors, n);
  if (n > 0 && (!tensors || !grads)) return fail(MPADAM_EINVAL, "tensors / grads is NULL");
  if (step < 1) return fail(MPADAM_EINVAL, "step must be >= 1 (got %lld)", (long long)step);
  int32_t rc = check_config(cfg);
  if (rc) return rc;
  const size_t wsz = elem_size(cfg->weight_dtype), msz = elem_size(cfg->moment_dtype),
               gsz = elem_size(cfg->grad_dtype);
  if (cfg->weight_dtype == MPADAM_E4M3 && (!fp8_exp || !fp8_amax || !is_aligned(fp8_exp, 4) || !is_aligned(fp8_amax, 4)))
    return fail(MPADAM_EINVAL, "E4M3 weights need 4-byte aligned fp8_exp and fp8_amax rings");
  int64_t total = 0, total_tiles = 0;
  for (int32_t k = 0; k < n; ++k) {
    const mpadam_tensor& t = tensors[k];
    if (t.numel < 0) return fail(MPADAM_EINVAL, "tensor %d: numel < 0", k);
    if (t.numel > 0) {
      if (!t.w || !t.m || !t.v || !t.ve || !grads[k]) return fail(MPADAM_EINVAL, "tensor %d: NULL pointer", k);
      if (!is_aligned(t.w, wsz) || !is_aligned(t.m, msz) || !is_aligned(t.v, msz) || !is_aligned(t.ve, msz) ||
          !is_aligned(grads[k], gsz))
        return fail(MPADAM_EINVAL, "tensor %d: pointer not aligned to its element size", k);
    }
    if (t.numel > (int64_t(1) << 56) || total > (int64_t(1) << 58))
      return fail(MPADAM_EINVAL, "tensor %d: element index space too large", k);
    total = (total + t.numel + 7) / 8 * 8;
    total_tiles += tiles_of(t.numel);
  }
  if (total_tiles == 0) return MPADAM_OK;

  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  unsigned char* scratch = nullptr;
  int sms = 0;
  rc = noalloc_setup(dev, &scratch, &sms);
  if (rc) return rc;
  const void* kernel = select_kernel(*cfg, cfg->weight_dtype);
  if (!kernel) return fail(MPADAM_EUNSUPPORTED, "no kernel for these formats");
  Geometry geo;
  rc = make_geometry(*cfg, cfg->weight_dtype, dev, &geo);
  if (rc) return rc;
  int32_t grid = 0;
  rc = prepare_kernel(kernel, geo, sms, &grid);
  if (rc) return rc;
  grid = std::min(grid, kNoAllocMaxCtas);

  TensorDesc* d_desc = reinterpret_cast<TensorDesc*>(scratch);
  const void** d_grads = reinterpret_cast<const void**>(scratch + sizeof(TensorDesc) * kNoAllocMaxTensors);
  int32_t* d_first = reinterpret_cast<int32_t*>(scratch + (sizeof(TensorDesc) + sizeof(void*)) * kNoAllocMaxTensors);

  // tensor and gradient tables, in chunks passed as kernel parameters
  FillTensorArgs fa;
  int64_t off = 0, toff = 0;
  for (int32_t k0 = 0; k0 < n; k0 += kFillChunk) {
    const int32_t cnt = std::min(kFillChunk, n - k0);
    for (int32_t i = 0; i < cnt; ++i) {
      const mpadam_tensor& t = tensors[k0 + i];
      fa.desc[i] = TensorDesc{t.w, t.m, t.v, t.ve, t.numel, off, toff, k0 + i, 0};
      fa.grads[i] = grads[k0 + i];
      off = (off + t.numel + 7) / 8 * 8;
      toff += tiles_of(t.numel);
    }
    fa.dst_desc = d_desc + k0;
    fa.dst_grads = d_grads + k0;
    fa.count = cnt;
    noalloc_fill_tensors<<<(cnt + 127) / 128, 128, 0, stream>>>(fa);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "launch of the table fill kernel");
  }
  // tensor holding each CTA's first tile
  FillCtaArgs fc;
  {
    int32_t k = 0;
    int64_t tile_off = 0;
    for (int32_t b = 0; b < grid; ++b) {
      const int64_t tb = (int64_t)b * total_tiles / grid;
      while (k < n && tile_off + tiles_of(tensors[k].numel) <= tb) {
        tile_off += tiles_of(tensors[k].numel);
        ++k;
      }
      fc.first[b] = k;
    }
  }
  fc.dst = d_first;
  fc.count = grid;
  noalloc_fill_ctas<<<(grid + 255) / 256, 256, 0, stream>>>(fc);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "launch of the CTA table fill kernel");

  StepArgs a;
  fill_common(a, *cfg, geo, total_tiles, n, fp8_exp, fp8_amax);
  a.desc = d_desc;
  a.grads = d_grads;
  a.cta_first = d_first;
  a.err = reinterpret_cast<int32_t*>(scratch + kNoAllocErrOffset);
  fill_step(a, *cfg, step);
  void* params[] = {&a};
  e = cudaLaunchKernel(kernel, dim3(grid), dim3(mpadam::kThreads), params, (size_t)geo.dyn_smem, stream);
  if (e != cudaSuccess) return cuda_fail(e, "launch of the step kernel");
  return MPADAM_OK;
}

extern "C" int32_t mpadam_noalloc_status(cudaStream_t stream, int32_t* code) {
  if (!code) return fail(MPADAM_EINVAL, "code is NULL");
  *code = 0;
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  unsigned char* scratch = nullptr;
  int sms = 0;
  int32_t rc = noalloc_setup(dev, &scratch, &sms);
  if (rc) return rc;
  int32_t* err = reinterpret_cast<int32_t*>(scratch + kNoAllocErrOffset);
  // read after the stream's steps, then clear for the calls that follow
  e = cudaMemcpyAsync(code, err, sizeof(int32_t), cudaMemcpyDeviceToHost, stream);
  if (e != cudaSuccess) return cuda_fail(e, "reading the error word");
  e = cudaMemsetAsync(err, 0, sizeof(int32_t), stream);
  if (e != cudaSuccess) return cuda_fail(e, "clearing the error word");
  e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  return MPADAM_OK;
}

// ---------------------------------------------------------------------------
// Matrix-fitting diagnostic (kernels in toy.cu)
// ---------------------------------------------------------------------------
struct mpadam_toy_state {
  mpadam::ToyArgs a{};
  int device = 0;
  int64_t* t_dev = nullptr;           // run mode step counter {t, first t}
  cudaStream_t cap = nullptr;         // capture stream of the run graph
  cudaGraphExec_t exec = nullptr;     // kToyGraphSteps steps for the pointers below
  const void* g_w = nullptr;
  const void* g_ws = nullptr;
  const void* g_loss = nullptr;
};

namespace {
constexpr int64_t kToyGraphSteps = 64;  // steps per replay of the run graph
}

extern "C" int32_t mpadam_toy_create(int64_t n, const mpadam_toy_config* cfg, mpadam_toy_state** out) {
  if (!out) return fail(MPADAM_EINVAL, "out is NULL");
  *out = nullptr;
  if (!cfg) return fail(MPADAM_EINVAL, "config is NULL");
  auto pow2 = [](int64_t x) { return x > 0 && (x & (x - 1)) == 0; };
  if (!pow2(n) || n < 64 || n > (int64_t(1) << 30)) return fail(MPADAM_EINVAL, "n must be a power of two in [64, 2^30]");
  if (cfg->mode < 0 || cfg->mode > 2) return fail(MPADAM_EINVAL, "mode must be 0, 1 or 2");
  if (cfg->split != 0 && cfg->split != 1) return fail(MPADAM_EINVAL, "split must be 0 or 1");
  if (cfg->reserved != 0) return fail(MPADAM_EINVAL, "reserved must be 0");
  const int64_t halves = cfg->split ? 2 : 1;
  if (!pow2(cfg->batch) || cfg->batch / halves < 32 || cfg->batch / halves > 32 * 2048)
    return fail(MPADAM_EINVAL, "batch must be a power of two with 32 to 65536 samples per problem");
  auto fin_nonneg = [](float x) { return std::isfinite(x) && x >= 0.0f; };
  if (!fin_nonneg(cfg->lr_add) || !fin_nonneg(cfg->lr_mul)) return fail(MPADAM_EINVAL, "learning rates must be finite, >= 0");
  if (!fin_nonneg(cfg->rmax) || !(std::isfinite(cfg->tau) && cfg->tau > 0.0f))
    return fail(MPADAM_EINVAL, "rmax must be finite >= 0 and tau finite > 0");
  if (!std::isfinite(cfg->c_lo) || !std::isfinite(cfg->c_hi)) return fail(MPADAM_EINVAL, "c_lo, c_hi must be finite");
  mpadam_toy_state* st = new (std::nothrow) mpadam_toy_state();
  if (!st) return fail(MPADAM_EALLOC, "host allocation failed");
  mpadam::ToyArgs& a = st->a;
  cudaError_t e = cudaGetDevice(&st->device);
  if (e != cudaSuccess) { delete st; return cuda_fail(e, "cudaGetDevice"); }
  const size_t B = (size_t)cfg->batch;
  if (dev_malloc(&a.cnt, sizeof(int32_t) * n) != cudaSuccess || dev_malloc(&a.first, sizeof(int32_t) * n) != cudaSuccess ||
      dev_malloc(&a.idx, sizeof(int32_t) * B) != cudaSuccess || dev_malloc(&a.res, sizeof(float) * B) != cudaSuccess ||
      dev_malloc(&st->t_dev, sizeof(int64_t) * 2) != cudaSuccess ||
      dev_malloc(&a.partial, sizeof(double) * (B / 256 + 2)) != cudaSuccess) {
    mpadam_toy_destroy(st);
    return fail(MPADAM_EALLOC, "allocation of the diagnostic's scratch failed");
  }
  if ((e = cudaMemset(a.cnt, 0, sizeof(int32_t) * n)) != cudaSuccess ||
      (e = cudaMemset(a.first, 0, sizeof(int32_t) * n)) != cudaSuccess ||
      (e = cudaDeviceSynchronize()) != cudaSuccess) {
    mpadam_toy_destroy(st);
    return cuda_fail(e, "clearing the diagnostic's scratch");
  }
  a.n = n;
  a.batch = cfg->batch;
  a.mode = cfg->mode;
  a.split = cfg->split;
  a.lr_add = cfg->lr_add;
  a.lr_mul = cfg->lr_mul;
  a.rmax = cfg->rmax;
  a.tau = cfg->tau;
  a.c_lo = cfg->c_lo;
  a.c_hi = cfg->split ? cfg->c_hi : cfg->c_lo;
  round_keys(cfg->seed, a.rk0, a.rk1);
  *out = st;
  return MPADAM_OK;
}

extern "C" int32_t mpadam_toy_step(mpadam_toy_state* s, uint16_t* w, const float* wstar, int64_t step,
                                   double* loss_out, cudaStream_t stream) {
  if (!s) return fail(MPADAM_EINVAL, "state is NULL");
  if (!w || !wstar || !is_aligned(w, 2) || !is_aligned(wstar, 4)) return fail(MPADAM_EINVAL, "w / wstar NULL or misaligned");
  if (loss_out && !is_aligned(loss_out, 8)) return fail(MPADAM_EINVAL, "loss_out misaligned");
  if (step < 1) return fail(MPADAM_EINVAL, "step must be >= 1");
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev != s->device) return fail(MPADAM_EINVAL, "current device %d differs from the state's device %d", dev, s->device);
  mpadam::ToyArgs a = s->a;
  a.w = w;
  a.wstar = wstar;
  a.loss_out = loss_out;
  a.t_lo = (uint32_t)(uint64_t)step;
  a.t_hi = (uint32_t)((uint64_t)step >> 32);
  e = mpadam::launch_toy_step(a, stream);
  if (e != cudaSuccess) return cuda_fail(e, "launch of the diagnostic's kernels");
  return MPADAM_OK;
}

extern "C" int32_t mpadam_toy_run(mpadam_toy_state* s, uint16_t* w, const float* wstar, int64_t first_step,
                                  int64_t steps, double* losses, cudaStream_t stream) {
  if (!s) return fail(MPADAM_EINVAL, "state is NULL");
  if (!w || !wstar || !is_aligned(w, 2) || !is_aligned(wstar, 4)) return fail(MPADAM_EINVAL, "w / wstar NULL or misaligned");
  if (losses && !is_aligned(losses, 8)) return fail(MPADAM_EINVAL, "losses misaligned");
  if (first_step < 1 || steps < 0) return fail(MPADAM_EINVAL, "first_step must be >= 1 and steps >= 0");
  if (steps == 0) return MPADAM_OK;
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev != s->device) return fail(MPADAM_EINVAL, "current device %d differs from the state's device %d", dev, s->device);
  mpadam::ToyArgs a = s->a;
  a.w = w;
  a.wstar = wstar;
  a.loss_out = nullptr;
  a.t_dev = s->t_dev;
  a.loss_base = losses;
  // the graph of kToyGraphSteps steps, captured once per set of pointers
  if (steps >= kToyGraphSteps && (!s->exec || s->g_w != w || s->g_ws != wstar || s->g_loss != losses)) {
    if (s->exec) { cudaGraphExecDestroy(s->exec); s->exec = nullptr; }
    if (!s->cap && (e = cudaStreamCreateWithFlags(&s->cap, cudaStreamNonBlocking)) != cudaSuccess)
      return cuda_fail(e, "cudaStreamCreate");
    if ((e = cudaStreamBeginCapture(s->cap, cudaStreamCaptureModeThreadLocal)) != cudaSuccess)
      return cuda_fail(e, "cudaStreamBeginCapture");
    cudaError_t le = cudaSuccess;
    for (int64_t i = 0; i < kToyGraphSteps && le == cudaSuccess; ++i) le = mpadam::launch_toy_step(a, s->cap);
    cudaGraph_t graph = nullptr;
    e = cudaStreamEndCapture(s->cap, &graph);
    if (le != cudaSuccess || e != cudaSuccess) {
      if (graph) cudaGraphDestroy(graph);
      return cuda_fail(le != cudaSuccess ? le : e, "capture of the diagnostic's run graph");
    }
    e = cudaGraphInstantiate(&s->exec, graph, 0);
    cudaGraphDestroy(graph);
    if (e != cudaSuccess) { s->exec = nullptr; return cuda_fail(e, "cudaGraphInstantiate"); }
    s->g_w = w;
    s->g_ws = wstar;
    s->g_loss = losses;
  }
  if ((e = mpadam::launch_toy_set_step(s->t_dev, first_step, stream)) != cudaSuccess)
    return cuda_fail(e, "launch of the step-counter kernel");
  int64_t done = 0;
  for (; s->exec && done + kToyGraphSteps <= steps; done += kToyGraphSteps)
    if ((e = cudaGraphLaunch(s->exec, stream)) != cudaSuccess) return cuda_fail(e, "cudaGraphLaunch");
  for (; done < steps; ++done)
    if ((e = mpadam::launch_toy_step(a, stream)) != cudaSuccess) return cuda_fail(e, "launch of the diagnostic's kernels");
  return MPADAM_OK;
}

extern "C" int32_t mpadam_toy_destroy(mpadam_toy_state* s) {
  if (!s) return MPADAM_OK;
  cudaDeviceSynchronize();
  if (s->exec) cudaGraphExecDestroy(s->exec);
  if (s->cap) cudaStreamDestroy(s->cap);
  if (s->t_dev) cudaFree(s->t_dev);
  mpadam::ToyArgs& a = s->a;
  for (void* p : {(void*)a.cnt, (void*)a.first, (void*)a.idx, (void*)a.res, (void*)a.partial})
    if (p) cudaFree(p);
  delete s;
  return MPADAM_OK;
}

// ---------------------------------------------------------------------------
// Huge-page, page-locked host buffers for mpadam_step_host
// ---------------------------------------------------------------------------
extern "C" int32_t mpadam_host_buffer_alloc(int64_t bytes, void** out) {
  if (!out) return fail(MPADAM_EINVAL, "out is NULL");
  *out = nullptr;
  if (bytes <= 0) return fail(MPADAM_EINVAL, "bytes must be > 0");
  void* p = mmap(nullptr, (size_t)bytes, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
  if (p == MAP_FAILED) return fail(MPADAM_EALLOC, "mmap of %lld bytes failed", (long long)bytes);
#ifdef MADV_HUGEPAGE
  madvise(p, (size_t)bytes, MADV_HUGEPAGE);  // advice only: a kernel without it still gives a valid buffer
#endif
  // Place the pages on the host NUMA node nearest the current GPU (as the
  // driver's own pinned allocations are): on multi-socket hosts, first touch
  // by a thread on the far socket put them across the socket link.
  int dev = 0, node = -1;
  if (cudaGetDevice(&dev) == cudaSuccess && cudaDeviceGetAttribute(&node, cudaDevAttrHostNumaId, dev) == cudaSuccess &&
      node >= 0 && node < 1024) {
    unsigned long mask[1024 / (8 * sizeof(unsigned long))] = {};
    mask[node / (8 * sizeof(unsigned long))] |= 1UL << (node % (8 * sizeof(unsigned long)));
    const long kMpolPreferred = 1;
    syscall(SYS_mbind, p, (unsigned long)bytes, kMpolPreferred, mask, 1024UL + 1UL, 0UL);  // advice: failure is harmless
  }
  std::memset(p, 0, (size_t)bytes);  // resident before registration
  cudaError_t e = cudaHostRegister(p, (size_t)bytes, cudaHostRegisterDefault);
  if (e != cudaSuccess) {
    munmap(p, (size_t)bytes);
    return cuda_fail(e, "cudaHostRegister");
  }
  *out = p;
  return MPADAM_OK;
}

extern "C" int32_t mpadam_host_buffer_free(void* ptr, int64_t bytes) {
  if (!ptr) return MPADAM_OK;
  if (bytes <= 0) return fail(MPADAM_EINVAL, "bytes must be > 0");
  cudaError_t e = cudaHostUnregister(ptr);
  munmap(ptr, (size_t)bytes);
  if (e != cudaSuccess) return cuda_fail(e, "cudaHostUnregister");
  return MPADAM_OK;
}

extern "C" int32_t mpadam_debug_fail_allocation(int32_t after) {
  if (after < -1) return fail(MPADAM_EINVAL, "after must be >= -1");
  g_fail_countdown.store(after);
  return MPADAM_OK;
}

extern "C" int32_t mpadam_debug_tile_schedule(const int64_t* numel, int32_t n, int32_t ctas, int32_t static_q,
                                              int32_t chunk_tiles, int64_t* cta_runs, int32_t* cta_first,
                                              int64_t* pool, int32_t pool_cap, int32_t* pool_count) {
  if (n < 0 || (n > 0 && !numel)) return fail(MPADAM_EINVAL, "numel is NULL or n < 0");
  if (ctas < 1 || ctas > (1 << 20)) return fail(MPADAM_EINVAL, "ctas must be in [1, 2^20]");
  if (static_q < 0 || static_q > 1024) return fail(MPADAM_EINVAL, "static_q must be in [0, 1024]");
  if (chunk_tiles < 1 || chunk_tiles > (1 << 20)) return fail(MPADAM_EINVAL, "chunk_tiles must be in [1, 2^20]");
  if (!cta_runs || !cta_first || !pool_count || (pool_cap > 0 && !pool) || pool_cap < 0)
    return fail(MPADAM_EINVAL, "NULL output or negative pool_cap");
  int64_t tiles = 0;
  for (int32_t k = 0; k < n; ++k) {
    if (numel[k] < 0) return fail(MPADAM_EINVAL, "numel[%d] < 0", k);
    tiles += tiles_of(numel[k]);
  }
  try {
    std::vector<mpadam::PoolChunk> chunks;
    pool_host(numel, n, tiles, ctas, static_q, chunk_tiles, chunks);
    *pool_count = (int32_t)std::min<size_t>(chunks.size(), (size_t)INT32_MAX);
    if (chunks.size() > (size_t)pool_cap) return fail(MPADAM_EINVAL, "pool_cap %d < %zu chunks", pool_cap, chunks.size());
    for (size_t i = 0; i < chunks.size(); ++i) {
      pool[3 * i] = chunks[i].start;
      pool[3 * i + 1] = chunks[i].count;
      pool[3 * i + 2] = chunks[i].first;
    }
    std::vector<int32_t> first(ctas);
    cta_first_table(numel, n, tiles, ctas, first.data());
    for (int32_t b = 0; b < ctas; ++b) {
      const int64_t tb = (int64_t)b * tiles / ctas, te = ((int64_t)b + 1) * tiles / ctas;
      // the kernel's split: a launch brings a pool only when it has chunks
      cta_runs[3 * b] = tb;
      cta_runs[3 * b + 1] = chunks.empty() ? te : tb + (te - tb) * static_q / 1024;
      cta_runs[3 * b + 2] = te;
      cta_first[b] = first[b];
    }
  } catch (const std::bad_alloc&) {
    return fail(MPADAM_EALLOC, "host allocation failed");
  }
  return MPADAM_OK;
}
