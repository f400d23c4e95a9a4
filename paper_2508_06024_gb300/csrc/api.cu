// C ABI of libec2moe.so (declared in include/ec2moe.h): host-side argument
// checks, workspace layout and the order of launches for each step of the
// EC^2MoE MoE-layer forward.
#include <cuda_runtime.h>

#include <stdlib.h>

#include <mutex>
#include <vector>

#include "ec2moe.h"
#include "internal.h"

namespace ec2moe {

namespace {
thread_local int t_launches = 0;
thread_local bool t_plain_next = false;

// Per-launch timing records (ec2moe_profile_*).  Events come from a pool that
// is reused after ec2moe_profile_reset.
struct ProfRecord {
  const char* name;
  cudaEvent_t start, stop;
};
std::mutex g_prof_mu;
bool g_prof_on = false;
int g_prof_only = -1;  // >= 0: bracket only the launch with this index in each call
std::vector<ProfRecord> g_prof;
std::vector<cudaEvent_t> g_pool;
size_t g_pool_used = 0;

// Records `e` on `s`; inside a stream capture the record becomes a graph node
// (cudaEventRecordExternal), so timings survive graph replay.
void record_on(cudaEvent_t e, cudaStream_t s) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusActive)
    cudaEventRecordWithFlags(e, s, cudaEventRecordExternal);
  else
    cudaEventRecord(e, s);
}

cudaEvent_t pool_event() {
  if (g_pool_used == g_pool.size()) {
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    g_pool.push_back(e);
  }
  return g_pool[g_pool_used++];
}
}  // namespace

void reset_launch_count() {
  t_launches = 0;
  t_plain_next = false;
}

bool next_launch_pdl() {
  static const bool disabled = [] {
    const char* v = getenv("EC2MOE_NO_PDL");
    return v && v[0] == '1';
  }();
  return !disabled && t_launches > 0 && !t_plain_next;
}
void plain_next_launch() { t_plain_next = true; }
int launch_count() { return t_launches; }

KernelScope::KernelScope(const char* name, cudaStream_t s) : name_(name), s_(s) {
  std::lock_guard<std::mutex> lock(g_prof_mu);
  if (g_prof_on && (g_prof_only < 0 || g_prof_only == t_launches)) {
    start_ = pool_event();
    if (start_) record_on(start_, s_);
  }
}

KernelScope::~KernelScope() {
  ++t_launches;
  t_plain_next = false;
  std::lock_guard<std::mutex> lock(g_prof_mu);
  if (g_prof_on && start_) {
    cudaEvent_t stop = pool_event();
    if (stop) {
      record_on(stop, s_);
      g_prof.push_back(ProfRecord{name_, start_, stop});
    }
  }
}

int sm_count() {
  static std::mutex mu;
  static std::vector<int> cache;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  std::lock_guard<std::mutex> lock(mu);
  if ((int)cache.size() <= dev) cache.resize(dev + 1, 0);
  if (cache[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 1;
    cache[dev] = n;
  }
  return cache[dev];
}

cudaError_t ensure_smem_attr(const void* kernel, int bytes) {
  struct Entry {
    int dev;
    const void* kernel;
    int bytes;
  };
  static std::mutex mu;
  static std::vector<Entry> set;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  for (Entry& en : set) {
    if (en.dev == dev && en.kernel == kernel) {
      if (en.bytes >= bytes) return cudaSuccess;
      e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
      if (e == cudaSuccess) en.bytes = bytes;
      return e;
    }
  }
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) set.push_back(Entry{dev, kernel, bytes});
  return e;
}

}  // namespace ec2moe

using namespace ec2moe;

namespace {

constexpr size_t ALIGN = 256;
size_t align_up(size_t x) { return (x + ALIGN - 1) / ALIGN * ALIGN; }
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t esize(const ec2moe_layer_desc* d) { return d->dtype == EC2MOE_BF16 ? 2 : 4; }
bool is_bf16(const ec2moe_layer_desc* d) { return d->dtype == EC2MOE_BF16; }

// Shape checks common to every entry point.
ec2moe_status check_desc(const ec2moe_layer_desc* d) {
  if (!d) return EC2MOE_ERR_INVALID_ARG;
  if (d->T < 0 || d->d <= 0 || d->E <= 0 || d->k <= 0 || d->n_groups <= 0 || d->r < 0 || d->n_shared < 0)
    return EC2MOE_ERR_INVALID_ARG;
  if (d->dtype != EC2MOE_F32 && d->dtype != EC2MOE_BF16) return EC2MOE_ERR_INVALID_ARG;
  if (d->act != EC2MOE_GELU && d->act != EC2MOE_SWIGLU) return EC2MOE_ERR_INVALID_ARG;
  if (d->renorm_topk != 0 && d->renorm_topk != 1) return EC2MOE_ERR_INVALID_ARG;
  if (d->top_groups < 0) return EC2MOE_ERR_INVALID_ARG;
  if (d->E % d->n_groups != 0) return EC2MOE_ERR_INVALID_ARG;
  if (d->k > d->E) return EC2MOE_ERR_TOO_FEW_EXPERTS;
  if (d->E > EC2MOE_MAX_EXPERTS || d->n_groups > EC2MOE_MAX_GROUPS || d->k > EC2MOE_MAX_TOPK ||
      d->n_shared > EC2MOE_MAX_SHARED)
    return EC2MOE_ERR_UNSUPPORTED;
  if ((long long)d->T * d->k + (long long)d->T * (d->n_shared + 1) > 0x7fffffffLL) return EC2MOE_ERR_UNSUPPORTED;
  // Row pitches must be multiples of 16 bytes (vector loads, TMA strides) and,
  // for the tensor-core path, output widths multiples of 32 columns.
  if (d->d % 8 != 0) return EC2MOE_ERR_MISALIGNED;
  return EC2MOE_OK;
}

ec2moe_status check_ffn(const ec2moe_layer_desc* d, int d_ff) {
  if (d_ff <= 0) return EC2MOE_ERR_INVALID_ARG;
  if (d_ff % 8 != 0) return EC2MOE_ERR_MISALIGNED;
  if (is_bf16(d) && (d_ff % 32 != 0 || d->d % 32 != 0)) return EC2MOE_ERR_UNSUPPORTED;
  return EC2MOE_OK;
}

ec2moe_status check_codec(const ec2moe_layer_desc* d) {
  if (d->r <= 0) return EC2MOE_ERR_INVALID_ARG;
  if (d->r % 8 != 0) return EC2MOE_ERR_MISALIGNED;
  if (is_bf16(d) && (d->r % 32 != 0 || d->d % 32 != 0)) return EC2MOE_ERR_UNSUPPORTED;
  return EC2MOE_OK;
}

ec2moe_status check_mask(const ec2moe_layer_desc* d, const uint8_t* mask, uint32_t bits[4]) {
  if (!mask) return EC2MOE_ERR_INVALID_ARG;
  bits[0] = bits[1] = bits[2] = bits[3] = 0;
  int n = 0;
  for (int e = 0; e < d->E; ++e)
    if (mask[e]) {
      bits[e >> 5] |= 1u << (e & 31);
      ++n;
    }
  if (n == 0) return EC2MOE_ERR_ALL_MASKED;
  if (n < d->k) return EC2MOE_ERR_TOO_FEW_EXPERTS;
  if (d->top_groups > 0 && d->n_groups > 1) {
    // top-group pruning: the G live groups with the fewest allowed experts
    // must still hold k candidates
    int sizes[EC2MOE_MAX_GROUPS];
    int live = 0;
    const int gsize = d->E / d->n_groups;
    for (int g = 0; g < d->n_groups; ++g) {
      int c = 0;
      for (int e = g * gsize; e < (g + 1) * gsize; ++e) c += mask[e] ? 1 : 0;
      if (c > 0) sizes[live++] = c;
    }
    if (d->top_groups < live) {
      for (int i = 1; i < live; ++i)
        for (int j = i; j > 0 && sizes[j] < sizes[j - 1]; --j) {
          const int t = sizes[j];
          sizes[j] = sizes[j - 1];
          sizes[j - 1] = t;
        }
      int floor_k = 0;
      for (int i = 0; i < d->top_groups; ++i) floor_k += sizes[i];
      if (floor_k < d->k) return EC2MOE_ERR_TOO_FEW_EXPERTS;
    }
  }
  return EC2MOE_OK;
}

#define EC2MOE_REQUIRE_PTR(p)                   \
  do {                                          \
    if (!(p)) return EC2MOE_ERR_INVALID_ARG;    \
    if (!aligned16(p)) return EC2MOE_ERR_MISALIGNED; \
  } while (0)

#define EC2MOE_CUDA(call)                        \
  do {                                           \
    if ((call) != cudaSuccess) return EC2MOE_ERR_CUDA; \
  } while (0)

// Workspace of ec2moe_layer_forward, each region 256-byte aligned.
// Split-K of the routed down projection for decode-sized batches: with few
// rows per expert only (experts with rows) x (d / 256) output tiles exist for
// a long K = d_ff, fewer than the SMs, each streaming its weights alone; the
// K range is split so every SM streams, the partial sums (fp32) are reduced,
// weighted and combined by one small kernel.
constexpr int SPLITK_MAX = 8;

// Decode steps of at most gate_prefetch_max_tokens() tokens whose up
// projection runs on the swapped-operand kernel: the small-batch decision
// kernel prefetches into L2 the first bytes of the weight tile each of that
// kernel's CTAs streams first (W1, and W3 for SwiGLU), about 80 MB in all,
// while the codec kernels between them leave HBM idle.
constexpr long long PREFETCH_BUDGET = 80LL << 20;
void set_weight_prefetch(const ec2moe_layer_desc* d, const ec2moe_layer_weights* w, int n_allowed, GateArgs* ga) {
  const long long n = (long long)d->T * d->k;
  if (d->dtype != EC2MOE_BF16 || !ga->gate_partial || d->T > gate_prefetch_max_tokens() || !swap_gemm_enabled() ||
      n > SWAP_MAX_ROWS)
    return;
  const bool glu = d->act == EC2MOE_SWIGLU;
  const int tile_rows = glu ? 64 : 128;  // rows of W1 (and W3) per swapped-GEMM weight tile
  if (d->d_ff % tile_rows != 0) return;
  const long long experts = n < n_allowed ? n : n_allowed;
  const long long units = experts * (d->d_ff / tile_rows);
  const int ctas = static_cast<int>(units < sm_count() ? units : sm_count());
  const long long per_row = PREFETCH_BUDGET / ((long long)ctas * tile_rows * (glu ? 2 : 1));
  const long long row_bytes = (long long)d->d * 2;
  const int bytes = static_cast<int>((per_row < row_bytes ? per_row : row_bytes) / 16 * 16);
  if (bytes < 16) return;
  ga->pf_w1 = w->W1;
  ga->pf_w3 = glu ? w->W3 : nullptr;
  ga->pf_dff = d->d_ff;
  ga->pf_tile_rows = tile_rows;
  ga->pf_units = ctas;
  ga->pf_row_bytes = bytes;
}
bool splitk_possible(const ec2moe_layer_desc* d) {
  const long long n = (long long)d->T * d->k;
  return d->dtype == EC2MOE_BF16 && n >= 1 && n <= 128 && d->d_ff >= 4096 && d->d % 4 == 0;
}
// The split whose (tile x K range) units fill whole waves of the SMs best.
// Groups of at most SWAP_MAX_ROWS rows go to the swapped tensor-core kernel
// (d / 128 weight tiles per expert with rows); otherwise the expected m-tiles
// are one per expert with rows, at least n / 128, with d / 256 tiles each.
int splitk_factor(const ec2moe_layer_desc* d, int n_allowed) {
  if (!splitk_possible(d)) return 1;
  const long long n = (long long)d->T * d->k;
  const long long experts = n < n_allowed ? n : n_allowed;
  if (swap_gemm_enabled() && n <= SWAP_MAX_ROWS)
    return swap_split_factor(experts * swap_tiles_per_group(d->d, EPI_PARTIAL), d->d_ff, SPLITK_MAX);
  if (n <= 4) return 1;  // the weight-streaming kernel takes the whole K
  const long long m_tiles = experts > (n + 127) / 128 ? experts : (n + 127) / 128;
  const long long tiles = m_tiles * ((d->d + 255) / 256);
  const long long sms = sm_count();
  int best = 1;
  double best_eff = -1.0;
  for (int sp = 1; sp <= SPLITK_MAX; ++sp) {
    const long long units = tiles * sp;
    const long long waves = (units + sms - 1) / sms;
    const double eff = (double)units / (double)(waves * sms) - 0.002 * sp;  // prefer fewer splits on ties
    if (eff > best_eff) {
      best_eff = eff;
      best = sp;
    }
  }
  return best;
}

// Split-K encoder for decode-sized batches: with T <= 256 rows the encoder
// has at most 2 x (r / 128) output tiles over K = d_model, so one CTA per tile
// would stream V_enc alone; the K range is split (at least two k-blocks of 64
// per range, at most 32 ranges, about one unit per SM) and one small kernel
// adds the fp32 partial sums into Z.
constexpr int ENC_SPLIT_MAX = 32;
int enc_split(const ec2moe_layer_desc* d) {
  if (!is_bf16(d) || d->r <= 0 || d->r % 128 != 0 || d->T > 256 || d->d < 1024) return 1;
  const long long tiles = (long long)((d->T + 127) / 128) * (d->r / 128);
  long long s = sm_count() / tiles;
  if (s > d->d / 128) s = d->d / 128;
  if (s > ENC_SPLIT_MAX) s = ENC_SPLIT_MAX;
  if (s < 2) return 1;
  // the count of non-empty ranges the GEMM derives from this request
  const long long nk = (d->d + 63) / 64, per = (nk + s - 1) / s;
  return static_cast<int>((nk + per - 1) / per);
}

struct LayerWs {
  size_t z, xa, h, slot, shared, perm, inv_perm, offsets, blk, wsplit, part, zpart, gpart, total;
};
LayerWs layer_ws(const ec2moe_layer_desc* d) {
  LayerWs w{};
  const size_t es = esize(d);
  const size_t T = d->T, k = d->k, dm = d->d;
  const size_t ff = d->d_ff > d->d_ff_shared ? d->d_ff : d->d_ff_shared;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t at = off;
    off += align_up(bytes);
    return at;
  };
  w.z = take(d->r > 0 ? T * d->r * es : 0);
  w.xa = take((T * k + T) * dm * es);                          // expert-ordered rows, then X_hat
  w.h = take((T * k + (size_t)d->n_shared * T) * ff * es);    // hidden activations
  const bool direct = (d->k == 1 && d->n_shared == 0);
  w.slot = take(direct ? 0 : T * k * dm * es);
  w.shared = take((size_t)d->n_shared * T * dm * es);
  w.perm = take(T * k * 4);
  w.inv_perm = take(T * k * 4);
  w.offsets = take((d->E + 1) * 4);
  w.blk = take((size_t)route_blocks((long long)T * k) * d->E * 4);
  w.wsplit = take(gate_split_bytes(d->E, d->n_groups, d->d, is_bf16(d)));
  w.part = take(splitk_possible(d) ? (size_t)SPLITK_MAX * T * k * dm * 4 : 0);
  w.zpart = take(is_bf16(d) && d->r > 0 && d->T <= 256 ? (size_t)ENC_SPLIT_MAX * T * d->r * 4 : 0);
  w.gpart = take(gate_partial_bytes(d->T, d->d, d->E, d->n_groups));
  w.total = off;
  return w;
}

GemmArgs gemm_base() {
  GemmArgs g{};
  g.timeout_cycles = default_timeout_cycles();
  g.self_row_base = -1;
  return g;
}

cudaError_t run_gemm(const ec2moe_layer_desc* d, const GemmArgs& g, int epi, cudaStream_t s) {
  if (!is_bf16(d)) return launch_gemm_simt(g, epi, s);
  // decode-sized groups: weight rows on the MMA's M side (tensor cores), else
  // streamed once on the CUDA cores
  if (gemm_swap_supported(g, epi)) return launch_gemm_swap(g, epi, s);
  if (gemm_skinny_supported(g, epi)) return launch_gemm_skinny(g, epi, s);
  return launch_gemm_tc(g, epi, s);
}

// Up projection (+ activation) then down projection over groups of rows.
//   routed: groups = experts by device offsets; down projection scatters with
//           perm and scales with the gate weights.
//   shared: groups = shared experts, each over all T rows of A.
cudaError_t run_ffn(const ec2moe_layer_desc* d, bool routed, const void* A, long long a_rows, long long a_row_base,
                    const int32_t* offsets, const void* W1, const void* W3, const void* W2, void* H, long long h_rows,
                    long long h_row_base, const int32_t* perm, const float* scale, void* out, long long out_row_base,
                    cudaStream_t s, int g_active = 0, float* partial = nullptr, int split_k = 1) {
  const int ff = routed ? d->d_ff : d->d_ff_shared;
  const int G = routed ? d->E : d->n_shared;
  const long long rows = routed ? (long long)d->T * d->k : (long long)d->T * d->n_shared;
  const int act_epi = d->act == EC2MOE_SWIGLU ? EPI_SWIGLU : EPI_GELU;
  GemmArgs up = gemm_base();
  up.name = routed ? "expert_up" : "shared_up";
  up.A = A;
  up.a_rows = a_rows;
  up.B = W1;
  up.B2 = W3;
  up.b_rows = (long long)G * ff;
  up.offsets = routed ? offsets : nullptr;
  up.G = G;
  up.M = routed ? 0 : d->T;
  up.a_shared = routed ? 0 : 1;
  up.a_row_base = a_row_base;
  up.out_row_base = h_row_base;
  up.N = ff;
  up.K = d->d;
  up.b_group_rows = ff;
  up.out = H;
  up.ldo = ff;
  up.max_rows = rows;
  up.group_rows_bound = routed ? rows : d->T;
  up.g_active = routed ? g_active : 0;
  cudaError_t e = run_gemm(d, up, act_epi, s);
  if (e != cudaSuccess) return e;
  GemmArgs dn = gemm_base();
  dn.name = routed ? "expert_down" : "shared_down";
  dn.A = H;
  dn.a_rows = h_rows;
  dn.B = W2;
  dn.B2 = nullptr;
  dn.b_rows = (long long)G * d->d;
  dn.offsets = routed ? offsets : nullptr;
  dn.G = G;
  dn.M = routed ? 0 : d->T;
  dn.a_shared = 0;
  dn.a_row_base = h_row_base;
  dn.out_row_base = routed ? 0 : out_row_base;
  dn.N = d->d;
  dn.K = ff;
  dn.b_group_rows = d->d;
  dn.out = out;
  dn.ldo = d->d;
  dn.perm = routed ? perm : nullptr;
  dn.scale = routed ? scale : nullptr;
  if (routed && split_k > 1 && partial) {
    // split-K partial sums; the gate weights and the unpermute come in the reduce
    dn.split_k = split_k;
    dn.partial = partial;
    dn.part_rows = rows;
    dn.max_rows = rows;
    dn.group_rows_bound = rows;
    return run_gemm(d, dn, EPI_PARTIAL, s);
  }
  dn.max_rows = rows;
  dn.group_rows_bound = routed ? rows : d->T;
  dn.g_active = routed ? g_active : 0;
  return run_gemm(d, dn, routed ? EPI_SCATTER : EPI_STORE, s);
}

// Codec GEMM.  With `inv_perm` (decode only), row t of X_hat is written to
// rows inv_perm[t*k + s] (s < k) of `out` -- the expert-ordered activations --
// and, when self_row_base >= 0, also to row self_row_base + t.
struct RelPlace {  // relative placement of decoded rows (routing fused into the gate)
  const int32_t* counts = nullptr;
  const int32_t* idx = nullptr;
  int32_t* perm_out = nullptr;
  int32_t* offsets_out = nullptr;
};

cudaError_t run_codec(const ec2moe_layer_desc* d, bool encode, const void* in, const void* V, void* out,
                      cudaStream_t s, const int32_t* inv_perm = nullptr, long long self_row_base = -1,
                      const RelPlace& rel = RelPlace(), float* enc_partial = nullptr) {
  GemmArgs g = gemm_base();
  g.name = encode ? "lr_encode" : "lr_decode";
  g.A = in;
  g.a_rows = d->T;
  g.B = V;
  g.b_rows = encode ? d->r : d->d;
  g.G = 1;
  g.M = d->T;
  g.N = encode ? d->r : d->d;
  g.K = encode ? d->d : d->r;
  g.b_group_rows = 0;
  g.out = out;
  g.ldo = g.N;
  g.max_rows = d->T;
  if (inv_perm) {
    g.perm = inv_perm;
    g.rep_k = d->k;
    g.self_row_base = self_row_base;
    g.rep_counts = rel.counts;
    g.rep_idx = rel.idx;
    g.rep_perm_out = rel.perm_out;
    g.rep_offsets_out = rel.offsets_out;
    g.rep_E = d->E;
    return run_gemm(d, g, EPI_REPLICATE, s);
  }
  const int split = encode && enc_partial ? enc_split(d) : 1;
  if (split > 1) {
    g.split_k = split;
    g.partial = enc_partial;
    g.part_rows = d->T;
    cudaError_t e = run_gemm(d, g, EPI_PARTIAL, s);
    if (e != cudaSuccess) return e;
    return launch_splitk_sum(enc_partial, split, d->T, d->r, out, s);
  }
  return run_gemm(d, g, EPI_STORE, s);
}

// Steps 4-5 of a layer call on one stream, after the expert-ordered rows
// (xa), perm and offsets exist: routed experts (gate scale and unpermute in
// the down projection, or split-K partial sums), the always-on shared
// experts, and the fixed-order combine or the split-K reduce into Y.
struct ExpertStage {
  const void* xa;               // [n + T, d]: expert-ordered rows, then X_hat
  const void* shared_a;         // rows the shared experts read
  long long shared_a_rows, shared_a_base;
  void* h;                      // hidden rows
  void* slot;                   // per-slot outputs (== Y when direct)
  void* shared;                 // shared experts' outputs
  float* partial;               // split-K partial sums (split > 1)
  int split;
  bool direct, routed;
  const int32_t* offsets;
  const int32_t* perm;
  const int32_t* inv_perm;
  const int32_t* topk_idx;
  const float* topk_w;
  void* Y;
  int n_allowed;
};

cudaError_t run_expert_stage(const ec2moe_layer_desc* d, const ec2moe_layer_weights* w, const ExpertStage& x,
                             cudaStream_t s) {
  const long long T = d->T, n = T * d->k;
  const bool bf = is_bf16(d);
  cudaError_t e = run_ffn(d, true, x.xa, n + T, 0, x.offsets, w->W1, w->W3, w->W2, x.h,
                          n + (long long)d->n_shared * T, 0, x.perm, x.topk_w, x.slot, 0, s, x.n_allowed, x.partial,
                          x.split);
  if (e != cudaSuccess) return e;
  if (d->n_shared > 0) {
    e = run_ffn(d, false, x.shared_a, x.shared_a_rows, x.shared_a_base, nullptr, w->W1s, w->W3s, w->W2s, x.h,
                n + (long long)d->n_shared * T, n, nullptr, nullptr, x.shared, 0, s);
    if (e != cudaSuccess) return e;
  }
  if (x.split > 1)
    return launch_splitk_combine(x.partial, x.split, n, x.offsets, x.topk_idx, x.inv_perm, x.routed, x.topk_w,
                                 x.shared, d->n_shared, x.Y, d->T, d->k, d->d, s);
  if (!x.direct) return launch_combine(x.slot, x.shared, d->n_shared, x.Y, d->T, d->k, d->d, bf, s);
  return cudaSuccess;
}

// Argument checks of a whole-layer call (everything but the workspace).
ec2moe_status check_layer_call(const ec2moe_layer_desc* desc, const ec2moe_layer_weights* w, const void* X,
                               const uint8_t* mask, void* Y, int32_t* topk_idx, float* topk_w, int32_t* counts,
                               void* Z, uint32_t mask_bits[4], bool* empty) {
  *empty = false;
  ec2moe_status st = check_desc(desc);
  if (st != EC2MOE_OK) return st;
  if (!w) return EC2MOE_ERR_INVALID_ARG;
  st = check_mask(desc, mask, mask_bits);
  if (st != EC2MOE_OK) return st;
  st = check_ffn(desc, desc->d_ff);
  if (st != EC2MOE_OK) return st;
  if (desc->n_shared > 0) {
    st = check_ffn(desc, desc->d_ff_shared);
    if (st != EC2MOE_OK) return st;
  }
  if (desc->r > 0) {
    st = check_codec(desc);
    if (st != EC2MOE_OK) return st;
  }
  if (desc->T == 0) {
    *empty = true;
    return EC2MOE_OK;
  }
  EC2MOE_REQUIRE_PTR(X);
  EC2MOE_REQUIRE_PTR(Y);
  EC2MOE_REQUIRE_PTR(topk_idx);
  EC2MOE_REQUIRE_PTR(topk_w);
  if (!counts) return EC2MOE_ERR_INVALID_ARG;
  EC2MOE_REQUIRE_PTR(w->W_local);
  EC2MOE_REQUIRE_PTR(w->b_local);
  if (desc->n_groups > 1) {
    EC2MOE_REQUIRE_PTR(w->W_global);
    EC2MOE_REQUIRE_PTR(w->b_global);
  }
  EC2MOE_REQUIRE_PTR(w->W1);
  EC2MOE_REQUIRE_PTR(w->W2);
  if (desc->act == EC2MOE_SWIGLU) EC2MOE_REQUIRE_PTR(w->W3);
  if (desc->n_shared > 0) {
    EC2MOE_REQUIRE_PTR(w->W1s);
    EC2MOE_REQUIRE_PTR(w->W2s);
    if (desc->act == EC2MOE_SWIGLU) EC2MOE_REQUIRE_PTR(w->W3s);
  }
  if (desc->r > 0) {
    EC2MOE_REQUIRE_PTR(w->V_enc);
    EC2MOE_REQUIRE_PTR(w->V_dec);
    if (Z && !aligned16(Z)) return EC2MOE_ERR_MISALIGNED;
  }
  return EC2MOE_OK;
}

}  // namespace

extern "C" {

size_t ec2moe_workspace_size(const ec2moe_layer_desc* desc) {
  if (check_desc(desc) != EC2MOE_OK) return 0;
  return layer_ws(desc).total;
}

size_t ec2moe_experts_workspace_size(const ec2moe_layer_desc* desc) {
  if (check_desc(desc) != EC2MOE_OK) return 0;
  const size_t T = desc->T, k = desc->k;
  const size_t routed = T * k * desc->d_ff;
  const size_t shared = (size_t)desc->n_shared * T * desc->d_ff_shared;
  return align_up((routed > shared ? routed : shared) * esize(desc));
}

size_t ec2moe_route_workspace_size(const ec2moe_layer_desc* desc) {
  if (check_desc(desc) != EC2MOE_OK) return 0;
  return align_up((size_t)route_blocks((long long)desc->T * desc->k) * desc->E * 4);
}

ec2moe_status ec2moe_gate(const ec2moe_layer_desc* desc, const void* X, const float* W_local, const float* b_local,
                          const float* W_global, const float* b_global, const uint8_t* mask, int32_t* topk_idx,
                          float* topk_w, ec2moe_stream_t stream) {
  reset_launch_count();
  ec2moe_status st = check_desc(desc);
  if (st != EC2MOE_OK) return st;
  GateArgs a{};
  st = check_mask(desc, mask, a.mask_bits);
  if (st != EC2MOE_OK) return st;
  if (desc->T == 0) return EC2MOE_OK;
  EC2MOE_REQUIRE_PTR(X);
  EC2MOE_REQUIRE_PTR(W_local);
  EC2MOE_REQUIRE_PTR(b_local);
  EC2MOE_REQUIRE_PTR(topk_idx);
  EC2MOE_REQUIRE_PTR(topk_w);
  if (desc->n_groups > 1) {
    EC2MOE_REQUIRE_PTR(W_global);
    EC2MOE_REQUIRE_PTR(b_global);
  }
  a.X = X;
  a.W_local = W_local;
  a.b_local = b_local;
  a.W_global = desc->n_groups > 1 ? W_global : nullptr;
  a.b_global = desc->n_groups > 1 ? b_global : nullptr;
  a.T = desc->T;
  a.d = desc->d;
  a.E = desc->E;
  a.K = desc->n_groups;
  a.k = desc->k;
  a.renorm = desc->renorm_topk;
  a.top_groups = desc->top_groups;
  a.topk_idx = topk_idx;
  a.topk_w = topk_w;
  EC2MOE_CUDA(launch_gate(a, is_bf16(desc), stream));
  return EC2MOE_OK;
}

ec2moe_status ec2moe_route(const ec2moe_layer_desc* desc, const int32_t* topk_idx, int32_t* counts, int32_t* offsets,
                           int32_t* perm, int32_t* inv_perm, const void* src, int32_t width, void* dst,
                           void* workspace, size_t ws_bytes, ec2moe_stream_t stream) {
  reset_launch_count();
  ec2moe_status st = check_desc(desc);
  if (st != EC2MOE_OK) return st;
  if (!counts || !offsets) return EC2MOE_ERR_INVALID_ARG;
  if ((src == nullptr) != (dst == nullptr)) return EC2MOE_ERR_INVALID_ARG;
  if (src) {
    if (width <= 0) return EC2MOE_ERR_INVALID_ARG;
    if ((width * esize(desc)) % 16 != 0 || !aligned16(src) || !aligned16(dst)) return EC2MOE_ERR_MISALIGNED;
  }
  const long long n = (long long)desc->T * desc->k;
  if (n > 0) {
    if (!topk_idx || !perm) return EC2MOE_ERR_INVALID_ARG;
    if (!workspace || ws_bytes < ec2moe_route_workspace_size(desc)) return EC2MOE_ERR_WORKSPACE;
  }
  EC2MOE_CUDA(launch_route(topk_idx, n, desc->E, static_cast<int32_t*>(workspace), counts, offsets, perm, inv_perm,
                           stream));
  if (src && n > 0) EC2MOE_CUDA(launch_gather(src, dst, perm, n, desc->k, width, is_bf16(desc), stream));
  return EC2MOE_OK;
}

ec2moe_status ec2moe_route_noalloc(const ec2moe_layer_desc* desc, const int32_t* topk_idx, int32_t* counts,
                                   int32_t* offsets, int32_t* perm, int32_t* inv_perm, const void* src, int32_t width,
                                   void* dst, ec2moe_stream_t stream) {
  reset_launch_count();
  ec2moe_status st = check_desc(desc);
  if (st != EC2MOE_OK) return st;
  if (!counts || !offsets) return EC2MOE_ERR_INVALID_ARG;
  if ((src == nullptr) != (dst == nullptr)) return EC2MOE_ERR_INVALID_ARG;
  if (src) {
    if (width <= 0) return EC2MOE_ERR_INVALID_ARG;
    if ((width * esize(desc)) % 16 != 0 || !aligned16(src) || !aligned16(dst)) return EC2MOE_ERR_MISALIGNED;
  }
  const long long n = (long long)desc->T * desc->k;
  if ((long long)route_blocks(n) * desc->E > EC2MOE_ROUTE_NOALLOC_MAX_CELLS) return EC2MOE_ERR_UNSUPPORTED;
  if (n > 0 && (!topk_idx || !perm)) return EC2MOE_ERR_INVALID_ARG;
  EC2MOE_CUDA(launch_route_noalloc(topk_idx, n, desc->E, counts, offsets, perm, inv_perm, stream));
  if (src && n > 0) EC2MOE_CUDA(launch_gather(src, dst, perm, n, desc->k, width, is_bf16(desc), stream));
  return EC2MOE_OK;
}

ec2moe_status ec2moe_experts(const ec2moe_layer_desc* desc, const void* X_perm, const int32_t* offsets, const void* W1,
                             const void* W3, const void* W2, const float* topk_w, const int32_t* perm, void* slot_out,
                             void* workspace, size_t ws_bytes, ec2moe_stream_t stream) {
  reset_launch_count();
  ec2moe_status st = check_desc(desc);
  if (st != EC2MOE_OK) return st;
  st = check_ffn(desc, desc->d_ff);
  if (st != EC2MOE_OK) return st;
  if (desc->T == 0) return EC2MOE_OK;
  EC2MOE_REQUIRE_PTR(X_perm);
  EC2MOE_REQUIRE_PTR(W1);
  EC2MOE_REQUIRE_PTR(W2);
  if (desc->act == EC2MOE_SWIGLU) EC2MOE_REQUIRE_PTR(W3);
  EC2MOE_REQUIRE_PTR(slot_out);
  if (!offsets || !topk_w || !perm) return EC2MOE_ERR_INVALID_ARG;
  if (!workspace || ws_bytes < ec2moe_experts_workspace_size(desc)) return EC2MOE_ERR_WORKSPACE;
  if (!aligned16(workspace)) return EC2MOE_ERR_MISALIGNED;
  const long long rows = (long long)desc->T * desc->k;
  EC2MOE_CUDA(run_ffn(desc, true, X_perm, rows, 0, offsets, W1, W3, W2, workspace, rows, 0, perm, topk_w, slot_out, 0,
                      stream));
  return EC2MOE_OK;
}

ec2moe_status ec2moe_shared_experts(const ec2moe_layer_desc* desc, const void* X, const void* W1s, const void* W3s,
                                    const void* W2s, void* shared_out, void* workspace, size_t ws_bytes,
                                    ec2moe_stream_t stream) {
  reset_launch_count();
  ec2moe_status st = check_desc(desc);
  if (st != EC2MOE_OK) return st;
  if (desc->n_shared == 0) return EC2MOE_OK;
  st = check_ffn(desc, desc->d_ff_shared);
  if (st != EC2MOE_OK) return st;
  if (desc->T == 0) return EC2MOE_OK;
  EC2MOE_REQUIRE_PTR(X);
  EC2MOE_REQUIRE_PTR(W1s);
  EC2MOE_REQUIRE_PTR(W2s);
  if (desc->act == EC2MOE_SWIGLU) EC2MOE_REQUIRE_PTR(W3s);
  EC2MOE_REQUIRE_PTR(shared_out);
  if (!workspace || ws_bytes < ec2moe_experts_workspace_size(desc)) return EC2MOE_ERR_WORKSPACE;
  if (!aligned16(workspace)) return EC2MOE_ERR_MISALIGNED;
  const long long hrows = (long long)desc->T * desc->n_shared;
  EC2MOE_CUDA(run_ffn(desc, false, X, desc->T, 0, nullptr, W1s, W3s, W2s, workspace, hrows, 0, nullptr, nullptr,
                      shared_out, 0, stream));
  return EC2MOE_OK;
}

ec2moe_status ec2moe_combine(const ec2moe_layer_desc* desc, const void* slot_out, const void* shared_out, void* Y,
                             ec2moe_stream_t stream) {
  reset_launch_count();
  ec2moe_status st = check_desc(desc);
  if (st != EC2MOE_OK) return st;
  if (desc->T == 0) return EC2MOE_OK;
  EC2MOE_REQUIRE_PTR(slot_out);
  EC2MOE_REQUIRE_PTR(Y);
  if (shared_out && !aligned16(shared_out)) return EC2MOE_ERR_MISALIGNED;
  EC2MOE_CUDA(launch_combine(slot_out, shared_out, desc->n_shared, Y, desc->T, desc->k, desc->d, is_bf16(desc), stream));
  return EC2MOE_OK;
}

ec2moe_status ec2moe_lr_encode(const ec2moe_layer_desc* desc, const void* X, const void* V_enc, void* Z,
                               ec2moe_stream_t stream) {
  reset_launch_count();
  ec2moe_status st = check_desc(desc);
  if (st != EC2MOE_OK) return st;
  st = check_codec(desc);
  if (st != EC2MOE_OK) return st;
  if (desc->T == 0) return EC2MOE_OK;
  EC2MOE_REQUIRE_PTR(X);
  EC2MOE_REQUIRE_PTR(V_enc);
  EC2MOE_REQUIRE_PTR(Z);
  EC2MOE_CUDA(run_codec(desc, true, X, V_enc, Z, stream));
  return EC2MOE_OK;
}

ec2moe_status ec2moe_lr_decode(const ec2moe_layer_desc* desc, const void* Z, const void* V_dec, void* X_hat,
                               ec2moe_stream_t stream) {
  reset_launch_count();
  ec2moe_status st = check_desc(desc);
  if (st != EC2MOE_OK) return st;
  st = check_codec(desc);
  if (st != EC2MOE_OK) return st;
  if (desc->T == 0) return EC2MOE_OK;
  EC2MOE_REQUIRE_PTR(Z);
  EC2MOE_REQUIRE_PTR(V_dec);
  EC2MOE_REQUIRE_PTR(X_hat);
  EC2MOE_CUDA(run_codec(desc, false, Z, V_dec, X_hat, stream));
  return EC2MOE_OK;
}

ec2moe_status ec2moe_layer_forward(const ec2moe_layer_desc* desc, const ec2moe_layer_weights* w, const void* X,
                                   const uint8_t* mask, void* Y, int32_t* topk_idx, float* topk_w, int32_t* counts,
                                   void* Z, void* workspace, size_t ws_bytes, ec2moe_stream_t stream) {
  reset_launch_count();
  GateArgs ga{};
  bool empty = false;
  ec2moe_status st = check_layer_call(desc, w, X, mask, Y, topk_idx, topk_w, counts, Z, ga.mask_bits, &empty);
  if (st != EC2MOE_OK || empty) return st;
  const LayerWs L = layer_ws(desc);
  if (!workspace || ws_bytes < L.total) return EC2MOE_ERR_WORKSPACE;
  if (!aligned16(workspace)) return EC2MOE_ERR_MISALIGNED;

  uint8_t* ws = static_cast<uint8_t*>(workspace);
  const bool bf = is_bf16(desc);
  const size_t es = esize(desc);
  const long long T = desc->T, k = desc->k, n = T * k;
  void* zbuf = (desc->r > 0) ? (Z ? Z : ws + L.z) : nullptr;
  uint8_t* xa = ws + L.xa;  // [n + T, d]: expert-ordered rows, then X_hat
  void* h = ws + L.h;
  int n_allowed = 0;
  for (int e = 0; e < desc->E; ++e) n_allowed += mask[e] ? 1 : 0;
  const int split = splitk_factor(desc, n_allowed);
  float* partial = split > 1 ? reinterpret_cast<float*>(ws + L.part) : nullptr;
  const bool direct = (k == 1 && desc->n_shared == 0 && split == 1);
  void* slot = direct ? Y : static_cast<void*>(ws + L.slot);
  void* shared = desc->n_shared > 0 ? static_cast<void*>(ws + L.shared) : nullptr;
  int32_t* perm = reinterpret_cast<int32_t*>(ws + L.perm);
  int32_t* inv_perm = reinterpret_cast<int32_t*>(ws + L.inv_perm);
  int32_t* offsets = reinterpret_cast<int32_t*>(ws + L.offsets);
  int32_t* blk = reinterpret_cast<int32_t*>(ws + L.blk);

  // Steps 1-3a on the end: mask, group gate, Top-k on the original activations.
  ga.X = X;
  ga.W_local = w->W_local;
  ga.b_local = w->b_local;
  ga.W_global = desc->n_groups > 1 ? w->W_global : nullptr;
  ga.b_global = desc->n_groups > 1 ? w->b_global : nullptr;
  ga.T = desc->T;
  ga.d = desc->d;
  ga.E = desc->E;
  ga.K = desc->n_groups;
  ga.k = desc->k;
  ga.renorm = desc->renorm_topk;
  ga.top_groups = desc->top_groups;
  ga.topk_idx = topk_idx;
  ga.topk_w = topk_w;
  // bf16 layers route inside the gate kernel (per-tile row reservations); the
  // decoder (or the gather) then places rows and writes perm and offsets.
  if (bf) {
    ga.route_counts = counts;
    ga.route_rel = inv_perm;
    if (gate_split_bytes(desc->E, desc->n_groups, desc->d, bf)) ga.w_split = ws + L.wsplit;
  }
  if (gate_partial_bytes(desc->T, desc->d, desc->E, desc->n_groups))
    ga.gate_partial = reinterpret_cast<float*>(ws + L.gpart);
  set_weight_prefetch(desc, w, n_allowed, &ga);
  bool routed = false;
  int gate_sms = 0;
  EC2MOE_CUDA(launch_gate(ga, bf, stream, &routed, &gate_sms));
  // Step 3b: routing tables (inside the gate kernel when it could take them).
  if (!routed) EC2MOE_CUDA(launch_route(topk_idx, n, desc->E, blk, counts, offsets, perm, inv_perm, stream));
  RelPlace rel;
  if (routed) {
    rel.counts = counts;
    rel.idx = topk_idx;
    rel.perm_out = perm;
    rel.offsets_out = offsets;
  }
  // Step 6: encode at the end; decode in the cloud straight into expert order
  // (the decoder's epilogue writes each X_hat row to its (token, slot)
  // positions, and to the tail rows the shared experts read).
  const void* shared_a = xa;
  long long shared_a_rows = n + T, shared_a_base = n;
  if (desc->r > 0 && routed && codec_fused_supported(desc->d, desc->r)) {
    // encoder and decoder in one kernel; Z stays on chip between them
    CodecArgs ca{};
    ca.X = X;
    ca.V_enc = w->V_enc;
    ca.V_dec = w->V_dec;
    ca.Z = zbuf;
    ca.out = xa;
    ca.T = desc->T;
    ca.d = desc->d;
    ca.r = desc->r;
    ca.k = desc->k;
    ca.E = desc->E;
    ca.rel = inv_perm;
    ca.counts = counts;
    ca.topk_idx = topk_idx;
    ca.perm_out = perm;
    ca.offsets_out = offsets;
    ca.self_row_base = desc->n_shared > 0 ? n : -1;
    ca.timeout_cycles = default_timeout_cycles();
    ca.busy_sms = gate_sms;
    EC2MOE_CUDA(launch_codec_fused(ca, stream));
  } else if (desc->r > 0) {
    EC2MOE_CUDA(run_codec(desc, true, X, w->V_enc, zbuf, stream, nullptr, -1, RelPlace(),
                          reinterpret_cast<float*>(ws + L.zpart)));
    EC2MOE_CUDA(run_codec(desc, false, zbuf, w->V_dec, xa, stream, inv_perm, desc->n_shared > 0 ? n : -1, rel));
  } else {
    // Step 3b (move): rows of X into expert order; shared experts read X itself.
    if (routed)
      EC2MOE_CUDA(launch_gather_rel(X, xa, topk_idx, counts, inv_perm, perm, offsets, desc->E, n, desc->k, desc->d, bf,
                                    stream));
    else
      EC2MOE_CUDA(launch_gather(X, xa, perm, n, desc->k, desc->d, bf, stream));
    shared_a = X;
    shared_a_rows = T;
    shared_a_base = 0;
  }
  // Steps 4-5: routed and shared experts, combine (or the split-K reduce).
  const ExpertStage xs{xa, shared_a, shared_a_rows, shared_a_base, h, slot, shared, partial, split, direct, routed,
                       offsets, perm, inv_perm, topk_idx, topk_w, Y, n_allowed};
  EC2MOE_CUDA(run_expert_stage(desc, w, xs, stream));
  return EC2MOE_OK;
}

size_t ec2moe_pipelined_workspace_size(const ec2moe_layer_desc* desc, int32_t n_micro) {
  if (check_desc(desc) != EC2MOE_OK || n_micro < 1 || n_micro > EC2MOE_MAX_MICRO) return 0;
  ec2moe_layer_desc sub = *desc;
  sub.T = (desc->T + n_micro - 1) / n_micro;
  return (size_t)n_micro * align_up(layer_ws(&sub).total) + align_up((size_t)n_micro * desc->E * 4);
}

// The end/cloud pipeline of the paper's PO-ECC stage on one GPU: the tokens
// are cut into n_micro contiguous micro-batches; the end stream runs the gate,
// the routing and the encoder (Z) of micro-batch i + 1 while the cloud stream
// runs the decoder, the experts and the combine of micro-batch i.  Each
// micro-batch has its own workspace region, so the two streams share only the
// events that hand Z (and the routing tables) from the end to the cloud.
ec2moe_status ec2moe_layer_forward_pipelined(const ec2moe_layer_desc* desc, const ec2moe_layer_weights* w,
                                             const void* X, const uint8_t* mask, void* Y, int32_t* topk_idx,
                                             float* topk_w, int32_t* counts, void* Z, void* workspace,
                                             size_t ws_bytes, int32_t n_micro, ec2moe_stream_t stream_end,
                                             ec2moe_stream_t stream_cloud) {
  reset_launch_count();
  GateArgs ga0{};
  bool empty = false;
  ec2moe_status st = check_layer_call(desc, w, X, mask, Y, topk_idx, topk_w, counts, Z, ga0.mask_bits, &empty);
  if (st != EC2MOE_OK || empty) return st;
  if (n_micro < 1 || n_micro > EC2MOE_MAX_MICRO) return EC2MOE_ERR_INVALID_ARG;
  const size_t need = ec2moe_pipelined_workspace_size(desc, n_micro);
  if (!workspace || need == 0 || ws_bytes < need) return EC2MOE_ERR_WORKSPACE;
  if (!aligned16(workspace)) return EC2MOE_ERR_MISALIGNED;

  const bool bf = is_bf16(desc);
  const size_t es = esize(desc);
  const int Tm = (desc->T + n_micro - 1) / n_micro;
  ec2moe_layer_desc full_sub = *desc;
  full_sub.T = Tm;
  const size_t region = align_up(layer_ws(&full_sub).total);
  uint8_t* base = static_cast<uint8_t*>(workspace);
  int32_t* parts = reinterpret_cast<int32_t*>(base + (size_t)n_micro * region);
  int n_allowed = 0;
  for (int e = 0; e < desc->E; ++e) n_allowed += mask[e] ? 1 : 0;

  // one event per micro-batch hand-off, plus the fork and the join
  thread_local std::vector<cudaEvent_t> events;
  while ((int)events.size() < n_micro + 2) {
    cudaEvent_t e = nullptr;
    EC2MOE_CUDA(cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
    events.push_back(e);
  }
  cudaStream_t se = stream_end, sc = stream_cloud;
  EC2MOE_CUDA(cudaEventRecord(events[0], se));
  EC2MOE_CUDA(cudaStreamWaitEvent(sc, events[0], 0));

  int used = 0;
  for (int i = 0; i < n_micro; ++i) {
    const long long t0 = (long long)i * Tm;
    if (t0 >= desc->T) break;
    ++used;
    ec2moe_layer_desc sub = *desc;
    sub.T = (int)((desc->T - t0) < Tm ? (desc->T - t0) : Tm);
    const LayerWs L = layer_ws(&sub);
    uint8_t* ws = base + (size_t)i * region;
    const long long T = sub.T, k = sub.k, n = T * k;
    const void* Xi = static_cast<const uint8_t*>(X) + (size_t)t0 * sub.d * es;
    void* Yi = static_cast<uint8_t*>(Y) + (size_t)t0 * sub.d * es;
    int32_t* idx_i = topk_idx + t0 * k;
    float* tw_i = topk_w + t0 * k;
    int32_t* cnt_i = parts + (size_t)i * desc->E;
    void* zbuf = (sub.r > 0) ? (Z ? static_cast<void*>(static_cast<uint8_t*>(Z) + (size_t)t0 * sub.r * es)
                                  : static_cast<void*>(ws + L.z))
                             : nullptr;
    uint8_t* xa = ws + L.xa;
    void* h = ws + L.h;
    // the regions are sized for full micro-batches: split-K only where that
    // layout holds the partial sums
    const int split = splitk_possible(&full_sub) ? splitk_factor(&sub, n_allowed) : 1;
    float* partial = split > 1 ? reinterpret_cast<float*>(ws + L.part) : nullptr;
    const bool direct = (k == 1 && sub.n_shared == 0 && split == 1);
    void* slot = direct ? Yi : static_cast<void*>(ws + L.slot);
    void* shared = sub.n_shared > 0 ? static_cast<void*>(ws + L.shared) : nullptr;
    int32_t* perm = reinterpret_cast<int32_t*>(ws + L.perm);
    int32_t* inv_perm = reinterpret_cast<int32_t*>(ws + L.inv_perm);
    int32_t* offsets = reinterpret_cast<int32_t*>(ws + L.offsets);
    int32_t* blk = reinterpret_cast<int32_t*>(ws + L.blk);

    // ---- end: gate, routing, encoder
    GateArgs ga = ga0;
    ga.X = Xi;
    ga.W_local = w->W_local;
    ga.b_local = w->b_local;
    ga.W_global = sub.n_groups > 1 ? w->W_global : nullptr;
    ga.b_global = sub.n_groups > 1 ? w->b_global : nullptr;
    ga.T = sub.T;
    ga.d = sub.d;
    ga.E = sub.E;
    ga.K = sub.n_groups;
    ga.k = sub.k;
    ga.renorm = sub.renorm_topk;
    ga.top_groups = sub.top_groups;
    ga.topk_idx = idx_i;
    ga.topk_w = tw_i;
    if (bf) {
      ga.route_counts = cnt_i;
      ga.route_rel = inv_perm;
      if (gate_split_bytes(sub.E, sub.n_groups, sub.d, bf)) ga.w_split = ws + L.wsplit;
    }
    if (gate_partial_bytes(sub.T, sub.d, sub.E, sub.n_groups)) ga.gate_partial = reinterpret_cast<float*>(ws + L.gpart);
    bool routed = false;
    EC2MOE_CUDA(launch_gate(ga, bf, se, &routed));
    if (!routed) EC2MOE_CUDA(launch_route(idx_i, n, sub.E, blk, cnt_i, offsets, perm, inv_perm, se));
    if (sub.r > 0)
      EC2MOE_CUDA(run_codec(&sub, true, Xi, w->V_enc, zbuf, se, nullptr, -1, RelPlace(),
                            reinterpret_cast<float*>(ws + L.zpart)));
    EC2MOE_CUDA(cudaEventRecord(events[1 + i], se));

    // ---- cloud: decoder into expert order, experts, combine
    EC2MOE_CUDA(cudaStreamWaitEvent(sc, events[1 + i], 0));
    plain_next_launch();
    RelPlace rel;
    if (routed) {
      rel.counts = cnt_i;
      rel.idx = idx_i;
      rel.perm_out = perm;
      rel.offsets_out = offsets;
    }
    const void* shared_a = xa;
    long long shared_a_rows = n + T, shared_a_base = n;
    if (sub.r > 0) {
      EC2MOE_CUDA(run_codec(&sub, false, zbuf, w->V_dec, xa, sc, inv_perm, sub.n_shared > 0 ? n : -1, rel));
    } else {
      if (routed)
        EC2MOE_CUDA(launch_gather_rel(Xi, xa, idx_i, cnt_i, inv_perm, perm, offsets, sub.E, n, sub.k, sub.d, bf, sc));
      else
        EC2MOE_CUDA(launch_gather(Xi, xa, perm, n, sub.k, sub.d, bf, sc));
      shared_a = Xi;
      shared_a_rows = T;
      shared_a_base = 0;
    }
    const ExpertStage xs{xa, shared_a, shared_a_rows, shared_a_base, h, slot, shared, partial, split, direct, routed,
                         offsets, perm, inv_perm, idx_i, tw_i, Yi, n_allowed};
    EC2MOE_CUDA(run_expert_stage(&sub, w, xs, sc));
  }
  // the layer's histogram is the sum of the micro-batches' ones
  EC2MOE_CUDA(launch_sum_counts(parts, used, desc->E, counts, sc));
  EC2MOE_CUDA(cudaEventRecord(events[n_micro + 1], sc));
  EC2MOE_CUDA(cudaStreamWaitEvent(se, events[n_micro + 1], 0));
  return EC2MOE_OK;
}

ec2moe_status ec2moe_last_device_error(ec2moe_stream_t stream) {
  if (cudaStreamSynchronize(stream) != cudaSuccess) return EC2MOE_ERR_CUDA;
  unsigned int tc = 0, codec = 0, gate = 0, route = 0, swap = 0, skinny = 0, simt = 0;
  if (read_tc_error(&tc) != cudaSuccess) return EC2MOE_ERR_CUDA;
  if (read_codec_error(&codec) != cudaSuccess) return EC2MOE_ERR_CUDA;
  if (read_gate_error(&gate) != cudaSuccess) return EC2MOE_ERR_CUDA;
  if (read_route_error(&route) != cudaSuccess) return EC2MOE_ERR_CUDA;
  if (read_swap_error(&swap) != cudaSuccess) return EC2MOE_ERR_CUDA;
  if (read_skinny_error(&skinny) != cudaSuccess) return EC2MOE_ERR_CUDA;
  if (read_simt_error(&simt) != cudaSuccess) return EC2MOE_ERR_CUDA;
  // bit 0 of the GEMM, codec and gate words: a bounded wait timed out;
  // bit 1 of the GEMM words and any bit of the routing word: an index outside
  // the call's rows or experts was skipped
  if ((tc | codec | gate | swap) & 1u) return EC2MOE_ERR_TIMEOUT;
  if (((tc | swap | skinny | simt) & 2u) || route) return EC2MOE_ERR_INVALID_ARG;
  return EC2MOE_OK;
}

int32_t ec2moe_last_launch_count(void) { return launch_count(); }

ec2moe_status ec2moe_set_wait_budget(int64_t cycles) {
  if (cycles < 0) return EC2MOE_ERR_INVALID_ARG;
  set_timeout_cycles(cycles == 0 ? 0 : cycles);
  return EC2MOE_OK;
}

int64_t ec2moe_get_wait_budget(void) { return default_timeout_cycles(); }

ec2moe_status ec2moe_profile_enable(int32_t enable) {
  std::lock_guard<std::mutex> lock(g_prof_mu);
  g_prof_on = enable != 0;
  return EC2MOE_OK;
}

ec2moe_status ec2moe_profile_only(int32_t launch_index) {
  if (launch_index < -1) return EC2MOE_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lock(g_prof_mu);
  g_prof_only = launch_index;
  return EC2MOE_OK;
}

int32_t ec2moe_profile_count(void) {
  std::lock_guard<std::mutex> lock(g_prof_mu);
  return static_cast<int32_t>(g_prof.size());
}

ec2moe_status ec2moe_profile_read(int32_t i, const char** name, float* ms) {
  std::lock_guard<std::mutex> lock(g_prof_mu);
  if (i < 0 || i >= (int32_t)g_prof.size() || !name || !ms) return EC2MOE_ERR_INVALID_ARG;
  const ProfRecord& r = g_prof[i];
  if (cudaEventSynchronize(r.stop) != cudaSuccess) return EC2MOE_ERR_CUDA;
  if (cudaEventElapsedTime(ms, r.start, r.stop) != cudaSuccess) return EC2MOE_ERR_CUDA;
  *name = r.name;
  return EC2MOE_OK;
}

void ec2moe_profile_reset(void) {
  std::lock_guard<std::mutex> lock(g_prof_mu);
  g_prof.clear();
  g_pool_used = 0;
}

const char* ec2moe_status_string(ec2moe_status s) {
  switch (s) {
    case EC2MOE_OK: return "ok";
    case EC2MOE_ERR_INVALID_ARG: return "invalid argument";
    case EC2MOE_ERR_ALL_MASKED: return "all experts masked";
    case EC2MOE_ERR_TOO_FEW_EXPERTS: return "fewer allowed experts than k";
    case EC2MOE_ERR_UNSUPPORTED: return "unsupported size";
    case EC2MOE_ERR_CUDA: return "CUDA error";
    case EC2MOE_ERR_TIMEOUT: return "device wait timed out";
    case EC2MOE_ERR_WORKSPACE: return "workspace too small";
    case EC2MOE_ERR_MISALIGNED: return "misaligned pointer or pitch";
  }
  return "unknown status";
}

}  // extern "C"
