// Internal launch interfaces shared by the translation units of libec2moe.so.
// Nothing here is exported; the public ABI is include/ec2moe.h.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace ec2moe {

// Kernels enqueued by the current public call on this host thread.
void reset_launch_count();
int launch_count();

// Wraps one kernel launch: counts it and, while profiling is enabled
// (ec2moe_profile_enable), brackets it with CUDA events on its stream.
class KernelScope {
 public:
  KernelScope(const char* name, cudaStream_t s);
  ~KernelScope();
  KernelScope(const KernelScope&) = delete;
  KernelScope& operator=(const KernelScope&) = delete;

 private:
  const char* name_;
  cudaStream_t s_;
  cudaEvent_t start_ = nullptr;
};

int sm_count();

// Whether the next launch of the current public call may overlap its
// predecessor (programmatic dependent launch): every launch but the first of
// a call, unless EC2MOE_NO_PDL=1 is set in the environment.  The first launch
// keeps full stream ordering, so work the caller enqueued earlier is never
// raced.  Kernels only read data produced earlier in the stream after
// griddepcontrol.wait.
bool next_launch_pdl();
// Makes the next launch of the current call a plain one (full stream
// ordering), e.g. the first kernel on a stream after a cross-stream wait.
void plain_next_launch();

template <typename... KArgs, typename... Args>
inline cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                                 Args&&... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = next_launch_pdl() ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// cudaFuncSetAttribute(MaxDynamicSharedMemorySize) once per (device, kernel),
// raised only when a launch needs more than was set before.
cudaError_t ensure_smem_attr(const void* kernel, int bytes);

// ----------------------------------------------------------------- gate (Eq. 4-7)
struct GateArgs {
  const void* X;  // [T, d] bf16 or fp32
  const float* W_local;
  const float* b_local;
  const float* W_global;  // nullptr when K == 1
  const float* b_global;
  uint32_t mask_bits[4];  // bit e = expert e allowed (E <= 128)
  int T, d, E, K, k, renorm;
  int top_groups;  // > 0: keep only that many live groups per token (top-group pruning)
  int32_t* topk_idx;
  float* topk_w;
  // Routing fused into the gate (layer path; both nullptr: gate only): the
  // kernel fills route_counts (the per-expert histogram; cleared by the host
  // first) and route_rel[T*k] (each entry's row relative to its expert's
  // first row).  Consumers place rows at offsets[e] + route_rel[i].
  int32_t* route_counts;
  int32_t* route_rel;
  // Optional workspace of gate_split_bytes() bytes (256-byte aligned): with
  // it the tensor-core gate reads the gate rows pre-split into three bf16
  // terms by a small kernel launched first; nullptr: the gate kernel splits
  // them itself.
  void* w_split;
  // Optional workspace of gate_partial_bytes() bytes (16-byte aligned): small
  // batches then split d_model across CTAs (partial logits, then a decision
  // kernel); nullptr: the per-tile gates.
  float* gate_partial;
  // Optional, with gate_partial and T <= gate_prefetch_max_tokens(): once the
  // decision kernel knows the chosen experts, pf_units of its CTAs each
  // prefetch into L2 the first pf_row_bytes of every weight row of one
  // weight tile of the decode up projection, in the order the swapped-operand
  // GEMM's CTAs take their first tiles (launch_gemm_swap: CTA u starts with
  // unit u = (chosen expert u / (d_ff / pf_tile_rows) in id order, tile u mod
  // that), pf_tile_rows rows of W1 and, for SwiGLU, the same rows of W3).
  // Results do not depend on it.  pf_w1 == nullptr: no prefetch.
  const void* pf_w1;  // [E, d_ff, d] bf16
  const void* pf_w3;  // [E, d_ff, d] bf16, or nullptr (GELU)
  int pf_dff, pf_tile_rows, pf_units, pf_row_bytes;
};
// Largest batch whose decision kernel can prefetch the up projection's weights.
int gate_prefetch_max_tokens();
// Bytes of the prepared split gate rows (0 when the tensor-core gate does not apply).
size_t gate_split_bytes(int E, int K, int d, bool bf16);
// Bytes of the small-batch gate's partial logits (0 when that gate does not apply).
size_t gate_partial_bytes(int T, int d, int E, int K);
// Launches the gate; with the routing fields set, also fills them when the
// fused path applies (*routed = true), else gate only.  *held_sms (optional)
// receives how many SMs the gate kernel's CTAs occupy while it runs.
cudaError_t launch_gate(const GateArgs& a, bool bf16, cudaStream_t s, bool* routed = nullptr,
                        int* held_sms = nullptr);
// Rows into expert order from relative positions: for entry i (token i / k),
// pos = offsets[e] + rel[i] with offsets = exclusive prefix of counts;
// dst[pos] = src[i / k], perm[pos] = i; block 0 writes offsets[0..E].
cudaError_t launch_gather_rel(const void* src, void* dst, const int32_t* topk_idx, const int32_t* counts,
                              const int32_t* rel, int32_t* perm, int32_t* offsets, int E, long long n, int k,
                              int width, bool bf16, cudaStream_t s);

// ----------------------------------------------------------- routing tables / moves
int route_blocks(long long n_entries);  // per-block histogram blocks
cudaError_t launch_route(const int32_t* topk_idx, long long n_entries, int E, int32_t* blk_counts,
                         int32_t* counts, int32_t* offsets, int32_t* perm, int32_t* inv_perm,
                         cudaStream_t s);
// Same as launch_route, but the per-block histograms live in a fixed device
// array inside the library instead of caller memory (ec2moe_route_noalloc).
// Returns cudaErrorInvalidValue when ceil(n_entries / 1024) * E exceeds
// EC2MOE_ROUTE_NOALLOC_MAX_CELLS.
cudaError_t launch_route_noalloc(const int32_t* topk_idx, long long n_entries, int E, int32_t* counts,
                                 int32_t* offsets, int32_t* perm, int32_t* inv_perm, cudaStream_t s);
// dst[p] = src[perm[p] / k] for p < rows, width elements per row.
cudaError_t launch_gather(const void* src, void* dst, const int32_t* perm, long long rows, int k, int width,
                          bool bf16, cudaStream_t s);
// counts[e] = sum_p parts[p*E + e], p ascending.
cudaError_t launch_sum_counts(const int32_t* parts, int n_parts, int E, int32_t* counts, cudaStream_t s);
// out[row][c] = bf16(partial[0][row][c] + ... + partial[S-1][row][c]) for
// rows < `rows`, c < N (N % 4 == 0): the split-K encoder's reduce.
cudaError_t launch_splitk_sum(const float* partial, int S, long long rows, int N, void* out, cudaStream_t s);
// Split-K expert output: y[t] = sum_slot w[t*k+slot] * sum_s partial[s][pos(t, slot)]
// + sum_j shared[j*T+t], with pos = offsets[idx[i]] + rel[i] (rel_mode) or rel[i].
cudaError_t launch_splitk_combine(const float* partial, int split_k, long long part_rows, const int32_t* offsets,
                                  const int32_t* idx, const int32_t* rel, bool rel_mode, const float* w,
                                  const void* shared, int n_shared, void* Y, int T, int k, int d, cudaStream_t s);
// y[t] = sum_s slot[t*k+s] + sum_j shared[j*T+t]
cudaError_t launch_combine(const void* slot, const void* shared, int n_shared, void* Y, int T, int k, int d,
                           bool bf16, cudaStream_t s);

// ------------------------------------------------------------------ grouped GEMMs
// EPI_PARTIAL: split-K partial sums, fp32, to partial[(split * part_rows + out_row) * N + col].
enum Epi { EPI_STORE = 0, EPI_GELU = 1, EPI_SWIGLU = 2, EPI_SCATTER = 3, EPI_REPLICATE = 4, EPI_PARTIAL = 5 };

// Group g of a grouped GEMM owns rows [row0(g), row0(g) + M_g) of A and of the
// pre-scatter output, with
//   offsets != nullptr: row0 = offsets[g], M_g = offsets[g+1] - offsets[g]
//   offsets == nullptr: M_g = M, row0_out = g*M, row0_A = a_shared ? 0 : g*M
// both shifted by a_row_base / out_row_base.  Group g multiplies by rows
// [g*b_group_rows, g*b_group_rows + N) of B (and of B2 for SwiGLU).
struct GemmArgs {
  const void* A; long long a_rows;   // A [a_rows, K]
  const void* B; const void* B2; long long b_rows;  // B, B2 [b_rows, K]
  const int32_t* offsets; int G; int M; int a_shared;
  long long a_row_base, out_row_base;
  int N, K, b_group_rows;
  void* out; long long ldo;          // output pitch in elements
  const int32_t* perm;               // EPI_SCATTER: dest row = perm[out_row]
                                     // EPI_REPLICATE: dest rows perm[out_row*rep_k + s], s < rep_k
  const float* scale;                // EPI_SCATTER: multiply by scale[dest] (nullptr = 1)
  int rep_k;                         // EPI_REPLICATE: copies per row
  long long self_row_base;           // EPI_REPLICATE: also write row self_row_base + out_row (< 0: no)
  // EPI_REPLICATE with relative positions (rep_counts != nullptr): `perm`
  // holds rows relative to each expert's first row; the destination of entry
  // i is offsets[e] + perm[i] with e = rep_idx[i] and offsets the exclusive
  // prefix of rep_counts[0..rep_E); the epilogue also writes rep_perm_out[dest]
  // = i, and CTA 0 writes rep_offsets_out[0..rep_E].
  const int32_t* rep_counts;
  const int32_t* rep_idx;
  int32_t* rep_perm_out;
  int32_t* rep_offsets_out;
  int rep_E;
  long long max_rows;                // upper bound of sum_g M_g (for the grid size)
  int g_active;                      // groups expected to hold rows (tile-count estimate; 0 = G)
  long long group_rows_bound;        // upper bound of every M_g known on the host (0 = none)
  int split_k;                       // EPI_PARTIAL: K ranges per output tile (1 = none)
  float* partial;                    // EPI_PARTIAL: fp32 [split_k][part_rows][N]
  long long part_rows;
  long long timeout_cycles;          // bounded-wait budget (tensor-core path)
  const char* name;                  // label for per-launch profiling (nullptr = by epilogue)
};
cudaError_t launch_gemm_tc(const GemmArgs& a, int epi, cudaStream_t s);    // bf16, tcgen05
cudaError_t launch_gemm_simt(const GemmArgs& a, int epi, cudaStream_t s);  // fp32, CUDA cores
// bf16 groups of at most 16 rows (decode batches): weight rows streamed once
// on the CUDA cores; every epilogue but EPI_REPLICATE.
bool gemm_skinny_supported(const GemmArgs& a, int epi);
cudaError_t launch_gemm_skinny(const GemmArgs& a, int epi, cudaStream_t s);
// bf16 groups of at most SWAP_MAX_ROWS rows on the tensor cores with the
// operands swapped (weight rows on the MMA's M side, tokens on N = 16);
// every epilogue but EPI_REPLICATE.  EPI_PARTIAL needs a split_k that leaves
// no K range of 64-column blocks empty (swap_split_factor picks one).
constexpr int SWAP_MAX_ROWS = 16;
bool swap_gemm_enabled();  // false when EC2MOE_GEMM_SWAP=0 is set in the environment
bool gemm_swap_supported(const GemmArgs& a, int epi);
cudaError_t launch_gemm_swap(const GemmArgs& a, int epi, cudaStream_t s);
// Weight tiles of one group along N for the swapped kernel.
long long swap_tiles_per_group(int N, int epi);
// The K-range count (<= max_split, no empty range) whose `tiles` x ranges
// units fill whole waves of one CTA per SM best.
int swap_split_factor(long long tiles, int K, int max_split);
// Reads and clears the swapped kernel's device error word (synchronous).
cudaError_t read_swap_error(unsigned int* word);
// 2-D bf16 tensor map over a row-major [rows, cols] matrix: box 64 columns x
// box_rows rows, 128-byte swizzle, zero fill out of bounds (cached).
bool make_tensor_map_bf16(CUtensorMap* m, const void* ptr, long long rows, long long cols, int box_rows);
// 2-D fp32 tensor map, box 64 columns x box_rows rows, no swizzle (cached).
bool make_tensor_map_f32(CUtensorMap* m, const void* ptr, long long rows, long long cols, int box_rows);

// Fused low-rank codec of the layer path (bf16): Z = X V_enc^T (stored), then
// X_hat = Z V_dec^T written straight into expert order with relative
// placement (see EPI_REPLICATE's relative mode), plus the tail rows
// [self_row_base + t] when self_row_base >= 0.  Needs r in {128, 256}.
struct CodecArgs {
  const void* X;
  const void* V_enc;
  const void* V_dec;
  void* Z;        // [T, r] out
  void* out;      // expert-ordered rows, pitch d
  int T, d, r, k, E;
  const int32_t* rel;      // [T*k] rows relative to each expert's first row
  const int32_t* counts;   // [E]
  const int32_t* topk_idx; // [T*k]
  int32_t* perm_out;       // [T*k]
  int32_t* offsets_out;    // [E+1]
  long long self_row_base;
  long long timeout_cycles;
  int busy_sms;            // SMs held by the kernel this one overlaps (the gate): the grid is sized to the rest
};
bool codec_fused_supported(int d, int r);
cudaError_t launch_codec_fused(const CodecArgs& a, cudaStream_t s);
cudaError_t read_codec_error(unsigned int* word);
// Reads and clears the tensor-core gate's device error word (synchronous).
cudaError_t read_gate_error(unsigned int* word);

// Reads and clears the tensor-core kernels' device error word (synchronous).
// In the grouped-GEMM words (tensor-core, swapped, weight-streaming, SIMT)
// bit 0 is a timed-out wait and bit 1 a group range (offsets) or a scatter
// destination (perm) outside the call's rows, skipped.
cudaError_t read_tc_error(unsigned int* word);
cudaError_t read_skinny_error(unsigned int* word);
cudaError_t read_simt_error(unsigned int* word);
// Reads and clears the routing kernels' device error word (synchronous):
// nonzero when an expert id outside [0, E) or a permutation entry outside
// [0, rows) was met (and skipped).
cudaError_t read_route_error(unsigned int* word);
long long default_timeout_cycles();
void set_timeout_cycles(long long cycles);

}  // namespace ec2moe
