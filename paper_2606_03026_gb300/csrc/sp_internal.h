// sp_internal.h -- definitions shared by the translation units of
// libspikeproj.so (host launch wrappers and the kernels' parameter blocks).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "spike_proj.h"

namespace sp {

// ---------------------------------------------------------------------------
// Gather decomposition.  A work unit is (problem j, token t, output tile of
// kGatherNT channels, chunk of kGatherCK input columns), one 128-thread CTA
// each.  One warp covers one output tile of one column with 16-byte loads
// (32 lanes x 16 B = 512 B).
constexpr int kGatherNT = 512;
constexpr int kGatherCK = 512;
constexpr int kGatherWarps = 4;
constexpr int kGatherThreads = kGatherWarps * 32;

// Union decomposition: a unit is (output tile of kUnionNT, chunk of
// kUnionCK columns) for all rows of the batch.  Lanes hold 8 channels.
constexpr int kUnionNT = 256;
constexpr int kUnionCK = 256;
constexpr int kUnionWarps = 8;
constexpr int kUnionThreads = kUnionWarps * 32;

// Device error codes written to a plan's / group's error word.
enum DeviceError : int {
  kErrNone = 0,
  kErrBadUnit = 1,        // a unit index decoded outside its problem
  kErrMbarTimeout = 2,    // a bounded mbarrier wait ran out (GEMM)
  kErrTmemAlloc = 3,      // tensor-memory allocation returned an odd address
  kErrFlagTimeout = 4,    // a bounded wait for another CTA's partial ran out (GEMM)
  kErrInjected = 5,       // a test fault (spike_proj_*_inject_fault) stopped the launch
};

// Test faults armed for the next launch of a plan or group (sp_fault).
enum Fault : int {
  kFaultNone = 0,
  kFaultAbort = 1,        // the launch raises kErrInjected and leaves its output unwritten
  kFaultStall = 2,        // GEMM: one TMA copy is never issued; waits bounded by kStallWait
};
// Wait bound of a launch with kFaultStall (SM cycles, about 2 ms).
constexpr long long kStallWaitCycles = 1ll << 22;

// One projection as the gather kernel sees it.
struct GatherProblem {
  const int8_t* W;        // column-major, W[k*ldw + m]
  const float* scale;     // [N]
  int32_t ldw;
  int32_t N;
  int32_t K;
  int32_t unit_begin;     // prefix sum of units_per_token over problems
  int32_t ws_begin;       // prefix sum of N (int32 elements of workspace)
  int32_t ticket_begin;   // prefix sum of output tiles
  // cluster form (set by the launcher): a cluster of kGatherCluster CTAs
  // holds tpc output tiles x kch column chunks of ck columns; ncl clusters
  int32_t ck, kch, tpc, ncl;
};

// Cluster form of the gather (one token per problem): clusters of 6 CTAs of
// 256 threads; a CTA sums chunks of at most 1024 columns.
constexpr int kGatherCluster = 6;
constexpr int kGatherClusterWarps = 8;
constexpr int kGatherClusterThreads = 32 * kGatherClusterWarps;
constexpr int kGatherClusterMaxCK = 1024;
constexpr int kGatherMaxClusterList = 256;   // clusters of a launch listed one by one

constexpr int kMaxProblems = SPIKE_PROJ_MAX_GROUP;

// Kernel parameters of one gather launch, passed by value (__grid_constant__):
// NP = 1 for single-plan calls, kMaxProblems for groups.
template <int NP>
struct GatherParamsT {
  GatherProblem prob[NP];
  int32_t nprob;
  int32_t B;              // tokens per problem (1 for groups)
  int32_t units_total;    // B * sum_j units_per_token(j)
  int32_t max_units;      // largest units_per_token(j): grid.x = B * max_units
  int32_t fmt;            // sp_fmt
  const void* spikes;     // row (j*B + t) at spikes + row*ld_spikes elements
  int64_t ld_spikes;
  int32_t* acc;           // row (j*B + t) at acc + row*ld_out (may be null)
  float* y;               // idem (may be null)
  int64_t ld_out;
  int32_t* ws;            // problem j token t: ws + (ws_begin_j*B + t*N_j); the gather kernel adds fp32 into it
  uint32_t* tickets;      // problem j token t tile n: ticket_begin_j*B + t*ntile_j + n
  int* err;
  // cluster form: cluster c of a 1-D grid is cluster (cl_list[c] & 0xff) of
  // problem (cl_list[c] >> 8); ncl_list == 0: grid (clusters x 6, problems)
  int32_t ncl_list;
  uint16_t cl_list[kGatherMaxClusterList];
  // fused spike producer (cluster form only): when lif_I is set, problem j's
  // spike row is made inside the kernel by one LIF step of row j of
  // (lif_vin, lif_I); the new state goes to lif_vout (and the spike words to
  // lif_bits when set), each element by exactly one CTA
  int32_t fault = 0;      // Fault armed for this launch (kFaultAbort)
  const float* lif_vin = nullptr;
  float* lif_vout = nullptr;
  const float* lif_I = nullptr;
  int64_t lif_ld = 0;
  float lif_beta = 0.f, lif_theta = 0.f;
  uint32_t* lif_bits = nullptr;
  int64_t lif_ld_bits = 0;
};
using GatherParams1 = GatherParamsT<1>;
using GatherParamsG = GatherParamsT<kMaxProblems>;

inline __host__ __device__ int ceil_div(int a, int b) { return (a + b - 1) / b; }
inline __host__ __device__ int gather_ntiles(int N) { return ceil_div(N, kGatherNT); }
inline __host__ __device__ int gather_kchunks(int K) { return ceil_div(K, kGatherCK); }
inline __host__ __device__ int gather_units(int N, int K) {
  return gather_ntiles(N) * gather_kchunks(K);
}

struct UnionParams {
  const int8_t* W;
  const float* scale;
  int32_t ldw, N, K, B;
  int32_t fmt;
  const void* spikes;
  int64_t ld_spikes;
  int32_t* acc;
  float* y;
  int32_t* ws;            // [B][N]
  uint32_t* tickets;      // [ceil(N/kUnionNT)]
  int* err;
  int32_t fault;          // Fault armed for this launch (kFaultAbort)
};
constexpr int kUnionMaxRows = 256;      // rows per union launch

// Tensor-core (tcgen05) prefill GEMM operands.
struct GemmParams {
  const float* scale;
  int32_t* acc;           // [T][N] or null
  float* y;               // [T][N] or null
  int32_t T, N, K;
  int* err;
  float* part;            // split-K partials, part_units x (128 x 256) fp32
  int32_t part_units;
  int32_t fault;          // Fault armed for this launch
};

// One continuous-input projection as the dense kernel sees it (row-major
// INT8 weights, FP32 activations; see spike_proj_dense).
struct DenseProblem {
  const int8_t* W;
  int64_t ldw;
  const float* scale;
  const float* x;
  int64_t ldx;
  float* y;
  int64_t ldy;
  int32_t N, K;
};
constexpr int kDenseMaxProblems = SPIKE_PROJ_DENSE_MAX_GROUP;
cudaError_t launch_dense(const DenseProblem* probs, int count, int B, cudaStream_t s);

// One LIF step of `rows` layers of K neurons into BITS32 spike rows (see
// spike_proj_lif).
cudaError_t launch_lif(float* v, const float* I, int K, int rows, int64_t ld, float beta,
                       float theta, uint32_t* bits, int64_t ld_bits, cudaStream_t s);
// The same for rows <= kMaxProblems rows of Ks[r] neurons each, the state read
// from vin and written to vout (which may equal vin).
cudaError_t launch_lif_rows(const float* vin, float* vout, const float* I, const int32_t* Ks,
                            int rows, int64_t ld, float beta, float theta, uint32_t* bits,
                            int64_t ld_bits, cudaStream_t s);

// One vocabulary-head call (see spike_proj_head); ws is the head's workspace
// of head_workspace_bytes(), zero when created (the kernels leave it so).
struct HeadArgs {
  const int8_t* W;
  int64_t ldw;
  const float* scale;
  int32_t V, K;
  const float* h;
  int64_t ldh;
  int32_t B;
  float tau;
  int32_t k_sel;
  int32_t* token;
  int32_t* verified;
  float* gap;
  int32_t* cand;
  float* r;
  float* z;
  int64_t ld_z;
  void* ws;
};
size_t head_workspace_bytes();
cudaError_t launch_head(const HeadArgs& a, cudaStream_t s);

// Launches `kernel` with programmatic stream serialization: its blocks may
// become resident while the previous kernel of the stream is still running
// and wait for it in pdl_wait (see sp_ptx.cuh) before touching memory.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr.val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// Measurement aid (sp_probe.cu): reads count pieces of piece_bytes (512, 1024
// or 1536) at base + 16 * offsets16[i], XOR of every word into *sink.
cudaError_t launch_probe_gather(const uint8_t* base, const uint32_t* offsets16, int count,
                                int piece_bytes, uint32_t* sink, cudaStream_t s);

// ---------------------------------------------------------------------------
// Host launch wrappers (defined next to their kernels).  Each returns the
// cudaError_t of the launch.
cudaError_t launch_gather(const GatherParams1& p, cudaStream_t s);
cudaError_t launch_gather(const GatherParamsG& p, cudaStream_t s);
cudaError_t launch_union(const UnionParams& p, cudaStream_t s);
// Counts active spikes: out[0] = sum over the B rows of |A_t| (out[1] unused).
cudaError_t launch_density(const void* spikes, int fmt, int64_t ld, int B, int K,
                           int32_t* out, cudaStream_t s);
// Spike rows in any format -> bytes 0 / 1 [T][Kp] (zero past K).
cudaError_t launch_spikes_to_01(const void* spikes, int fmt, int64_t ld, int T, int K, int Kp,
                                uint8_t* Xs, cudaStream_t s);

}  // namespace sp
