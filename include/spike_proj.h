/*
 * spike_proj.h -- C ABI of libspikeproj.so: the spike-gated INT8 projection
 * on NVIDIA GB300 (sm_103a).
 *
 * Operation (Section 2.3, Eq. (sparse); Section 2.2 for the layout):
 *
 *     A     = { k : x_k = 1 }                 active columns of one spike row
 *     acc_m = sum_{k in A} Q_{m,k}            INT32, exact
 *     y_m   = s_m * (float)acc_m              one FP32 multiply, round to
 *                                             nearest even, per output m
 *
 *   Q   INT8 weights of N outputs by K inputs, COLUMN-MAJOR: element (m, k)
 *       at W[k * ldw + m], so each active column is one contiguous read of N
 *       bytes across the output channels (Section 2.2).
 *   s   FP32 scale per output channel, length N (Section 2.3 quantiser).
 *   x   binary spikes, one row per token, in one of three formats (sp_fmt).
 *
 * Only the active columns are read on the gather paths; the dense
 * tensor-core path (SP_GEMM) reads all of Q and is chosen only where the
 * measured density makes that cheaper.  Every path produces the same INT32
 * accumulators bit for bit, and therefore the same FP32 outputs.
 *
 * Around the projection the library also has the paper's continuous-input
 * projection (spike_proj_dense: row-major INT8 weights, FP32 activations),
 * a spike producer (spike_proj_lif, and spike_proj_group_decode_lif with the
 * producer inside the decode launch), and the vocabulary head with INT8
 * activations and FP32 recomputation of the top candidates (spike_proj_head,
 * Section 5).  Each is documented at its declaration below.
 *
 * Conventions for every call
 *   - Pointers named d_* or documented as "device" are CUDA device pointers
 *     on the current device; the caller owns them.  A plan BORROWS W and the
 *     scale: they must stay allocated and unchanged while the plan lives.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = the legacy
 *     default stream) unless documented otherwise.  Argument errors are
 *     detected on the host and returned before anything is enqueued.
 *   - Nothing aborts, traps or spins without bound.  Kernel-side failures set
 *     an error word read by spike_proj_plan_status / spike_proj_group_status.
 *   - A plan or group owns workspace that its kernels leave zeroed for the
 *     next call; calls on one plan (or group) must not overlap on the GPU:
 *     use one stream per plan, or order the streams.
 *   - Exactness bound: |acc| <= 128 * K must stay below 2^24 so that the
 *     INT32 -> FP32 conversion is exact on every path; hence K <= 131072.
 */
#ifndef SPIKE_PROJ_H
#define SPIKE_PROJ_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SPIKE_PROJ_ABI_VERSION 1
#define SPIKE_PROJ_MAX_K 131072        /* 128 * K < 2^24: exact FP32 conversion */
#define SPIKE_PROJ_MAX_GROUP 64        /* projections per group */
#define SPIKE_PROJ_NOALLOC_MAX_N 32768 /* largest N of spike_proj_decode_noalloc */
#define SPIKE_PROJ_DENSE_MAX_B 4       /* activation rows per spike_proj_dense call */
#define SPIKE_PROJ_DENSE_MAX_GROUP 128 /* problems per spike_proj_dense call */
#define SPIKE_PROJ_HEAD_MAX_B 4        /* hidden states per spike_proj_head call */
#define SPIKE_PROJ_HEAD_MAX_CAND 64    /* largest k_sel of spike_proj_head */
#define SPIKE_PROJ_HEAD_MAX_K 8192     /* largest hidden width of a head */
#define SPIKE_PROJ_HEAD_MAX_V (1 << 26) /* largest vocabulary of a head */

typedef struct sp_plan_s *sp_plan_t;
typedef struct sp_group_s *sp_group_t;
typedef struct sp_head_s *sp_head_t;
typedef void *sp_stream_t;             /* a cudaStream_t */

typedef enum sp_status {
    SP_OK = 0,
    SP_EINVAL = 1,        /* NULL where required, size out of range, bad enum */
    SP_EALIGN = 2,        /* pointer / leading dimension breaks an alignment rule */
    SP_EDEVICE = 3,       /* current device is not compute capability 10.3 */
    SP_ECUDA = 4,         /* a CUDA runtime call failed: spike_proj_last_cuda_error() */
    SP_ENOMEM = 5,        /* workspace allocation failed */
    SP_ERANGE = 6,        /* K above SPIKE_PROJ_MAX_K, or batch above the plan's max */
    SP_EKERNEL = 7,       /* a kernel raised the device error word */
    SP_EUNSUPPORTED = 8,  /* strategy not available for this plan (e.g. SP_GEMM
                             without SP_PLAN_GEMM) */
    SP_ESCRATCH = 9       /* N above SPIKE_PROJ_NOALLOC_MAX_N: the fixed scratch
                             of spike_proj_decode_noalloc is too small */
} sp_status;

/* Spike row formats.
 *   SP_SPIKES_BITS32: uint32 words; column k is bit (k % 32) of word (k / 32),
 *                     least significant bit first; bits at or past K are
 *                     ignored.  A row holds ceil(K/32) words; row stride
 *                     (ld_spikes) is counted in words.
 *   SP_SPIKES_U8:     one byte per column, any nonzero byte is a spike; row
 *                     stride counted in bytes.
 *   SP_SPIKES_BOOL8:  one byte per column holding exactly 0 or 1 (the bytes
 *                     of a C bool array or a torch.bool tensor); row stride
 *                     counted in bytes.  Every path accepts it; SP_GEMM reads
 *                     such rows in place when the base is 16-byte aligned and
 *                     the row stride a multiple of 16 (other formats go
 *                     through a 0/1 staging pass first).  A byte other than 0
 *                     or 1 gives an unspecified result on that path (no
 *                     fault); the gather and union paths treat it as U8. */
typedef enum sp_fmt {
    SP_SPIKES_BITS32 = 0,
    SP_SPIKES_U8 = 1,
    SP_SPIKES_BOOL8 = 2
} sp_fmt;

/* Kernel strategies for multi-token calls.
 *   SP_AUTO    count the active spikes on the device, read the count back
 *              (one stream synchronisation) and pick SP_GATHER or, on a plan
 *              made with SP_PLAN_GEMM, SP_GEMM when its modelled time is
 *              lower (large batches and dense prefill).
 *   SP_GATHER  per-token active-column gather (the batch-1 kernel per row).
 *   SP_UNION   one fetch of each column in the union of the rows' active sets,
 *              added into every row whose spike is set.
 *   SP_GEMM    dense tensor-core contraction over all columns (tcgen05
 *              e4m3 x e4m3 with fp32 accumulation in tensor memory: spike
 *              bytes 0 / 1 read as 0 and 2^-9, each weight split into two
 *              e4m3-exact planes 16 h + l; exact because every partial sum
 *              is a multiple of 2^-9 with at most 24 significant bits). */
typedef enum sp_kernel {
    SP_AUTO = 0,
    SP_GATHER = 1,
    SP_UNION = 2,
    SP_GEMM = 3
} sp_kernel;

/* Plan flags. */
#define SP_PLAN_GEMM 0x1u  /* also build the tensor-core operand copy of W:
                              two e4m3 planes, 2*N*Kp bytes (Kp = K rounded up
                              to a multiple of 64), owned by the plan */

/* ---------------------------------------------------------------------------
 * spike_proj_plan -- describe one projection and allocate its workspace.
 *
 *   plan       out: the new plan (unchanged on error).
 *   W          device, INT8, column-major: W[k*ldw + m] for m < N, k < K.
 *              16-byte aligned.  Borrowed.
 *   ldw        leading dimension in bytes (elements): ldw >= N, ldw % 16 == 0.
 *   scale      device, FP32 [N], one scale per OUTPUT channel m (not per
 *              input column: a [K]-long scale is a layout error the caller
 *              must not make; Appendix A.2 records that defect).  4-byte
 *              aligned.  Borrowed.
 *   N          output channels, 16 <= N, N % 16 == 0.
 *   K          input columns, 1 <= K <= SPIKE_PROJ_MAX_K (else SP_ERANGE).
 *   max_batch  largest B / T accepted by spike_proj_batched / _prefill on this
 *              plan (>= 1; sizes the workspace: 4*N*max_batch bytes, plus
 *              Kp*ceil(max_batch/128)*128 bytes of 0/1 spike staging with
 *              SP_PLAN_GEMM).
 *   flags      0 or SP_PLAN_GEMM.
 *   stream     used for the workspace clear and the operand copy; the call
 *              synchronises it before returning.
 * Errors: SP_EINVAL, SP_EALIGN, SP_ERANGE, SP_EDEVICE, SP_ENOMEM, SP_ECUDA.
 * ------------------------------------------------------------------------- */
sp_status spike_proj_plan(sp_plan_t *plan, const int8_t *W, int64_t ldw,
                          const float *scale, int32_t N, int32_t K,
                          int32_t max_batch, uint32_t flags, sp_stream_t stream);

/* Frees the plan's workspace (synchronises the device).  NULL is a no-op. */
sp_status spike_proj_plan_destroy(sp_plan_t plan);

/* ---------------------------------------------------------------------------
 * spike_proj_decode -- one spike row (batch 1), Eq. (sparse).
 *
 *   spikes  device, one row in `fmt` (ceil(K/32) words or K bytes); 4-byte
 *           aligned for SP_SPIKES_BITS32.
 *   acc     device INT32 [N] or NULL; y device FP32 [N] or NULL (not both
 *           NULL).  4-byte aligned.
 * Compacts the row into its active-column list on the device (warp ballot and
 * popcount) and sums only those columns.  Never reads an inactive column.
 * ------------------------------------------------------------------------- */
sp_status spike_proj_decode(sp_plan_t plan, const void *spikes, sp_fmt fmt,
                            int32_t *acc, float *y, sp_stream_t stream);

/* ---------------------------------------------------------------------------
 * spike_proj_batched -- B independent spike rows sharing the plan's W.
 *
 *   spikes     device, B rows, row b at spikes + b*ld_spikes (words for
 *              BITS32, bytes for U8 and BOOL8); ld_spikes >= ceil(K/32) or
 *              >= K.
 *   B          1 <= B <= plan's max_batch (else SP_ERANGE).
 *   acc, y     device [B][N] row-major (either may be NULL, not both).
 *   strategy   SP_AUTO, SP_GATHER, SP_UNION or SP_GEMM (SP_GEMM needs a plan
 *              made with SP_PLAN_GEMM, else SP_EUNSUPPORTED).
 * Row b of the result equals spike_proj_decode on row b, bit for bit.
 * ------------------------------------------------------------------------- */
sp_status spike_proj_batched(sp_plan_t plan, const void *spikes, sp_fmt fmt,
                             int32_t B, int64_t ld_spikes, int32_t *acc,
                             float *y, sp_kernel strategy, sp_stream_t stream);

/* ---------------------------------------------------------------------------
 * spike_proj_prefill -- T prompt tokens at once: ACC = X Q^T, Y = ACC * s
 * per column (Eq. (sparse) for every row of X).
 *
 *   X          device, uint8 [T][ldx] with X[t][k] nonzero = spike; ldx >= K.
 *   T          1 <= T <= plan's max_batch.
 *   acc, y     device [T][N] row-major (either may be NULL, not both).
 *   strategy   as for spike_proj_batched; SP_AUTO picks SP_GEMM on a plan
 *              with SP_PLAN_GEMM when the measured density makes the dense
 *              contraction cheaper than the gathers.
 * On SP_GEMM these rows first go through the 0/1 staging pass (any nonzero
 * byte fires); rows already holding exactly 0 / 1 (a torch.bool tensor) can
 * skip it: spike_proj_batched with SP_SPIKES_BOOL8 reads them in place.
 * ------------------------------------------------------------------------- */
sp_status spike_proj_prefill(sp_plan_t plan, const uint8_t *X, int32_t T,
                             int64_t ldx, int32_t *acc, float *y,
                             sp_kernel strategy, sp_stream_t stream);

/* Strategy and total active count (sum over rows of |A|) of the last
 * batched / prefill call with SP_AUTO on this plan; the count is -1 when the
 * last call did not measure it. */
sp_status spike_proj_last_dispatch(sp_plan_t plan, sp_kernel *chosen,
                                   int32_t *active_count);

/* Reads and clears the plan's device error word; synchronises `stream`.
 * Returns SP_EKERNEL if a kernel raised it (and re-zeroes the workspace),
 * SP_OK otherwise. */
sp_status spike_proj_plan_status(sp_plan_t plan, sp_stream_t stream);

/* ---------------------------------------------------------------------------
 * Groups: several independent batch-1 projections in ONE kernel launch, e.g.
 * the 44 binary-input projections of one 22-block decode step (per block,
 * the sequence mixer's TCAM projection and the FFN's down projection,
 * Section 2.1).  All projections of a group run concurrently, so their combined
 * active-column traffic can fill the memory system.
 *
 * spike_proj_group_create: plans[0..count) (1 <= count <= SPIKE_PROJ_MAX_GROUP)
 *   are borrowed and must outlive the group.  The group owns its own
 *   workspace (the plans' workspaces are not used by group calls).
 * ------------------------------------------------------------------------- */
sp_status spike_proj_group_create(sp_group_t *group, const sp_plan_t *plans,
                                  int32_t count, sp_stream_t stream);
sp_status spike_proj_group_destroy(sp_group_t group);

/* spike_proj_group_decode: projection j reads its spike row at
 *   spikes + j*ld_spikes   (words for BITS32, bytes for U8 and BOOL8)
 * and writes acc + j*ld_out, y + j*ld_out (device; either may be NULL, not
 * both).  ld_spikes must cover the largest K of the group; ld_out >= the
 * largest N. */
sp_status spike_proj_group_decode(sp_group_t group, const void *spikes,
                                  sp_fmt fmt, int64_t ld_spikes, int32_t *acc,
                                  float *y, int64_t ld_out, sp_stream_t stream);

/* spike_proj_group_prefill: T spike rows per member through the dense
 * tensor-core contraction of spike_proj_prefill (SP_GEMM), ACC_j = X_j Q_j^T
 * and Y_j = ACC_j * s_j per column (Eq. (sparse) for every row, Section 3.2's
 * 512-token prefill), for EVERY member of the group in ONE persistent launch:
 * the output tiles of all members (128 rows x 256 channels each) are shared
 * out over the SMs, and each tile runs over its whole K.  The members are
 * independent; nothing of member j reaches member i.  Results equal
 * spike_proj_prefill / spike_proj_batched on each member's plan, bit for bit.
 *
 *   X     host array of `count` device pointers; member j's rows at
 *         X[j] + t*ldx (t < T; words for BITS32, bytes for U8 and BOOL8).
 *         BOOL8 rows with a 16-byte aligned base and ldx % 16 == 0 are read
 *         in place; other rows go first through a 0/1 staging pass into the
 *         member plan's staging copy (one small launch per member).
 *   T     1 <= T <= every member plan's max_batch (else SP_ERANGE).
 *   ldx   row stride; ldx >= ceil(K_j/32) words (BITS32) or K_j bytes.
 *   acc   host array of `count` device pointers, member j's INT32 [T][N_j]
 *         row-major at acc[j], or NULL for no acc;
 *   y     likewise FP32 [T][N_j] (acc and y not both NULL).
 * Every member plan must have been made with SP_PLAN_GEMM (else
 * SP_EUNSUPPORTED).  The group's error word records a kernel fault
 * (spike_proj_group_status).  Errors: SP_EINVAL, SP_EALIGN, SP_ERANGE,
 * SP_EUNSUPPORTED, SP_ENOMEM (the member table, allocated on the host by the
 * first call), SP_ECUDA. */
sp_status spike_proj_group_prefill(sp_group_t group, const void *const *X,
                                   sp_fmt fmt, int32_t T, int64_t ldx,
                                   int32_t *const *acc, float *const *y,
                                   sp_stream_t stream);

/* spike_proj_group_decode_host: the same with HOST buffers.  Page-locked
 * buffers (cudaHostAlloc, cudaHostRegister, torch pin_memory) are read and
 * written by the kernel in place, over the CPU-GPU link, with no copy; for
 * pageable buffers the call enqueues the copy of count rows of spikes into
 * group-owned device staging, the kernel, and the copies of acc / y back.
 * Returns once enqueued; the host buffers must not be touched until `stream`
 * has been synchronised.  Errors as spike_proj_group_decode (SP_EALIGN for a
 * spike word or output pointer that is not 4-byte aligned). */
sp_status spike_proj_group_decode_host(sp_group_t group, const void *h_spikes,
                                       sp_fmt fmt, int64_t ld_spikes,
                                       int32_t *h_acc, float *h_y,
                                       int64_t ld_out, sp_stream_t stream);

/* spike_proj_group_decode_lif: the decode step with its spike producer
 * fused in.  Projection j's spike row is made by one LIF step (the reading
 * spike_proj_lif states) of row j of the state and current, inside the same
 * launch that projects it:
 *
 *     u = fmaf(beta, v_in[j][k], I[j][k]);  x_k = (u >= theta);
 *     v_out[j][k] = x_k ? u - theta : u;    y_j = s ⊙ (Q_j x)     (k < K_j)
 *
 * so the step needs one launch instead of producer + decode.  Results equal
 * spike_proj_lif on a copy of v_in followed by spike_proj_group_decode on its
 * bits, bit for bit.
 *
 *   v_in, I  device FP32, row j at + j*ld (ld >= the largest K); read only.
 *   v_out    device FP32, same layout; elements k < K_j of row j are written,
 *            the rest untouched.  Must not overlap v_in or I (swap two state
 *            buffers from step to step).
 *   bits     NULL, or device uint32 rows at bits + j*ld_bits (ld_bits >=
 *            ceil(largest K / 32)) that receive row j's ceil(K_j/32) spike
 *            words (bits past K_j zero); must not overlap the other buffers.
 *   acc, y, ld_out  as spike_proj_group_decode.
 * All of v_in, v_out, I, bits 4-byte aligned (SP_EALIGN).  The fused form
 * needs every K_j <= 6144 and the group's tiles resident at once; otherwise
 * the call runs the producer and the decode as two launches, same results. */
sp_status spike_proj_group_decode_lif(sp_group_t group, const float *v_in,
                                      float *v_out, const float *I, int64_t ld,
                                      float beta, float theta, uint32_t *bits,
                                      int64_t ld_bits, int32_t *acc, float *y,
                                      int64_t ld_out, sp_stream_t stream);

/* Reads and clears the group's device error word (synchronises `stream`). */
sp_status spike_proj_group_status(sp_group_t group, sp_stream_t stream);

/* ---------------------------------------------------------------------------
 * spike_proj_decode_noalloc -- a batch-1 decode with the same result as
 * spike_proj_decode, that allocates no memory at all.  The paper has no
 * counterpart: this is a library convenience, not part of the method.
 *
 * Who needs it: callers that may not allocate device memory on their decode
 * path -- a serving loop where cudaMalloc / cudaFree would synchronise the
 * device and stall every other stream, a process whose device memory is
 * already handed out in full by another allocator, or code that has no place
 * to keep a plan handle and free it later.  It takes the projection's
 * arguments directly (no plan) and gives the same bits as
 * spike_proj_decode on a plan of the same W, scale, N and K.
 *
 * Scratch: the split-K workspace and tile tickets live in one fixed array of
 * static device memory inside the library (128 KiB + 256 bytes per device:
 * SPIKE_PROJ_NOALLOC_MAX_N INT32 words plus one word per 512 outputs), so N is
 * limited to SPIKE_PROJ_NOALLOC_MAX_N; a larger N returns SP_ESCRATCH before
 * anything is enqueued.  No cudaMalloc, cudaFree or other allocating call is
 * made, on the first call or later.  The kernel it runs returns the scratch
 * to zero, so nothing has to be cleared between calls.  Its only wait is
 * bounded (about a second, for the partial sums of the other CTAs of its
 * thread-block cluster); should that wait ever run out, acc and y are left
 * unwritten and nothing reports it: this entry point has no status word.
 *
 * First call per device: it checks the device, looks up the scratch address
 * on the current device, clears the scratch on `stream` (defensively: it is
 * zero when the library loads) and synchronises that stream.  Make the first
 * call on each device before any stream capture begins; later calls on that
 * device only enqueue the kernel.  The address is kept for the life of the
 * process: after cudaDeviceReset do not call this entry point again.
 *
 * Concurrency: every call on one device shares the one scratch, whatever its
 * W.  Calls whose kernels can overlap on the GPU race on it and give wrong
 * results: issue them on one stream, or order the streams.
 *
 *   W, ldw, scale, N, K   as for spike_proj_plan (W, scale borrowed for the
 *                         duration of the call); N <= SPIKE_PROJ_NOALLOC_MAX_N.
 *   spikes, fmt, acc, y   as for spike_proj_decode.
 * Errors: SP_EINVAL, SP_EALIGN, SP_ERANGE, SP_ESCRATCH, SP_EDEVICE, SP_ECUDA.
 * ------------------------------------------------------------------------- */
sp_status spike_proj_decode_noalloc(const int8_t *W, int64_t ldw,
                                    const float *scale, int32_t N, int32_t K,
                                    const void *spikes, sp_fmt fmt,
                                    int32_t *acc, float *y,
                                    sp_stream_t stream);

/* ---------------------------------------------------------------------------
 * Continuous-input projections: the paper's other kernel (Section 2.3: for
 * continuous inputs the INT8 weights are converted to FP32, multiplied with
 * the FP32 activations and accumulated, and the row scale is applied after;
 * Section 2.2: these projections keep ROW-MAJOR weights, one contiguous dot
 * product per output).  For each problem and each activation row b < B:
 *
 *     y[b*ldy + m] = s_m * sum_{k<K} float(W[m*ldw + k]) * x[b*ldx + k]
 *
 * computed in FP32: each lane of a warp accumulates the products of its
 * 16-column chunks (columns 16 l .. 16 l + 15 of every 512) with fmaf in
 * ascending k, the 32 lane sums meet in a 5-level butterfly, and one FP32
 * multiply applies s_m.  Each y is thus the FP32 value of a fixed summation
 * tree of depth d <= 16 * ceil(K / 512) + 5, identical on every run, with
 * |y - s_m * exact| <= |s_m| * gamma(d) * sum_k |W x| + u |y| (u = 2^-24,
 * gamma(d) = d u / (1 - d u)).  Weights are read once per call for all B rows.
 *
 *   problems[j]  one projection (fields below); count in 1 ..
 *                SPIKE_PROJ_DENSE_MAX_GROUP.  All run in ONE kernel launch.
 *   B            activation rows, 1 .. SPIKE_PROJ_DENSE_MAX_B.
 * Fields of sp_dense (device pointers, caller-owned, not retained):
 *   W      INT8 row-major, element (m, k) at W[m*ldw + k]; 16-byte aligned;
 *          ldw >= K, ldw % 16 == 0 (bytes past K in a row are never used).
 *   scale  FP32 [N], one per output row; 4-byte aligned.
 *   x      FP32, row b at x + b*ldx; 16-byte aligned; ldx >= K, ldx % 4 == 0.
 *   y      FP32, row b at y + b*ldy; 4-byte aligned; ldy >= N.  Must not
 *          overlap W, scale, x or another problem's y.
 *   N, K   1 <= N; 1 <= K <= SPIKE_PROJ_MAX_K.
 * Errors: SP_EINVAL, SP_EALIGN, SP_ERANGE, SP_EDEVICE, SP_ECUDA (nothing is
 * enqueued on an error).  The kernel cannot fail once launched.
 * ------------------------------------------------------------------------- */
/* ---------------------------------------------------------------------------
 * spike_proj_lif -- spike producer: one leaky integrate-and-fire step for
 * `rows` layers of K neurons, written straight into SP_SPIKES_BITS32 rows
 * (what spike_proj_decode, _group_decode and _batched read).  The paper names
 * LIF dynamics (Section 1) without giving the update; this is the reading:
 *
 *     v <- fmaf(beta, v, I);   x = (v >= theta);   v <- v - theta where x
 *
 * FP32 IEEE operations throughout (no flush of subnormals), so v and the bits
 * equal the definition's exactly, on every run (a NaN state stays NaN and
 * never fires; its payload is not preserved).
 *
 *   v        device FP32, row r at v + r*ld, updated in place; 4-byte aligned.
 *   I        device FP32 input current, row r at I + r*ld; 4-byte aligned.
 *   K        neurons per row, 1 <= K <= SPIKE_PROJ_MAX_K; ld >= K.
 *   rows     1 <= rows.
 *   bits     device uint32, row r at bits + r*ld_bits, ld_bits >= ceil(K/32);
 *            4-byte aligned; bits at or past K are written 0.  Must not
 *            overlap v or I.
 * Errors: SP_EINVAL, SP_EALIGN, SP_ERANGE, SP_EDEVICE, SP_ECUDA.
 * ------------------------------------------------------------------------- */
sp_status spike_proj_lif(float *v, const float *I, int32_t K, int32_t rows,
                         int64_t ld, float beta, float theta, uint32_t *bits,
                         int64_t ld_bits, sp_stream_t stream);

typedef struct sp_dense {
    const int8_t *W;
    int64_t ldw;
    const float *scale;
    const float *x;
    int64_t ldx;
    float *y;
    int64_t ldy;
    int32_t N;
    int32_t K;
} sp_dense;

sp_status spike_proj_dense(const sp_dense *problems, int32_t count, int32_t B,
                           sp_stream_t stream);

/* ---------------------------------------------------------------------------
 * Vocabulary head with INT8 activations and candidate-row verification
 * (Section 5, trace configuration; Appendix D).  The head's weights are a
 * continuous-input projection: W ROW-MAJOR INT8, row m (one vocabulary slot)
 * at W + m*ldw, K bytes used, with one FP32 scale per row.  For each hidden
 * state h, in ONE kernel launch:
 *
 *   1. INT8 activations (the paper does not state the activation quantiser;
 *      this reads it as the weight rule of Section 2.3 applied to h):
 *        s_x = max(max_k |h_k|, 1e-8) / 127,  q_k = clip(rint(h_k / s_x), +-127)
 *   2. approximate logits z_m = s_m * (s_x * float(sum_k W[m][k] q_k))
 *      (exact integer sum, two FP32 multiplies)
 *   3. rows ordered by z descending, equal z by lower row;
 *      gap = z_(1) - z_(2) (FP32)
 *   4. the gate: verification when gap < tau (0.5 in the paper's trace
 *      configuration, 4.0 in its power configuration)
 *   5. the first k_sel rows of the order (the candidates) recomputed with the
 *      FP32 activations: r_m = s_m * sum_k float(W[m][k]) h_k
 *   6. token = the candidate with the largest r (equal r: lower row) when
 *      verified, else the first row of the order.
 *
 * z, the gap, the gate decision and the candidates equal the definition's
 * bit for bit; r is an FP32 sum of K products of depth <= 16*ceil(K/512) + 5
 * (the bound of spike_proj_dense).  The weights are read once per call (the
 * call is HBM-bound on V*K bytes).
 *
 * spike_proj_head_create: W device, 16-byte aligned, ldw >= K with
 *   ldw % 16 == 0 (SP_EALIGN); scale device FP32 [V], 4-byte aligned;
 *   2 <= V <= SPIKE_PROJ_HEAD_MAX_V, 1 <= K <= SPIKE_PROJ_HEAD_MAX_K
 *   (SP_ERANGE).  W and scale are borrowed and must outlive the head, which
 *   owns a 3 MiB workspace.  A head serves one stream at a time.
 * ------------------------------------------------------------------------- */
sp_status spike_proj_head_create(sp_head_t *head, const int8_t *W, int64_t ldw,
                                 const float *scale, int32_t V, int32_t K,
                                 sp_stream_t stream);
sp_status spike_proj_head_destroy(sp_head_t head);

/* spike_proj_head: B hidden states (1 .. SPIKE_PROJ_HEAD_MAX_B), row b at
 * h + b*ldh (device FP32, h 16-byte aligned, ldh >= K with ldh % 4 == 0,
 * else SP_EALIGN / SP_EINVAL); 1 <= k_sel <= min(V, SPIKE_PROJ_HEAD_MAX_CAND).
 * Outputs, device, 4-byte aligned, row b of each:
 *   token     int32 [B] (required)
 *   verified  int32 [B]: 1 when the gate opened (may be NULL)
 *   gap       FP32 [B] (may be NULL)
 *   cand      int32 [B][k_sel]: the candidate rows in order (may be NULL)
 *   r         FP32 [B][k_sel]: their recomputed logits, written only for
 *             the rows whose gate opened (may be NULL)
 *   z         FP32 rows at z + b*ld_z, ld_z >= V: the approximate logits
 *             (may be NULL)
 * A tau of +inf always verifies, 0 or NaN never does.  Non-finite h gives
 * unspecified (but in-range) results. */
sp_status spike_proj_head(sp_head_t head, const float *h, int64_t ldh, int32_t B,
                          float tau, int32_t k_sel, int32_t *token,
                          int32_t *verified, float *gap, int32_t *cand, float *r,
                          float *z, int64_t ld_z, sp_stream_t stream);

/* ---------------------------------------------------------------------------
 * Test faults -- FOR TESTS OF THE ERROR PATH ONLY (the paper has no
 * counterpart).  A fault armed on a plan or group applies to the next kernel
 * launch of that plan or group (any decode, batched, prefill or group call;
 * the argument checks come first) and is then disarmed:
 *   SP_FAULT_ABORT  the launch raises the device error word and returns
 *                   without writing its outputs and without cleaning its
 *                   workspace (split-K partials and tile tickets stay dirty),
 *                   as a kernel that failed half way would.
 *   SP_FAULT_STALL  a wait that runs out, in the kernels that wait on other
 *                   CTAs.  A tensor-core launch of a plan (SP_GEMM): one TMA
 *                   copy of the first CTA is never issued, and every wait of
 *                   that launch is bounded by about 2 ms instead of 1 s, so
 *                   the MMA's wait for the missing copy runs out: the kernel
 *                   raises the error word, stops issuing, drains the copies
 *                   it issued and frees its tensor memory.  A batch-1 decode
 *                   of a plan or group in thread-block clusters: the first
 *                   CTA never stores its partial sums into the owners'
 *                   shared memory, and the owners' waits (bounded by about
 *                   2 ms) run out: the kernel raises the error word and those
 *                   owners leave their outputs unwritten.  Other kernels
 *                   ignore it (it is still disarmed by their launch).
 * No fault traps, faults the GPU or spins without bound.  spike_proj_plan_status
 * / spike_proj_group_status then return SP_EKERNEL, clear the error word and
 * re-zero the workspace, and the next call is exact again.
 * Errors: SP_EINVAL (NULL, unknown fault).
 * ------------------------------------------------------------------------- */
typedef enum sp_fault {
    SP_FAULT_NONE = 0,
    SP_FAULT_ABORT = 1,
    SP_FAULT_STALL = 2
} sp_fault;
sp_status spike_proj_plan_inject_fault(sp_plan_t plan, int32_t fault);
sp_status spike_proj_group_inject_fault(sp_group_t group, int32_t fault);

/* ---------------------------------------------------------------------------
 * spike_proj_probe_gather -- MEASUREMENT AID, not part of the method (the
 * paper has no counterpart).  Reads `count` pieces of `piece_bytes`
 * contiguous bytes (512, 1024 or 1536), piece i at base + 16 * offsets16[i],
 * and nothing else: the pieces are dealt out round-robin over every warp of a
 * grid shaped like the gather's (4 CTAs of 256 threads per SM), each lane
 * reading 16 bytes of every 512 of each of its warp's pieces, all in one
 * round of loads, with the gather's programmatic dependent launch.  Given the
 * active-column pieces of a decode step (512-byte tile segments, as the
 * gather kernel reads them, or whole 1536-byte columns), its time per launch
 * is the practical ceiling of that access pattern, free of the method's
 * spike-word prologue and reduction; with count = 0 it measures the launch
 * and dependency floor alone.
 *
 *   base         device, 16-byte aligned.
 *   offsets16    device uint32 [count], in units of 16 bytes (so base may
 *                span 64 GB); every piece must lie inside an allocation.
 *   piece_bytes  512, 1024 or 1536 (else SP_EINVAL).
 *   sink         device uint32: the XOR of every 32-bit word read is XORed
 *                into it (so the bytes read can be checked).
 * Errors: SP_EINVAL, SP_EALIGN, SP_EDEVICE, SP_ECUDA.
 * ------------------------------------------------------------------------- */
sp_status spike_proj_probe_gather(const void *base, const uint32_t *offsets16,
                                  int32_t count, int32_t piece_bytes,
                                  uint32_t *sink, sp_stream_t stream);

/* --------------------------------------------------------------------------- */
const char *spike_proj_strerror(sp_status status);
/* cudaError_t code of the last failing CUDA call made by this thread. */
int spike_proj_last_cuda_error(void);
int spike_proj_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SPIKE_PROJ_H */
