/*
 * dtp.h -- C ABI of libdtp, the GB300 (sm_103a) hot path of affinity-aware
 * sharding for Delayed Tensor Parallelism ("Affinity-Aware Sharding for
 * Delayed Tensor Parallelism", arXiv 2609.13846).
 *
 * Two parts, both defined in Sec. 3 of the paper:
 *   1. the first-order head->neuron affinity of one layer ("Affinity scores"),
 *   2. the coordinate-ascent layout optimiser over balanced head partitions
 *      and neuron assignments ("Objective", "Optimiser").
 *
 * Conventions for every entry point:
 *   - Tensor arguments are DEVICE pointers owned by the caller; the library
 *     never frees or retains them.  Scratch memory is passed in as a
 *     caller-owned device workspace whose size the *_workspace_size query
 *     returns.  No call allocates device memory.  The one exception to the
 *     workspace rule is dtp_affinity_accumulate_noalloc, whose scratch is a
 *     fixed 16 MiB + 256 B array that the library holds on every GPU that
 *     loads it (a static device array, reserved when the library's module is
 *     loaded, not by any call).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Calls are asynchronous on it unless stated otherwise.
 *   - Arrays are row-major, contiguous, 16-byte aligned.
 *   - Every call returns a dtp_status; no C++ exception crosses the ABI.
 *     Argument errors are found on the host before anything is launched and
 *     leave every output untouched.
 *   - Calls on different streams with disjoint outputs and workspaces may run
 *     concurrently; a workspace must not be shared by calls in flight.
 */
#ifndef DTP_H_
#define DTP_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    DTP_OK = 0,
    DTP_ERR_ARG = -1,            /* invalid size, pointer, alignment or combination      */
    DTP_ERR_CUDA = -2,           /* a CUDA runtime/driver call failed                      */
    DTP_ERR_NOT_CONVERGED = -3,  /* a bounded device loop or wait hit its limit            */
    DTP_ERR_UNSUPPORTED = -4,    /* valid request the library does not handle (e.g. no GPU) */
    DTP_ERR_WORKSPACE = -5       /* workspace NULL or smaller than the size query's value  */
} dtp_status;

typedef enum {
    DTP_BF16 = 0, /* bf16 operands, fp32 accumulation (tcgen05 tensor cores)      */
    DTP_F32 = 1   /* fp32 operands and arithmetic (CUDA cores; tight-check mode) */
} dtp_dtype;

/* Library version as major*10000 + minor*100 + patch. */
int dtp_version(void);

/* Static, human-readable text for a dtp_status value. */
const char* dtp_status_string(int status);

/* ------------------------------------------------------------------------ */
/* 1. First-order affinity (Sec. 3 "Affinity scores")                        */
/* ------------------------------------------------------------------------ */

/*
 * Bytes of device workspace dtp_affinity_accumulate needs for these sizes and
 * dtype (written to *bytes).  Returns DTP_ERR_ARG for invalid sizes.
 */
int dtp_affinity_workspace_size(int64_t T, int d, int H_kv, int N, int dtype, size_t* bytes);

/*
 * A[h,k] += sum_{t<T} Delta_{t,h,k}^2, the first-order damage to SwiGLU
 * neuron k's output silu(g_k) u_k from removing KV head h's piece of the FFN
 * input (Sec. 3, the equation for Delta_hk):
 *     g = x_t . w^g_k,  u = x_t . w^u_k,  pg = c_{h,t} . w^g_k,  pu = c_{h,t} . w^u_k
 *     Delta = silu'(g) u pg + silu(g) pu,   silu'(g) = s (1 + g (1 - s)),  s = 1/(1+e^-g)
 *
 *   X       [T, d]        FFN input after the pre-norm (x / r * gamma), dtype
 *   C       [H_kv, T, d]  each KV group's piece p_h of that input, in the same
 *                         (post-norm) units, dtype
 *   W_gate  [N, d]        gate projection rows w^g_k (nn.Linear [out, in]), dtype
 *   W_up    [N, d]        up projection rows w^u_k, dtype
 *   A       [H_kv, N]     fp32, ACCUMULATED (zero it before the first chunk);
 *                         token chunks of one layer can therefore be streamed
 *                         through successive calls
 *   workspace             device scratch of at least
 *                         dtp_affinity_workspace_size(...) bytes
 *
 * The E_t mean and the ||w^d_k||^2 factor of the paper's S^{up,fo} are applied
 * by dtp_affinity_finalize.  The result is deterministic: the same inputs give
 * bitwise the same A (no floating-point atomics).
 * Requirements: T >= 0 (T == 0 returns DTP_OK at once and accepts NULL
 * pointers), d >= 8 and d % 8 == 0 (16-byte rows), 1 <= H_kv <= 16, N >= 1,
 * all pointers 16-byte aligned.
 * Asynchronous on `stream`.  A device-side wait that exceeds its limit sets
 * the workspace status word (see dtp_workspace_status).
 */
int dtp_affinity_accumulate(const void* X, const void* C, const void* W_gate, const void* W_up,
                            int64_t T, int d, int H_kv, int N, int dtype, float* A,
                            void* workspace, size_t workspace_bytes, void* stream);

/*
 * dtp_affinity_accumulate plus the down-edge activation term of Sec. 3
 * ("Affinity scores", down edge: neuron k writes alpha_k w^d_k into the
 * residual, alpha_k = silu(g_k) u_k its activation):
 *     act2[k] += sum_{t<T} alpha_k(t)^2 / rms_next[t]^2
 *   rms_next [T] fp32  rms r' of the residual entering the next layer's
 *                      pre-norm (> 0)
 *   act2     [N] fp32  accumulated
 * rms_next and act2 are both NULL (then this is dtp_affinity_accumulate) or
 * both set.  The workspace is sized by dtp_affinity_workspace_size, which
 * covers both forms.  A is bitwise the same as without the extra term.
 */
int dtp_affinity_accumulate_ex(const void* X, const void* C, const void* W_gate, const void* W_up,
                               const float* rms_next, int64_t T, int d, int H_kv, int N, int dtype,
                               float* A, float* act2, void* workspace, size_t workspace_bytes,
                               void* stream);

/*
 * Launch options of the bf16 affinity pass.
 *   max_ctas   0: one persistent CTA per SM (the default of the other entry
 *              points); n > 0: at most n CTAs, leaving the other SMs to
 *              kernels running concurrently on other streams (for instance the
 *              layout search of the previous layer, which runs on one SM).
 *              When the layer's W_gate and W_up fit in half of the L2 cache
 *              the kernel runs as pairs of CTAs, and n is then rounded down
 *              to an even count (at least one pair: 2 CTAs for n = 1)
 *   flags      DTP_AFFINITY_DEFER_REDUCE: launch only the main kernel; its
 *              per-unit partial sums stay in the workspace and
 *              dtp_affinity_reduce adds them into A (and act2) later, possibly
 *              on another stream (bf16 only)
 *   reserved   must be zero
 */
#define DTP_AFFINITY_DEFER_REDUCE 1
typedef struct dtp_affinity_opts {
    int max_ctas;
    int flags;
    int reserved[6];
} dtp_affinity_opts;

/*
 * dtp_affinity_accumulate_ex with launch options (opts non-NULL).  The
 * result does not depend on max_ctas (the reduction order is fixed by the
 * work units, not by the grid).  The fp32 mode ignores the options.  Same
 * workspace and errors as dtp_affinity_accumulate_ex.
 */
int dtp_affinity_accumulate_opts(const void* X, const void* C, const void* W_gate, const void* W_up,
                                 const float* rms_next, int64_t T, int d, int H_kv, int N, int dtype,
                                 float* A, float* act2, const dtp_affinity_opts* opts, void* workspace,
                                 size_t workspace_bytes, void* stream);

/*
 * The second half of a deferred affinity pass: adds the workspace's per-unit
 * partial sums into A [H_kv, N] (and, when act2 is non-NULL, the down-edge
 * activation sums into act2 [N]), in the same fixed order as the undeferred
 * call, so the result is bitwise the same.  T, d, H_kv, N and the workspace
 * are those of the deferred call; the stream must be ordered after it (the
 * caller records an event) and before the workspace is reused.
 *   max_blocks  0: a grid over the whole GPU; n > 0: n blocks of 1024 threads,
 *               for a reduce that runs beside a kernel holding the other SMs
 *   overwrite   nonzero: A (and act2) receive the sums instead of adding them
 *               (equal bit for bit to zeroing them first)
 */
int dtp_affinity_reduce(const void* workspace, size_t workspace_bytes, int64_t T, int d, int H_kv, int N,
                        float* A, float* act2, int max_blocks, int overwrite, void* stream);

/*
 * The first-order score per query head, summed over the query heads of each
 * KV group (Sec. 3, "Affinity scores": E_t[Delta_hk^2] is taken per query head
 * h from that head's own write p_h, and the group's score is the sum of its
 * query heads' scores):
 *   A[g,k] += sum over h = g*q_per_group .. (g+1)*q_per_group - 1 of
 *             sum_t Delta_{t,h,k}^2
 * This is a sum of squares, not the square of the group's summed write that
 * dtp_affinity_accumulate takes when given one C row per KV group.
 *   X, W_gate, W_up, rms_next, act2, dtype: as dtp_affinity_accumulate_ex
 *   C_q          [H_q, T, d], device: each query head's write p_h into the
 *                residual (the head's slice of W_o applied to its output)
 *   H_q          query heads, 1..128, a multiple of q_per_group
 *   q_per_group  query heads per KV group (1..16); H_q / q_per_group <= 16
 *   A            [H_q / q_per_group, N] fp32, device, accumulated into
 * Query heads are processed in chunks of at most 16 (whole groups); the X
 * pass runs once per chunk and act2 (when requested) is added once.  Row g's
 * sum runs over its query heads in order, then token tiles, so the result is
 * deterministic; with q_per_group == 1 it equals dtp_affinity_accumulate_ex.
 * Workspace from dtp_affinity_grouped_workspace_size.  Errors as
 * dtp_affinity_accumulate_ex.
 */
int dtp_affinity_grouped_workspace_size(int64_t T, int d, int H_q, int q_per_group, int N, int dtype,
                                        size_t* bytes);
int dtp_affinity_accumulate_grouped(const void* X, const void* C_q, const void* W_gate, const void* W_up,
                                    const float* rms_next, int64_t T, int d, int H_q, int q_per_group, int N,
                                    int dtype, float* A, float* act2, void* workspace, size_t workspace_bytes,
                                    void* stream);

/*
 * Where a layer's affinity concentrates (Sec. 5): for each neuron the largest
 * KV group's share of its column, max_g A[g,k] / sum_g A[g,k], averaged over
 * the neurons whose column is not zero (0 when none is); 1/H_kv when the groups
 * contribute equally.  fp64 arithmetic, fixed reduction order.
 *   A      [layers, H_kv, N] fp32, device, entries finite and >= 0
 *   share  [layers] double out, device
 * Asynchronous; no workspace.
 */
int dtp_affinity_top_share(const float* A, int layers, int H_kv, int N, double* share, void* stream);

/*
 * The ADD score of Sec. 3 before the mean: the squared additive contribution
 * of KV group h's piece to neuron k's pre-activations, ignoring the operating
 * point and ||w^d_k||:
 *     A_add[h,k] += sum_{t<T} (c_{h,t} . w^g_k)^2 + (c_{h,t} . w^u_k)^2
 * C [H_kv, T, d], W_gate/W_up [N, d] bf16; A_add [H_kv, N] fp32 accumulated.
 * Same size rules as dtp_affinity_accumulate; workspace from
 * dtp_affinity_add_workspace_size.  Deterministic.  Asynchronous.
 */
int dtp_affinity_add_workspace_size(int64_t T, int d, int H_kv, int N, size_t* bytes);
int dtp_affinity_add_accumulate(const void* C, const void* W_gate, const void* W_up, int64_t T, int d,
                                int H_kv, int N, float* A_add, void* workspace,
                                size_t workspace_bytes, void* stream);

/*
 * The ADD score per query head, summed over the query heads of each KV group
 * (Sec. 3):  A_add[g,k] += sum over the group's query heads h of
 *            sum_t (p_{h,t} . w^g_k)^2 + (p_{h,t} . w^u_k)^2
 * C_q [H_q, T, d] bf16 (each query head's write), A_add [H_q / q_per_group, N]
 * fp32 accumulated; H_q and q_per_group as dtp_affinity_accumulate_grouped.
 * Workspace from dtp_affinity_add_grouped_workspace_size.  Deterministic;
 * with q_per_group == 1 equals dtp_affinity_add_accumulate.  Asynchronous.
 */
int dtp_affinity_add_grouped_workspace_size(int64_t T, int d, int H_q, int q_per_group, int N, size_t* bytes);
int dtp_affinity_add_accumulate_grouped(const void* C_q, const void* W_gate, const void* W_up, int64_t T, int d,
                                        int H_q, int q_per_group, int N, float* A_add, void* workspace,
                                        size_t workspace_bytes, void* stream);

/*
 * Down-edge weight factor (Sec. 3): bn[g,k] = ||b_gk||^2 with
 * b_gk = W^qkv_g (gamma' . w^d_k), the column w^d_k of this layer's down
 * projection seen by KV group g of the next layer through its pre-norm gain.
 *   Wqkv_next  [H_kv, R, d] bf16: the next layer's q, k and v projection rows of
 *              each KV group (the group's query heads with its key and value
 *              head), R rows per group
 *   gamma_next [d] bf16: the next layer's attention pre-norm gain
 *   W_down     [d, N] bf16 (nn.Linear [out=d, in=N])
 *   bn         [H_kv, N] fp32 out (overwritten)
 * gamma' . w^d_k is rounded to bf16 once before the tensor-core product.
 * Requirements: d % 8 == 0; dtype DTP_BF16 (others: DTP_ERR_UNSUPPORTED).
 * Workspace from dtp_down_weight_workspace_size.  Asynchronous.
 */
int dtp_down_weight_workspace_size(int H_kv, int R, int d, int N, size_t* bytes);
int dtp_down_weight_sqnorm(const void* Wqkv_next, const void* gamma_next, const void* W_down,
                           int H_kv, int R, int d, int N, int dtype, float* bn, void* workspace,
                           size_t workspace_bytes, void* stream);

/*
 * The down-edge affinity of Sec. 3: S_down[g,k] = act2[k] / T_total * bn[g,k]
 * = E_t[alpha_k^2 / r'^2] ||b_gk||^2, how much KV group g of the next layer
 * depends on neuron k of this layer.  Stored [H_kv, N] (the transpose of the
 * paper's I x G orientation).  All device fp32.  Asynchronous.
 */
int dtp_down_finalize(const float* act2, const float* bn, int H_kv, int N, int64_t T_total,
                      float* S_down, void* stream);

/*
 * A[h,k] *= wd_sqnorm[k] / T_total, the token mean E_t and the squared norm of
 * neuron k's down-projection column (Sec. 3, S^{up,fo} = E_t[Delta^2] ||w^d_k||^2).
 * wd_sqnorm: device fp32 [N], or NULL for a factor of 1.  T_total >= 1.
 * Both factors are positive, so neither changes the layout the optimiser finds
 * except through the per-neuron ||w^d_k||^2.  Asynchronous on `stream`.
 */
int dtp_affinity_finalize(float* A, int H_kv, int N, int64_t T_total, const float* wd_sqnorm,
                          void* stream);

/*
 * out[k] = sum_i W_down[i,k]^2 = ||w^d_k||^2 for W_down [d, N] (nn.Linear
 * [out=d, in=N]) of the given dtype; out is device fp32 [N].  The input of
 * dtp_affinity_finalize (Sec. 3, "w^d_k the down-projection column").
 */
int dtp_down_sqnorm(const void* W_down, int d, int N, int dtype, float* out, void* stream);

/*
 * dtp_affinity_accumulate with DTP_BF16 for callers that cannot allocate
 * device memory or pass a workspace (e.g. a plugin whose host application
 * owns every device allocation, or a runtime with a fixed memory plan that
 * must not grow after start-up).  The paper has no counterpart: this entry
 * point only changes where the scratch lives.
 *
 * Same arguments, layouts and accumulation as dtp_affinity_accumulate (bf16
 * inputs only), minus the workspace; the same kernels in the same launch
 * shape give A bit for bit equal to that call's.  Scratch comes from one fixed
 * device array of 16 MiB + 256 B inside the library, present on every GPU
 * that loads it until the process exits; the call allocates nothing.
 *   - Limit: c * ceil(N/128) * H_kv <= 32768 per call, with c = ceil(T/128)
 *     rounded up to an even count, else DTP_ERR_WORKSPACE (stream longer
 *     inputs as token chunks; A accumulates).
 *   - Every call shares the array and it keeps the last call's contents:
 *     calls that overlap on the GPU race and must be serialised by the caller.
 *   - The first call on a device looks up the array's device address with
 *     that device current; make it before any stream capture begins.  The
 *     address is kept for the life of the process: no call may follow a
 *     cudaDeviceReset of that device.
 *   - A bounded device-side wait that gives up leaves the partial sums of
 *     its units unwritten, and the reduce still adds every slot into A, so A
 *     is then wrong.  The kernels record this in the array's status word:
 *     dtp_affinity_noalloc_status reads it back after the call.
 * Asynchronous on `stream`.
 */
int dtp_affinity_accumulate_noalloc(const void* X, const void* C, const void* W_gate,
                                    const void* W_up, int64_t T, int d, int H_kv, int N, float* A,
                                    void* stream);

/*
 * Device-side status of the last dtp_affinity_accumulate_noalloc call on the
 * current device (no paper passage: this library's failure reporting).
 * Synchronises `stream` (pass the stream of that call), then reads the status
 * word in the library's fixed scratch array: DTP_OK, or DTP_ERR_NOT_CONVERGED
 * if a bounded wait of the call's kernels gave up (A is then not valid).
 * Calls of dtp_affinity_accumulate_noalloc that are still queued on other
 * streams may overwrite the word; order them before this read.  Returns
 * DTP_ERR_CUDA if the copy or the synchronisation fails.  Allocates nothing.
 */
int dtp_affinity_noalloc_status(void* stream);

/*
 * Synchronises `stream`, then reads the status word that kernels of the last
 * call using `workspace` leave in it: DTP_OK, DTP_ERR_NOT_CONVERGED if a
 * bounded device-side wait or loop gave up, or DTP_ERR_ARG if the layout
 * search found an invalid entry of A.  workspace_bytes as passed to that call.
 */
int dtp_workspace_status(const void* workspace, size_t workspace_bytes, void* stream);

/*
 * Self-test of the bounded device-side waits every kernel here relies on (no
 * paper passage: a check of this library's failure reporting).  One block:
 * thread 0 waits on an mbarrier with limit_ns (1 us .. 1 s); with complete = 0
 * nothing ever arrives, the wait gives up, sets the shared abort flag and the
 * workspace status word (DTP_ERR_NOT_CONVERGED), and a second thread waiting
 * on another never-completed barrier with the library's own limit (2 s) must
 * leave on that flag; with complete = 1 another warp arrives first and the
 * status stays DTP_OK.  Writes the two waits' durations (ns) to
 * elapsed_ns[0..1] (host, 2 entries; the second is 0 when complete = 1) and
 * synchronises `stream`.  Read the status with dtp_workspace_status.
 * workspace: device, at least 256 bytes.  DTP_ERR_ARG for a null pointer, a
 * small workspace or a limit outside the range.
 */
int dtp_selftest_bounded_wait(uint64_t limit_ns, int complete, void* workspace, size_t workspace_bytes,
                              uint64_t* elapsed_ns, void* stream);

/* ------------------------------------------------------------------------ */
/* 2. Layout optimiser (Sec. 3 "Objective", "Optimiser")                     */
/* ------------------------------------------------------------------------ */

/*
 * Bytes of device workspace dtp_search_layout(_batched) needs for `layers`
 * layers of [H_kv, N] affinities over D devices.
 */
int dtp_search_workspace_size(int layers, int H_kv, int N, int D, size_t* bytes);

/*
 * Coordinate ascent on the up-edge objective of one layer (Sec. 3):
 *   J(h, nu) = sum over (g,k) with h(g) == nu(k) of S[g,k] / sum S,
 * over balanced layouts: h assigns H_kv/D KV groups and nu assigns N/D neurons
 * to each of the D devices.
 *
 *   - Exact arithmetic: the layer's matrix is mapped to the fixed-point form
 *     q[g,k] = floor(A[g,k] * 2^(40-e)), max(A) < 2^e; unit-mass normalisation
 *     is a positive scale and is applied only to the reported score.
 *   - Start: contiguous heads h(g) = floor(g*D/H_kv).
 *   - Iteration: neuron step (the optimal balanced assignment nu given h; the
 *     gain of neuron k on device l is M[k,l] = sum over g with h(g) == l of
 *     q[g,k]), then head step (the best of all H_kv!/((H_kv/D)!)^D labelled
 *     balanced partitions given nu).
 *   - Ties: the lexicographically smallest optimal nu, and the
 *     lexicographically smallest best h.
 *   - Stop after `iters` iterations or after the first iteration whose
 *     integer score does not strictly exceed the previous one.
 *
 *   A           [H_kv, N] fp32, device, finite and >= 0
 *   head_part   [H_kv] int32 out (device): h(g) in 0..D-1
 *   neuron_dev  [N] int32 out (device): nu(k) in 0..D-1
 *   score_q     int64 out (device): co-located fixed-point mass
 *   score       double out (device): score_q / sum(q), in [0,1] (0 if A == 0)
 *   iters_done  int32 out (device): iterations run (1..iters)
 * Requirements: 2 <= D <= 8, D | H_kv, D | N, H_kv <= 16, N <= 262144,
 * H_kv * N <= 4194304, iters >= 1, the partition count <= 2^26.
 * Asynchronous on `stream`.  A negative or non-finite entry of A
 * (DTP_ERR_ARG) or a bounded device loop that hit its limit
 * (DTP_ERR_NOT_CONVERGED) is reported through the workspace status word,
 * read with dtp_workspace_status; that layer's outputs are then not written.
 */
int dtp_search_layout(const float* A, int H_kv, int N, int D, int iters,
                      int32_t* head_part, int32_t* neuron_dev, int64_t* score_q, double* score,
                      int32_t* iters_done, void* workspace, size_t workspace_bytes, void* stream);

/*
 * dtp_search_layout on `layers` independent layers at once (the up-edge
 * objective decouples across layers); layer i reads A + i*H_kv*N and writes
 * head_part + i*H_kv, neuron_dev + i*N, score_q[i], score[i], iters_done[i].
 * One thread block per layer.  Asynchronous; the workspace status word holds
 * the most severe device-side status over the layers (DTP_ERR_NOT_CONVERGED
 * before DTP_ERR_ARG before DTP_OK).
 */
int dtp_search_layout_batched(const float* A, int layers, int H_kv, int N, int D, int iters,
                              int32_t* head_part, int32_t* neuron_dev, int64_t* score_q,
                              double* score, int32_t* iters_done, void* workspace,
                              size_t workspace_bytes, void* stream);

/*
 * The whole-model objective of Sec. 3 (Eq. objective, both sums) and its
 * optimiser over `layers` layers:
 *   J(h, nu) = sum_i sum over (g,k) with h_i(g) == nu_i(k) of S_up_i[g,k] / sum S_up_i
 *            + sum_{i<layers-1} sum over (g,k) with nu_i(k) == h_{i+1}(g) of
 *                                               S_down_i[g,k] / sum S_down_i
 * J lies in [0, 2*layers - 1]; a uniform random balanced layout scores
 * (2*layers - 1)/D in expectation.
 *   - Exact arithmetic: each matrix is mapped to n = floor(q 2^43 / sum q),
 *     q = floor(S 2^(40-e)), max(S) < 2^e (the product in 128 bits); J_q =
 *     sum of co-located n.
 *   - Start: contiguous heads in every layer.  One iteration: every layer's
 *     neuron step given all head partitions (gain M_kl of Sec. 3 with the up
 *     term from h_i and the down term from h_{i+1}), then every layer's head
 *     step given all neuron assignments (up term over nu_i, down term over
 *     nu_{i-1}).  Each step maximises J exactly given the other block.
 *   - Ties: lexicographically smallest nu_i and h_i, as in dtp_search_layout.
 *   - Stop after `iters` iterations or the first without a strict increase.
 *
 *   S_up       [layers, H_kv, N] fp32, device, finite and >= 0
 *   S_down     [layers-1, H_kv, N] fp32 (S_down[i][g,k]: group g of layer i+1
 *              on neuron k of layer i; dtp_down_finalize's layout), or NULL
 *              when layers == 1
 *   head_part  [layers, H_kv] int32 out; neuron_dev [layers, N] int32 out
 *   J_q        int64 out, J in units of 2^-43; J double out; iters_done int32 out
 * Same size rules as dtp_search_layout; workspace from
 * dtp_search_chain_workspace_size.  Asynchronous; invalid entries or loop
 * limits are reported through the workspace status word.
 */
int dtp_search_chain_workspace_size(int layers, int H_kv, int N, int D, size_t* bytes);
int dtp_search_chain(const float* S_up, const float* S_down, int layers, int H_kv, int N, int D,
                     int iters, int32_t* head_part, int32_t* neuron_dev, int64_t* J_q, double* J,
                     int32_t* iters_done, void* workspace, size_t workspace_bytes, void* stream);

/*
 * The exact maximum of each layer's up-edge objective over every balanced
 * layout (Sec. 3 "Objective": J of one layer, Sec. 3 "Optimiser" uses it only
 * through the ascent; this is the reference the ascent is measured against).
 * J is unchanged when device labels are permuted jointly in h and nu, so the
 * maximum is the best exact neuron step over the unlabelled balanced head
 * partitions, H_kv! / ((H_kv/D)!^D D!) of them (35 for H_kv=8, D=2; 105 for
 * D=4; 1 for D=8).  Each partition is taken in its canonical labelling (a
 * device label first appears after every smaller one); the first partition in
 * lexicographic order with the largest value wins, with its exact neuron
 * step's lexicographically smallest assignment.  Arithmetic and A as in
 * dtp_search_layout_batched (score_q exact, score = score_q / sum q).
 *   A           [layers, H_kv, N] fp32, device
 *   head_part   [layers, H_kv] int32 out (canonical labels)
 *   neuron_dev  [layers, N] int32 out;  score_q [layers] int64, score [layers]
 *               double out
 * Size rules of dtp_search_layout, and at most 2^20 unlabelled partitions per
 * layer.  Workspace from dtp_search_global_workspace_size.  Asynchronous;
 * invalid entries are reported through the workspace status word.
 */
int dtp_search_global_workspace_size(int layers, int H_kv, int N, int D, size_t* bytes);
int dtp_search_global(const float* A, int layers, int H_kv, int N, int D, int32_t* head_part,
                      int32_t* neuron_dev, int64_t* score_q, double* score, void* workspace,
                      size_t workspace_bytes, void* stream);

/*
 * dtp_search_chain with the ablations of Sec. 3 ("Optimiser"; the layouts of
 * Table 4): restricting which layers move, freezing heads or neurons, or
 * minimising J (the anti-optimised layout).
 *   move_heads    [layers] uint8, device, or NULL (= every layer): 0 keeps
 *                 layer i's head partition at the contiguous start
 *   move_neurons  [layers] uint8, device, or NULL: 0 keeps layer i's neuron
 *                 assignment contiguous (nu_i(k) = floor(k D / N))
 *   minimize      nonzero: every step minimises J exactly given the other
 *                 block (ties: lexicographically smallest, as when
 *                 maximising); the stop rule applies to -J
 * dtp_search_chain(...) equals dtp_search_chain_ex(..., NULL, NULL, 0, ...).
 * The flag arrays are read by the kernels, so they must stay valid until the
 * stream reaches the end of this call's work.  Same workspace and errors as
 * dtp_search_chain.
 */
int dtp_search_chain_ex(const float* S_up, const float* S_down, int layers, int H_kv, int N, int D, int iters,
                        const uint8_t* move_heads, const uint8_t* move_neurons, int minimize, int32_t* head_part,
                        int32_t* neuron_dev, int64_t* J_q, double* J, int32_t* iters_done, void* workspace,
                        size_t workspace_bytes, void* stream);

/*
 * J of a given layout (Eq. objective, both sums) and its per-edge terms; the
 * paper scores random layouts this way alongside the optimiser (Sec. 3).
 *   head_part   [layers, H_kv] int32, device, entries in [0, D)
 *   neuron_dev  [layers, N] int32, device, entries in [0, D)
 *   edge_q      [2*layers - 1] int64 out, device, or NULL: edge 2i is the
 *               co-located mass of layer i's up edge, edge 2i+1 that of its
 *               down edge, each in units of 2^-43 of that edge's own total
 *               (edge_q / 2^43 is the co-located fraction of the edge)
 *   J_q, J      the sum, as in dtp_search_chain
 * The layout need not be balanced.  S_up, S_down and the size rules are those
 * of dtp_search_chain (D as given); workspace from
 * dtp_search_chain_workspace_size.  Asynchronous; negative or non-finite
 * affinities and layout entries outside [0, D) are reported as DTP_ERR_ARG
 * through the workspace status word.
 */
int dtp_chain_score(const float* S_up, const float* S_down, int layers, int H_kv, int N, int D,
                    const int32_t* head_part, const int32_t* neuron_dev, int64_t* edge_q, int64_t* J_q, double* J,
                    void* workspace, size_t workspace_bytes, void* stream);

/*
 * The producer of C (Sec. 3, "Affinity scores"): each attention head's write
 * into the FFN input, with the rms held fixed,
 *     C[j, t, :] = gamma . ( sum over heads h of row j of a_{h,t} W_o^(h)T ) / rms[t]
 *   attn   [T, H_q*head_dim] bf16, device: the heads' outputs before o_proj
 *          (head h in columns h*head_dim .. h*head_dim + head_dim - 1)
 *   W_o    [d, H_q*head_dim] bf16, device: o_proj (nn.Linear [out, in])
 *   gamma  [d] fp32, device, 16-byte aligned: the FFN pre-norm gain
 *   rms    [T] fp32, device, > 0: rms of the residual entering that norm
 *   q_per_row  heads per output row: 1 = one row per query head (for
 *          dtp_affinity_accumulate_grouped), query heads per KV group = the
 *          group's combined write (for dtp_affinity_accumulate)
 *   C      [H_q / q_per_row, T, d] bf16 out, device (rounded once, RN)
 * head_dim a multiple of 16; d a multiple of 8; H_q * head_dim <= 2^20.
 * tcgen05 GEMM with fp32 accumulation; the fp32 product is scaled by
 * gamma / rms before the rounding.  Workspace: dtp_head_writes_workspace_size
 * bytes (a status word).  Asynchronous; T == 0 returns DTP_OK.
 */
int dtp_head_writes_workspace_size(size_t* bytes);
int dtp_head_writes(const void* attn, const void* W_o, const float* gamma, const float* rms, int64_t T, int d,
                    int H_q, int head_dim, int q_per_row, void* C, void* workspace, size_t workspace_bytes,
                    void* stream);

/*
 * Applying a layout to the dense weights (Sec. 3: the permuted dense model is
 * sharded into contiguous slices).  dtp_layout_order turns device labels into
 * the order that lists every device's items contiguously:
 *     order[i][p] = the item at position p when layer i's items are listed
 *                   device by device, each device's in increasing index
 *   labels  [layers, n] int32, device: head_part or neuron_dev
 *   order   [layers, n] int32 out, device
 *   balanced  nonzero: also require n / D items per device, so that position
 *             p belongs to device floor(p D / n)
 * Labels outside [0, D), or an unbalanced layer when `balanced`, are reported
 * as DTP_ERR_ARG through the workspace status word (order undefined).
 * Workspace: dtp_head_writes_workspace_size bytes.  Asynchronous.
 */
int dtp_layout_order(const int32_t* labels, int layers, int n, int D, int balanced, int32_t* order,
                     void* workspace, size_t workspace_bytes, void* stream);

/*
 * Gathers that apply the order to weights stored [layers, rows, ...]
 * contiguous (one matrix per layer, back to back), src and dst distinct:
 *   dtp_permute_rows: dst[i][b*block_rows + r][:] = src[i][perm[i][b]*block_rows + r][:]
 *     rows of row_bytes bytes; q_proj (block = query heads per group *
 *     head_dim rows per KV group), k_proj / v_proj (block = head_dim),
 *     gate_proj / up_proj (block = 1 row per neuron)
 *   dtp_permute_cols: dst[i][r][b*block_cols + c] = src[i][r][perm[i][b]*block_cols + c]
 *     elements of elem_bytes bytes; o_proj (block = query heads per group *
 *     head_dim columns), down_proj (block = 1 column per neuron)
 *   perm  int32, device, layer i's entries at perm + i * perm_layer_stride
 * An entry of perm outside [0, blocks) is not followed (nothing is read
 * through it): the affected elements of dst are left unwritten or, where dst
 * is written in 16-byte words that they share with valid elements, set to
 * zero, and DTP_ERR_ARG is reported through the workspace status word.
 * Workspace: dtp_head_writes_workspace_size bytes.  Asynchronous.
 */
int dtp_permute_rows(const void* src, void* dst, int layers, int64_t rows, int64_t row_bytes, int block_rows,
                     const int32_t* perm, int64_t perm_layer_stride, void* workspace, size_t workspace_bytes,
                     void* stream);
int dtp_permute_cols(const void* src, void* dst, int layers, int64_t rows, int64_t cols, int elem_bytes,
                     int block_cols, const int32_t* perm, int64_t perm_layer_stride, void* workspace,
                     size_t workspace_bytes, void* stream);

/*
 * The whole layout application of Sec. 3 in one call: the orders of the head
 * partitions and neuron assignments of `layers` layers, and the gathers of
 * the seven weight matrices, stacked [layers, ...] in one element type:
 *   src[0], dst[0]  q_proj  [layers, H_kv*q_per_group*head_dim, d]  (rows by KV group)
 *   src[1], dst[1]  k_proj  [layers, H_kv*head_dim, d]               (rows by KV group)
 *   src[2], dst[2]  v_proj  [layers, H_kv*head_dim, d]               (rows by KV group)
 *   src[3], dst[3]  o_proj  [layers, d, H_kv*q_per_group*head_dim]   (columns by KV group)
 *   src[4], dst[4]  gate_proj [layers, N, d]                         (rows by neuron)
 *   src[5], dst[5]  up_proj   [layers, N, d]                         (rows by neuron)
 *   src[6], dst[6]  down_proj [layers, d, N]                         (columns by neuron)
 * src and dst are host arrays of 7 device pointers (dst distinct from src);
 * head_part [layers, H_kv] and neuron_dev [layers, N] int32 device, balanced;
 * head_order [layers, H_kv] and neuron_order [layers, N] int32 device out
 * (dtp_layout_order's).  Device l's shard of the permuted weights is then the
 * l-th contiguous slice.  Workspace: dtp_head_writes_workspace_size bytes;
 * unbalanced layouts and labels outside [0, D) are reported through its status
 * word.  Asynchronous; 9 launches.
 */
int dtp_apply_layout(const int32_t* head_part, const int32_t* neuron_dev, int layers, int H_kv, int N, int D,
                     int q_per_group, int head_dim, int d, int elem_bytes, const void* const* src,
                     void* const* dst, int32_t* head_order, int32_t* neuron_order, void* workspace,
                     size_t workspace_bytes, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* DTP_H_ */
