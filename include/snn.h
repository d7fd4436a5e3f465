/*
 * snn.h — C ABI of libsnn: the fused temporal scan of spiking-neuron state
 * equations on one GPU (sm_103a), forward over T steps and the BPTT reverse
 * scan with a surrogate gradient, plus the dense input-current GEMM.
 *
 * Method: arXiv 2211.10725, Sec. III-A/III-B.
 *   Eq. (3)      z_t = 1 if u_t > u_thr else 0 (strict).
 *   Eq. (4)      Leaky:     u_t = beta*u_{t-1} + I_t - z_{t-1}*u_thr
 *   Eqs. (5)(6)  Synaptic:  i_t = alpha*i_{t-1} + I_t,
 *                           u_t = beta*u_{t-1} + i_t - z_{t-1}*u_thr
 *   Eqs. (8)(9)  fast-sigmoid surrogate for dz/du (arctan is the other choice)
 *   Sec. II-A/B  BPTT over the unrolled graph.
 * I_t = w x_t is the input current; the (1-beta) factor of Eq. (2) is absorbed
 * into it.  Reset-to-zero (u_t = beta*(1-z_{t-1})*u_{t-1} + I_t, clears only u
 * in the Synaptic neuron) and "no reset" are extensions the paper names but
 * does not write out.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Tensors of a scan are [T, B, N] row-major with t outermost: lane
 *   l = b*N + n, element (t, l) at offset t*B*N + l.  Per-lane states and
 *   their gradients (mem0, syn0, mem_final, grad_mem0, ...) are fp32 [B, N].
 * - Every pointer argument is a DEVICE pointer unless stated, owned by the
 *   caller; the library allocates nothing.  Between calls it keeps only a
 *   process-wide count of its kernel launches (snn_kernel_launches), per
 *   device caches of launch plans and device attributes, and the fixed
 *   device array of snn_leaky_bwd_noalloc.  Results never depend on them.
 *   Outputs are overwritten, never accumulated into.
 * - Calls are asynchronous on `stream` and never synchronise it (except
 *   snn_workspace_status).  Arguments are checked before anything is
 *   launched; a failed check returns an error code and launches nothing.
 * - Device pointers must be 16-byte aligned (SNN_ERR_ALIGNMENT otherwise).
 *   Shapes whose per-step row (B*N*element size) is a multiple of 16 bytes
 *   take the TMA-staged kernels; any other shape takes a plain per-lane
 *   kernel with identical arithmetic.
 * - Spin-waits inside kernels are bounded (snn_scan_desc.wait_limit_ns); a
 *   kernel that gives up records SNN_ERR_TIMEOUT in the workspace status word
 *   and returns.  snn_workspace_status reports it.
 */
#ifndef SNN_H_
#define SNN_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif
#if defined(__GNUC__)
#pragma GCC visibility push(default)
#endif

/* Same object as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* snn_stream_t;

typedef enum {
  SNN_OK = 0,
  SNN_ERR_INVALID_ARG = 1, /* null/inconsistent argument or out-of-range enum  */
  SNN_ERR_ALIGNMENT = 2,   /* a device pointer is not 16-byte aligned          */
  SNN_ERR_UNSUPPORTED = 3, /* valid request that this build does not implement */
  SNN_ERR_WORKSPACE = 4,   /* workspace missing or smaller than required       */
  SNN_ERR_CUDA = 5,        /* a CUDA runtime call or kernel launch failed      */
  SNN_ERR_TIMEOUT = 6      /* a bounded in-kernel wait gave up                 */
} snn_status_t;

typedef enum { SNN_F32 = 0, SNN_BF16 = 1, SNN_F16 = 2 } snn_dtype_t;

typedef enum {
  SNN_RESET_SUBTRACT = 0, /* Eq. (4): - z_{t-1} * u_thr                       */
  SNN_RESET_ZERO = 1,     /* u_t = beta*(1 - z_{t-1})*u_{t-1} + input         */
  SNN_RESET_NONE = 2      /* no reset term                                    */
} snn_reset_t;

typedef enum {
  SNN_SG_FAST_SIGMOID = 0, /* dz/du <- 1/(1 + k|u-thr|)^2, k = sg_param (Eq. 9 at k=1) */
  SNN_SG_ATAN = 1          /* dz/du <- (a/2)/(1 + (pi*a*(u-thr)/2)^2), a = sg_param  */
} snn_surrogate_t;

typedef enum {
  SNN_P_SCALAR = 0,     /* one value                                           */
  SNN_P_PER_NEURON = 1, /* [N], indexed by n                                   */
  SNN_P_PER_CHANNEL = 2 /* [C], channel of neuron n is (n / HW) % C            */
} snn_pmode_t;

typedef enum {
  SNN_SAVE_MEM = 0,      /* BPTT reads the stored mem (and spk) traces          */
  SNN_SAVE_RECOMPUTE = 1 /* BPTT recomputes u from I and fp32 checkpoints taken
                            every ckpt_every steps by the forward              */
} snn_save_t;

/* Debug flags (snn_scan_desc.debug_flags); 0 in normal use. */
#define SNN_DEBUG_PRODUCER_IDLE 1u /* staged kernels issue no copy, so every
                                      consumer wait runs out: exercises the
                                      timeout path without any fault          */
#define SNN_DEBUG_FORCE_PLAIN 2u   /* take the plain per-lane kernels even
                                      where the staged ones apply             */
#define SNN_DEBUG_NO_SEGMENT 4u    /* recompute BPTT of the Leaky neuron: take
                                      the shared-memory replay kernel even
                                      where the register-segment one applies  */

typedef struct snn_scan_desc {
  int64_t T, B, N;       /* time steps, batch, neurons per sample (C*H*W maps) */
  int64_t C, HW;         /* per-channel parameters: channel = (n / HW) % C     */
  int32_t in_dtype;      /* snn_dtype_t of I                                   */
  int32_t io_dtype;      /* of spk, mem, syn, grad_spk, grad_mem, grad_I       */
  int32_t reset;         /* snn_reset_t                                        */
  int32_t detach_reset;  /* 1: z_{t-1} in the reset term is a constant in BPTT */
  int32_t surrogate;     /* snn_surrogate_t                                    */
  float sg_param;        /* fast-sigmoid slope k, or arctan alpha              */
  int32_t beta_mode, thr_mode, alpha_mode; /* snn_pmode_t; alpha_mode is the
                            layout of alpha (Synaptic) or of v (recurrent)     */
  int32_t save;          /* snn_save_t                                         */
  int32_t ckpt_every;    /* K >= 1 for SNN_SAVE_RECOMPUTE                      */
  int32_t reserved0;     /* must be 0                                          */
  int64_t wait_limit_ns; /* bound on each in-kernel wait; 0 = 2 s              */
  uint32_t debug_flags;  /* SNN_DEBUG_*                                        */
  uint32_t reserved1;    /* must be 0                                          */
} snn_scan_desc;

/* Human-readable name of a status code (static string, never NULL). */
const char* snn_status_string(snn_status_t status);

/* Number of kernels this library has launched in this process (a launch
 * captured into a CUDA graph counts once, at capture): the difference over
 * one eagerly issued step is that step's launch count. */
uint64_t snn_kernel_launches(void);

/* Library version, as 10000*major + 100*minor + patch. */
int snn_version(void);

/* sizeof(snn_scan_desc) as compiled into the library (ABI check). */
size_t snn_scan_desc_size(void);

/* Bytes of device workspace every scan call of `desc` needs (a status word,
 * per-lane parameter-gradient partials, reduction scratch in 8-byte slots
 * and the reductions' completion tickets).  0 if desc is invalid.  The tickets must
 * start at zero (snn_workspace_init) and each reduction leaves them at zero;
 * after a call that reported SNN_ERR_TIMEOUT, initialise the workspace
 * again. */
size_t snn_scan_workspace_bytes(const snn_scan_desc* desc);

/* Number of fp32 elements of the ckpt buffer passed to the forward and the
 * backward of one sequence:
 *   SNN_SAVE_RECOMPUTE: (ceil(T/K) - 1) * B*N for Leaky, twice that for
 *     Synaptic (u then i per checkpoint);
 *   SNN_SAVE_MEM with a bf16/fp16 io_dtype: T rows of ceil(B*N/8) bytes
 *     rounded up to 16, in fp32 units: the spike bits (bit k of byte j of
 *     row t is z_t of lane 8j + k).  Optional: given to both calls, the
 *     backward reads 1 bit per neuron-step instead of the 16-bit spk row
 *     (used when B*N is a multiple of 8; otherwise spk is read);
 *   SNN_SAVE_MEM with fp32 io: 0.
 * 0 for an invalid desc. */
int64_t snn_scan_ckpt_elems(const snn_scan_desc* desc, int synaptic);

/* Zero a workspace (its status word included); asynchronous on stream.
 * Call once after allocating it. */
snn_status_t snn_workspace_init(void* ws, size_t ws_bytes, snn_stream_t stream);

/* Synchronise stream, return the sticky status recorded by kernels in ws
 * (SNN_OK or SNN_ERR_TIMEOUT) and clear it. */
snn_status_t snn_workspace_status(void* ws, snn_stream_t stream);

/*
 * Leaky LIF forward, Eqs. (3)-(4), over t = 0..T-1.
 *   I        [T,B,N] in_dtype            input current w x_t
 *   beta,thr fp32, shape per beta_mode/thr_mode
 *   mem0     fp32 [B,N] or NULL          u_{-1}; NULL means u_{-1}=0, z_{-1}=0,
 *                                        else z_{-1} = [mem0 > thr]
 *   spk      [T,B,N] io_dtype  (out)     z_t in {0,1}
 *   mem      [T,B,N] io_dtype  (out)     u_t; required for SNN_SAVE_MEM, else
 *                                        optional (NULL = not written)
 *   ckpt     fp32 (out)                  SNN_SAVE_RECOMPUTE: u at the end of every
 *                                        segment but the last.  Segments are aligned
 *                                        to the end of the sequence: the first has
 *                                        T-(ceil(T/K)-1)*K steps, the others K.
 *                                        SNN_SAVE_MEM, half io: the spike bits, or
 *                                        NULL (see snn_scan_ckpt_elems).
 *   mem_final fp32 [B,N] (out) or NULL   u_{T-1}
 *   ws       workspace of snn_scan_workspace_bytes(desc) bytes
 * State is kept in fp32; the step is evaluated as Eq. (4) is written:
 * (beta*u_{t-1} + I_t) - z_{t-1}*thr, each operation rounded to nearest.
 */
snn_status_t snn_leaky_fwd(const snn_scan_desc* desc, const void* I, const float* beta,
                           const float* thr, const float* mem0, void* spk, void* mem,
                           float* ckpt, float* mem_final, void* ws, size_t ws_bytes,
                           snn_stream_t stream);

/*
 * Leaky LIF BPTT (Sec. II-A/B) with the surrogate of Sec. III-B.
 * Inputs of the saved forward:
 *   SNN_SAVE_MEM:       mem [T,B,N] io_dtype; spk [T,B,N] io_dtype, needed
 *                       when io_dtype is not fp32 (a rounded mem cannot give
 *                       back the spike decision) unless the forward wrote the
 *                       spike bits to ckpt and B*N is a multiple of 8; may be
 *                       NULL for fp32.  ckpt: the forward's spike bits or NULL.
 *   SNN_SAVE_RECOMPUTE: I [T,B,N] in_dtype and ckpt from snn_leaky_fwd.
 *   beta, thr, mem0 as in the forward.
 * Upstream gradients:
 *   grad_spk [T,B,N] io_dtype            dL/dz_t
 *   grad_mem [T,B,N] io_dtype or NULL    dL/du_t through the mem output
 *   grad_mem_final fp32 [B,N] or NULL    dL/du_{T-1} through mem_final
 * Outputs:
 *   grad_I   [T,B,N] io_dtype            dL/dI_t
 *   grad_beta, grad_thr fp32, parameter's shape, or NULL; summed over t and
 *            over the lanes that share the parameter
 *   grad_mem0 fp32 [B,N] or NULL         dL/du_{-1}
 * Reverse recurrence, with s_t = surrogate(u_t - thr):
 *   dz_t = grad_spk_t + [not detach] * (d u_{t+1}/d z_t) * du_{t+1}
 *   du_t = grad_mem_t + (d u_{t+1}/d u_t) * du_{t+1} + s_t * dz_t
 * where d u_{t+1}/d u_t = beta (subtract/none) or beta*(1-z_t) (zero) and
 * d u_{t+1}/d z_t = -thr (subtract), -beta*u_t (zero), 0 (none).
 * Parameter sums are accumulated in fp32 per lane and reduced across lanes
 * in a fixed order (deterministic): runs of a few lanes in fp32, everything
 * above them in compensated fp32 (a sum and the rounding error of its
 * additions, two-sum).
 * SNN_SAVE_RECOMPUTE replays Eq. (4) from each checkpoint bit for bit as the
 * forward evaluated it.  With ckpt_every 8 (any dtype pair), 12 or 16 (bf16
 * or fp16 input and io), no grad_mem, a reset other than SNN_RESET_NONE and B*N
 * a multiple of 8, the replayed segment stays in registers and a segment's
 * rows stream in whole (the fast path); otherwise the replay goes through
 * shared memory.  Both give the same spikes and trace, and gradients within
 * fp32 rounding of each other.
 */
snn_status_t snn_leaky_bwd(const snn_scan_desc* desc, const void* I, const float* ckpt,
                           const void* mem, const void* spk, const float* beta,
                           const float* thr, const float* mem0, const void* grad_spk,
                           const void* grad_mem, const float* grad_mem_final, void* grad_I,
                           float* grad_beta, float* grad_thr, float* grad_mem0, void* ws,
                           size_t ws_bytes, snn_stream_t stream);

/*
 * Current-based (Synaptic) LIF forward, Eqs. (3), (5), (6).  As
 * snn_leaky_fwd, plus:
 *   alpha    fp32, shape per alpha_mode  synaptic decay
 *   syn0     fp32 [B,N] or NULL          i_{-1} (NULL means 0)
 *   syn      [T,B,N] io_dtype (out) or NULL   i_t; needed by a SNN_SAVE_MEM
 *                                        backward that asks for grad_alpha
 *   syn_final fp32 [B,N] (out) or NULL   i_{T-1}
 * ckpt holds u then i for every checkpoint (2*B*N fp32 each).
 */
snn_status_t snn_synaptic_fwd(const snn_scan_desc* desc, const void* I, const float* alpha,
                              const float* beta, const float* thr, const float* mem0,
                              const float* syn0, void* spk, void* mem, void* syn,
                              float* ckpt, float* mem_final, float* syn_final, void* ws,
                              size_t ws_bytes, snn_stream_t stream);

/*
 * Synaptic BPTT.  As snn_leaky_bwd, plus:
 *   syn      [T,B,N] io_dtype            SNN_SAVE_MEM with grad_alpha != NULL
 *   grad_syn_final fp32 [B,N] or NULL    dL/di_{T-1}
 *   grad_alpha fp32 or NULL; grad_syn0 fp32 [B,N] or NULL
 *   di_t = alpha*di_{t+1} + du_t,  grad_I_t = di_t.
 */
snn_status_t snn_synaptic_bwd(const snn_scan_desc* desc, const void* I, const float* ckpt,
                              const void* mem, const void* spk, const void* syn,
                              const float* alpha, const float* beta, const float* thr,
                              const float* mem0, const float* syn0, const void* grad_spk,
                              const void* grad_mem, const float* grad_mem_final,
                              const float* grad_syn_final, void* grad_I, float* grad_alpha,
                              float* grad_beta, float* grad_thr, float* grad_mem0,
                              float* grad_syn0, void* ws, size_t ws_bytes,
                              snn_stream_t stream);

/*
 * Dense-layer input current, the synaptic operation w.x of Fig. 3 (Sec. III,
 * "the current injection term is replaced with a weighted input"), for all
 * T*B rows at once on the tcgen05 tensor cores:
 *   I[M, N] = X[M, K] * W[N, K]^T
 *   X  bf16 [M, K] row-major (M = T*B rows of layer input, e.g. spikes)
 *   W  bf16 [N, K] row-major (N outputs, K inputs; no bias)
 *   I  fp32 [M, N] row-major (out), fp32 accumulation
 *   ws device workspace of at least 256 bytes (status word, as for the scans)
 * K must be a multiple of 8 (16-byte rows for the tensor memory accelerator),
 * else SNN_ERR_UNSUPPORTED.  K = 0 writes zeros.
 */
snn_status_t snn_dense_layer_fwd(int64_t M, int64_t K, int64_t N, const void* X, const void* W,
                                 float* I, void* ws, size_t ws_bytes, snn_stream_t stream);

/* Workspace bytes of snn_dense_layer_bwd: a status word (the operands are
 * read in place, W and X and dI through MN-major tensor-core tiles), plus,
 * when dW's few output tiles would each sum a long M (a convolution's
 * weight gradient sums over every patch row), S fp32 partial copies of dW
 * [N, K]: the rows are split S ways, S a function of (M, K, N) alone, and
 * the partials are added in split order (the same bits on every call). */
size_t snn_dense_workspace_bytes(int64_t M, int64_t K, int64_t N);

/*
 * Backward of snn_dense_layer_fwd, given dI = dL/dI (bf16 [M, N], e.g. the
 * grad_I of a scan with bf16 io):
 *   dX bf16 [M, K] (out, or NULL) = dI * W          (input gradient)
 *   dW fp32 [N, K] (out, or NULL) = dI^T * X        (weight gradient)
 * M, K and N must be multiples of 8.  ws: snn_dense_workspace_bytes(M,K,N).
 */
snn_status_t snn_dense_layer_bwd(int64_t M, int64_t K, int64_t N, const void* X, const void* W,
                                 const void* dI, void* dX, float* dW, void* ws, size_t ws_bytes,
                                 snn_stream_t stream);

/*
 * Recurrent Leaky LIF forward, Eqs. (3) and (7): the spike of step t-1 is
 * fed back through a one-to-one recurrent weight v,
 *   u_t = beta*u_{t-1} + I_t + z_{t-1}*(v - thr),
 * evaluated as (beta*u_{t-1} + I_t) + z_{t-1}*(v - thr), each operation
 * rounded to nearest.  Arguments as snn_leaky_fwd, plus:
 *   v        fp32, shape per desc->alpha_mode (scalar, [N] or [C])
 * desc->reset must be SNN_RESET_SUBTRACT (Eq. 7 resets by subtraction),
 * else SNN_ERR_UNSUPPORTED.
 */
snn_status_t snn_rleaky_fwd(const snn_scan_desc* desc, const void* I, const float* v,
                            const float* beta, const float* thr, const float* mem0, void* spk,
                            void* mem, float* ckpt, float* mem_final, void* ws, size_t ws_bytes,
                            snn_stream_t stream);

/*
 * Recurrent Leaky LIF BPTT.  Arguments as snn_leaky_bwd, plus v and
 *   grad_v   fp32, v's shape, or NULL: dL/dv summed over t and the lanes
 *            sharing v (d u_{t+1}/d v = z_t).
 * The recurrent connection always carries gradient; detach_reset detaches
 * only the -z_{t-1}*thr part:
 *   dz_t = grad_spk_t + (v - [not detach]*thr) * du_{t+1}.
 */
snn_status_t snn_rleaky_bwd(const snn_scan_desc* desc, const void* I, const float* ckpt,
                            const void* mem, const void* spk, const float* v, const float* beta,
                            const float* thr, const float* mem0, const void* grad_spk,
                            const void* grad_mem, const float* grad_mem_final, void* grad_I,
                            float* grad_v, float* grad_beta, float* grad_thr, float* grad_mem0,
                            void* ws, size_t ws_bytes, snn_stream_t stream);

/*
 * Rate-coded readout loss (Sec. V-A: the predicted class is the output
 * neuron, or with a population code (Sec. VII) the population of pop
 * neurons, that fires most): cross-entropy of the spike counts over T.
 *   spk   [T, B, ld] in `dtype` (snn_dtype_t); the first C*pop of ld
 *         neurons are the classes' populations, class c owning neurons
 *         c*pop .. c*pop + pop - 1 (C <= 1024, pop >= 1, C*pop <= 32768)
 *   labels int32 [B]
 *   batch_total  the batch the mean is taken over: 0 for B; the global batch
 *         (>= B) when these B samples are one data-parallel shard, so that
 *         the shards' losses and gradients add up to the global ones
 *   loss  fp32 [1] (out) = sum_b CE(counts_b, y_b) / batch_total, with
 *         counts_b[c] = sum_t sum_j spk[t, b, c*pop + j]
 *   grad_spk [T, B, ld] (out) = (softmax - onehot)[class of the neuron] /
 *         batch_total for every t; 0 for neurons C*pop .. ld-1
 *   ws    device workspace of snn_rate_ce_workspace_bytes(B) bytes, 16-byte
 *         aligned, zeroed once before the first call (every call leaves its
 *         completion ticket at zero; re-zero after an error)
 * One block per sample; the loss terms are added in a fixed order
 * (deterministic).
 */
size_t snn_rate_ce_workspace_bytes(int64_t B);
snn_status_t snn_rate_ce_loss(int64_t T, int64_t B, int64_t C, int64_t pop, int64_t ld,
                              int64_t batch_total, int32_t dtype, const void* spk,
                              const int32_t* labels, float* loss, void* grad_spk, void* ws,
                              size_t ws_bytes, snn_stream_t stream);

/*
 * The rate-coded loss of snn_rate_ce_loss fused with the BPTT of the
 * readout layer that produced spk (a Leaky layer, Eq. 4; reverse pass of
 * Sec. III-B): the spike gradient of every output neuron is the loss
 * gradient above, and the same launch runs the neuron's reverse scan on the
 * stored trace and writes its dL/dI.
 *   desc  the readout layer: T, B, N = ld neurons per sample, io_dtype (any),
 *         save SNN_SAVE_MEM, any reset, detach and surrogate; beta_mode and
 *         thr_mode scalar or per neuron (of ld)
 *   C, pop, batch_total, labels, loss, ws   as for snn_rate_ce_loss
 *   spk   [T, B, ld] the layer's spikes (io dtype); also the spike decisions
 *         of the reverse scan unless ckpt is given
 *   mem   [T, B, ld] the layer's stored membrane trace (io dtype)
 *   ckpt  the spike bits its store-mode forward wrote, or NULL
 *   grad_spk [T, B, ld] (out, nullable): the loss gradient, as written by
 *         snn_rate_ce_loss
 *   grad_I [T, B, ld] (out): the readout's dL/dI (io dtype)
 * No parameter or initial-state gradients (snn_leaky_bwd gives those).
 */
snn_status_t snn_rate_ce_leaky_bwd(const snn_scan_desc* desc, int64_t C, int64_t pop,
                                   int64_t batch_total, const void* spk, const int32_t* labels,
                                   const float* beta, const float* thr, const void* mem,
                                   const float* ckpt, float* loss, void* grad_spk, void* grad_I,
                                   void* ws, size_t ws_bytes, snn_stream_t stream);

/*
 * Dense layer fused with its Leaky scan (Fig. 3's synaptic operation w.x
 * feeding Eqs. 3-4): the currents of all T steps come out of one tcgen05
 * GEMM and are scanned in its epilogue, so they never reach HBM.
 *   desc     the Leaky layer: T <= 128, B, N = P*Nout neurons per sample
 *            (channel-last: neuron p*Nout + n is output column n at row p),
 *            io_dtype SNN_BF16, save SNN_SAVE_MEM (the BPTT reads the stored
 *            trace: snn_leaky_bwd in store mode), any reset; beta_mode and
 *            thr_mode scalar, per neuron (P = 1) or per channel with
 *            C = Nout, HW = 1.  Nout and K multiples of 8.
 *   X        bf16 [T, B*P, K]: row (t, r) of the layer input (r = b*P + p)
 *   W        bf16 [Nout, K]
 *   spk, mem bf16 [T, B, N] (out): z_t and u_t, as snn_leaky_fwd writes them
 *   ckpt     the spike bits of store mode (see snn_scan_ckpt_elems), or NULL
 *   ws       at least 256 bytes (status word)
 * Initial state zero (no mem0); mem_final is not produced.  Returns
 * SNN_ERR_UNSUPPORTED for other modes or shapes.
 */
snn_status_t snn_dense_leaky_fwd(const snn_scan_desc* desc, int64_t P, int64_t K, const void* X,
                                 const void* W, const float* beta, const float* thr, void* spk,
                                 void* mem, float* ckpt, void* ws, size_t ws_bytes,
                                 snn_stream_t stream);

/*
 * The dense backward fused with the BPTT of the layer below (the converse of
 * snn_dense_leaky_fwd): the product dX = dI_up * W of the layer above, whose
 * rows are the spike gradients dL/dz_t of this layer, is computed on the
 * tcgen05 tensor cores and this layer's reverse scan (Sec. III-B, the
 * store-mode arithmetic of snn_leaky_bwd) runs on it in the epilogue; the
 * spike gradient is neither rounded nor written.
 *   desc    this (lower) Leaky layer: T <= 128, B, N neurons (multiple of 8),
 *           io_dtype SNN_BF16, save SNN_SAVE_MEM, any reset, detach and
 *           surrogate; beta_mode / thr_mode scalar or per neuron
 *   dI_up   bf16 [T*B, K]: dL/dI of the layer above (K its neurons, multiple
 *           of 8)
 *   W       bf16 [K, N]: the layer above's weights (its [N_out, K_in] matrix)
 *   mem     bf16 [T, B, N] stored trace; ckpt its spike bits, or NULL with
 *           spk bf16 [T, B, N] instead
 *   grad_I  bf16 [T, B, N] (out): this layer's dL/dI
 * No grad_mem, grad_mem_final, mem0 or parameter gradients (use
 * snn_leaky_bwd for those).  ws: at least 256 bytes.
 */
snn_status_t snn_dense_leaky_bwd(const snn_scan_desc* desc, int64_t K, const void* dI_up,
                                 const void* W, const float* beta, const float* thr,
                                 const void* mem, const void* spk, const float* ckpt,
                                 void* grad_I, void* ws, size_t ws_bytes, snn_stream_t stream);

/*
 * Convolutional SNN layout kernels (Tab. I CSNN: 5x5 convolutions, 2x2 max
 * pooling) on channel-last bf16 activations [M, H, W, C], M = T*B.  A
 * convolution is a snn_dense_layer_fwd/bwd over the patch rows:
 *   snn_im2col_nhwc: cols [M*Ho*Wo, Kpad] (out), Ho = H-KH+1, Wo = W-KW+1,
 *     cols[(m, oy, ox), (ky*KW + kx)*Cin + c] = X[m, oy+ky, ox+kx, c], zero
 *     for columns KH*KW*Cin .. Kpad-1 (Kpad a multiple of 8, >= KH*KW*Cin;
 *     cols 16-byte aligned).  With filters W [Cout, Kpad] (same column
 *     order), snn_dense_layer_fwd(cols, W) is the valid, stride-1
 *     convolution.
 *   snn_col2im_nhwc: dX [M, H, W, Cin] (out) = the patch-row gradient dcols
 *     [M*Ho*Wo, Kpad] summed back onto the input pixels each column read
 *     (fp32 sums in (ky, kx) order, rounded to bf16).
 *   snn_maxpool2_fwd_nhwc: Y [M, H/2, W/2, C] (out) = the maximum of each
 *     2x2 window (H, W even); idx uint8 [M, H/2, W/2, C] (out) = the
 *     window position (0..3, row major) of its first maximum.
 *   snn_maxpool2_bwd_nhwc: dX [M, H, W, C] (out) = dY at the recorded
 *     position of each window, 0 at the other three.
 * Asynchronous on stream; SNN_ERR_INVALID_ARG / SNN_ERR_ALIGNMENT for bad
 * shapes or pointers.
 */
snn_status_t snn_im2col_nhwc(int64_t M, int64_t H, int64_t W, int64_t Cin, int64_t KH, int64_t KW,
                             int64_t Kpad, const void* X, void* cols, snn_stream_t stream);
snn_status_t snn_col2im_nhwc(int64_t M, int64_t H, int64_t W, int64_t Cin, int64_t KH, int64_t KW,
                             int64_t Kpad, const void* dcols, void* dX, snn_stream_t stream);
snn_status_t snn_maxpool2_fwd_nhwc(int64_t M, int64_t H, int64_t W, int64_t C, const void* X,
                                   void* Y, uint8_t* idx, snn_stream_t stream);
snn_status_t snn_maxpool2_bwd_nhwc(int64_t M, int64_t H, int64_t W, int64_t C, const void* dY,
                                   const uint8_t* idx, void* dX, snn_stream_t stream);

/*
 * Convolution with few input channels on the CUDA cores (the CSNN's first
 * layer, Tab. I: 5x5 filters over the 1-channel input map), where the patch
 * rows of a GEMM would be mostly padding: KH*KW*Cin <= 32, Cout <= 16 and a
 * multiple of 4, H*W*Cin <= 8192 (else SNN_ERR_UNSUPPORTED).
 *   X  bf16 [M, H, W, Cin] channel-last;  Wt bf16 [Cout, ldw] filters with
 *      column k = (ky*KW + kx)*Cin + c (the im2col order), ldw >= KH*KW*Cin
 *   snn_conv2d_small_fwd_nhwc: I fp32 [M, Ho, Wo, Cout] (out, 16-byte
 *      aligned) = the valid stride-1 convolution, fp32 fused multiply-adds
 *      in k order
 *   snn_conv2d_small_dw_nhwc: dW fp32 [Cout, ldw] (out; 0 past column K) =
 *      sum over (m, oy, ox) of dI[m, oy, ox, o] * X[m, oy+ky, ox+kx, c] for
 *      dI bf16 [M, Ho, Wo, Cout]; a fixed number of blocks each sum a fixed
 *      set of images, the block partials (ws, at least
 *      snn_conv2d_small_dw_workspace_bytes, 16-byte aligned) are added in
 *      block order: the same bits on every call
 * Asynchronous on stream.
 */
snn_status_t snn_conv2d_small_fwd_nhwc(int64_t M, int64_t H, int64_t W, int64_t Cin, int64_t Cout,
                                       int64_t KH, int64_t KW, int64_t ldw, const void* X,
                                       const void* Wt, float* I, snn_stream_t stream);
size_t snn_conv2d_small_dw_workspace_bytes(int64_t M, int64_t H, int64_t W, int64_t Cin,
                                           int64_t Cout, int64_t KH, int64_t KW);
snn_status_t snn_conv2d_small_dw_nhwc(int64_t M, int64_t H, int64_t W, int64_t Cin, int64_t Cout,
                                      int64_t KH, int64_t KW, int64_t ldw, const void* X,
                                      const void* dI, float* dW, void* ws, size_t ws_bytes,
                                      snn_stream_t stream);

/*
 * AdamW update of n fp32 master weights (the optimiser of the paper's
 * training runs, Sec. V; decoupled weight decay):
 *   m <- beta1 m + (1 - beta1) g ;  v <- beta2 v + (1 - beta2) g^2
 *   w <- w (1 - lr weight_decay) - lr / (1 - beta1^step) * m / (sqrt(v / (1 - beta2^step)) + eps)
 *   w, m, v  fp32 [n] (in/out, device);  grad fp32 [n] (in)
 *   w_bf16   bf16 [n] (out, or NULL): the updated weights rounded to bf16
 *            (round to nearest even) for the next forward GEMM
 *   step     1 for the first update (used when step_counter is NULL)
 *   step_counter  device int64 [2], or NULL: {updates done, 0}, zeroed by the
 *            caller before the first update.  The launch then uses step =
 *            step_counter[0] + 1 and advances step_counter[0] itself, so a
 *            captured CUDA graph replays successive steps.  One counter per
 *            parameter buffer; launches sharing a counter must not overlap.
 * All pointers 16-byte aligned (SNN_ERR_ALIGNMENT); step < 1 without a
 * counter, beta outside (0, 1) or eps <= 0 give SNN_ERR_INVALID_ARG.
 * Asynchronous on stream.
 */
snn_status_t snn_adamw_step(int64_t n, float* w, void* w_bf16, const float* grad, float* m,
                            float* v, float lr, float beta1, float beta2, float eps,
                            float weight_decay, int64_t step, int64_t* step_counter,
                            snn_stream_t stream);

/*
 * Leaky BPTT that allocates nothing (no counterpart in the paper; it exists
 * for callers of this library that cannot allocate device memory: hosts
 * whose device memory is budgeted by another runtime, real-time loops that
 * must not call cudaMalloc because it can synchronise the device, plain C
 * hosts without an allocator).
 * Arguments and results are those of snn_leaky_bwd, without ws/ws_bytes:
 * the workspace is a fixed 16 MiB array in the library's device memory,
 * held by every GPU that loads the library until the process exits.
 *   status   device int (4-byte aligned) or NULL: receives SNN_OK or
 *            SNN_ERR_TIMEOUT from the kernels (asynchronously, on stream)
 * Argument checks and their order are those of snn_leaky_bwd; a request
 * whose snn_scan_workspace_bytes(desc) exceeds 16 MiB fails them with
 * SNN_ERR_WORKSPACE, launching nothing.  Allocates nothing.
 * The first call on each device looks up the array's device address (a
 * one-time set-up that is not a stream operation); make that first call
 * before any stream capture.  Every call shares the one array and it keeps
 * the last call's contents.  Each call zeroes, on stream and before its
 * kernels, the status word and every completion ticket its reductions take,
 * so a call is correct whatever the previous call's shape or parameter
 * layouts were and after a call that reported SNN_ERR_TIMEOUT.  Calls whose
 * work overlaps on the GPU (other streams, other host threads) race on the
 * array and must be serialised by the caller.
 */
snn_status_t snn_leaky_bwd_noalloc(const snn_scan_desc* desc, const void* I, const float* ckpt,
                                   const void* mem, const void* spk, const float* beta,
                                   const float* thr, const float* mem0, const void* grad_spk,
                                   const void* grad_mem, const float* grad_mem_final,
                                   void* grad_I, float* grad_beta, float* grad_thr,
                                   float* grad_mem0, int* status, snn_stream_t stream);

#if defined(__GNUC__)
#pragma GCC visibility pop
#endif
#ifdef __cplusplus
}
#endif
#endif /* SNN_H_ */
