// Fused temporal-scan kernels for the Leaky (Eq. 4) and Synaptic (Eqs. 5-6)
// neurons of arXiv 2211.10725, forward and BPTT (Sec. II-A/B, III-B).
//
// Layout: every [T, B, N] tensor is t-major, so the L = B*N lanes of one step
// are contiguous.  A lane is independent of every other lane and sequential
// in t: each thread owns 8 (Leaky) or 4 (Synaptic) consecutive lanes and keeps their state (u, i,
// z and, backward, the adjoints) in registers for the whole scan.
//
// Staged kernels (the fast path): a CTA owns a contiguous strip of lanes.
// One producer thread streams the strip's row of every input tensor, step by
// step, into a ring of shared-memory stages with 1-D bulk copies (TMA,
// cp.async.bulk) completing on a "full" mbarrier per stage; the consumer
// warps wait on it, read their lanes, compute and store the step, and only
// then release the stage on its "empty" mbarrier.  The ring depth, not the
// thread count, supplies the bytes in flight that HBM needs.  Ring position
// (stage index and phase parity) advances incrementally: no division in the
// loop.  Reset mode and surrogate are template parameters (-1 = read at run
// time) so the specialised loops carry no mode branches.
//
// Plain kernels: one lane per thread, direct loads; taken for shapes whose
// rows are not 16-byte multiples.  Both use the same per-lane step code, so
// they give bit-identical forward results.
#pragma once

#include "launch.cuh"
#include "snn_device.cuh"

namespace snn {

enum { RESET_SUBTRACT = 0, RESET_ZERO = 1, RESET_NONE = 2 };
enum { SG_FAST_SIGMOID = 0, SG_ATAN = 1 };
enum { PM_SCALAR = 0, PM_PER_NEURON = 1, PM_PER_CHANNEL = 2 };
constexpr uint32_t DEBUG_PRODUCER_IDLE = 1u;
constexpr uint32_t DEBUG_NO_SEGMENT = 4u;
constexpr int VEC = 8;                 // lane granularity of a staged CTA strip
constexpr int kBarrierBytes = 1024;    // full[60], empty[60], ck_full[2], ck_empty[2]
constexpr int kMaxStages = 60;
constexpr int kMaxStagedThreads = 512;
constexpr uint64_t kDrainNs = 1000000000ull;

struct ScanArgs {
  int64_t T, L, N, C, HW;
  int K;      // checkpoint interval (recompute); T in store mode
  int nseg;   // ceil(T / K)
  int reset, detach, sg;
  int rec;           // recurrent Leaky neuron (Eq. 7): alpha holds v, part_alpha dv
  float sg_a, sg_b;  // fast sigmoid: a = slope; atan: a = alpha/2, b = pi*alpha/2
  int beta_mode, thr_mode, alpha_mode;
  const float* beta;
  const float* thr;
  const float* alpha;
  const float* mem0;
  const float* syn0;
  // forward
  const void* I;
  void* spk;
  void* mem;
  void* syn;
  float* ckpt;  // forward: written; backward: read
  // store mode, half io: spike bits (bit k of byte j of row t = z_t of lane
  // 8j + k), rows of bits_row bytes; forward: written; backward: read
  unsigned char* bits;
  int64_t bits_row;
  float* mem_final;
  float* syn_final;
  // backward
  const void* spk_in;
  const void* mem_in;
  const void* syn_in;
  const void* gs;
  const void* gm;
  const float* gmf;
  const float* gsf;
  void* gI;
  float* part_beta;  // per-lane parameter-gradient partials (workspace) or null
  float* part_thr;
  float* part_alpha;
  float* gmem0;
  float* gsyn0;
  // control
  int* status;
  uint64_t wait_ns;
  uint32_t debug;
  // staged tiling
  int lanes_per_cta;
  int stages;
  int stage_bytes;
};

// ---------------------------------------------------------------------------
// Per-lane arithmetic
// ---------------------------------------------------------------------------

__device__ __forceinline__ float lane_param(const float* p, int mode, int64_t l,
                                            const ScanArgs& a) {
  if (mode == PM_SCALAR) return __ldg(p);
  const int64_t n = l % a.N;
  if (mode == PM_PER_NEURON) return __ldg(p + n);
  return __ldg(p + (n / a.HW) % a.C);
}

// Checkpoint segments are aligned to the end of the sequence: segment k of
// nseg covers [t0, t1) with t1 = r + k*K, r = T - (nseg-1)*K, so only the
// first segment (k = 0, starting at t = 0) can be shorter than K.  The
// forward stores u (and i) at t1 - 1 of every segment but the last.
__device__ __forceinline__ void seg_bounds(const ScanArgs& a, int k, int64_t& t0, int64_t& t1) {
  const int64_t r = a.T - (int64_t)(a.nseg - 1) * a.K;
  t1 = r + (int64_t)k * a.K;
  t0 = k == 0 ? 0 : t1 - a.K;
}

// Position inside its checkpoint segment of step t = 0: the forward's step
// counter starts here so that its segment ends fall at t1 - 1.
__device__ __forceinline__ int seg_phase0(const ScanArgs& a) {
  return (int)(a.K - (a.T - (int64_t)(a.nseg - 1) * a.K));
}

// One forward step, Eq. (4) / Eqs. (5)-(6), evaluated left to right as the
// equations are written, one rounded fp32 operation at a time (no FMA that
// would fuse two of them), so the forward and the backward's recomputation
// agree bit for bit.  The subtract reset u - z*thr is one rounding since
// z*thr is exact (z in {0,1}); reset-to-zero scales u by (1 - z) exactly.
template <bool SYN, int RESET, int REC = 0>
__device__ __forceinline__ void fwd_step(int reset_rt, float beta, float thr, float alpha,
                                         float x, float& u, bool& z, float& i,
                                         bool rec_rt = false) {
  const int reset = RESET >= 0 ? RESET : reset_rt;
  const bool rec = REC > 0 || (REC < 0 && rec_rt);  // Eq. (7): alpha is v
  float in = x;
  if (SYN) {
    i = __fadd_rn(__fmul_rn(alpha, i), x);
    in = i;
  }
  float un;
  if (reset == RESET_ZERO) {
    // (1 - z) u: u, or a zero with u's sign (as the float evaluation gives)
    un = __fadd_rn(__fmul_rn(beta, z ? __fmul_rn(u, 0.0f) : u), in);
  } else {
    un = __fadd_rn(__fmul_rn(beta, u), in);
    if (reset == RESET_SUBTRACT && z) un = rec ? __fadd_rn(un, __fsub_rn(alpha, thr)) : __fsub_rn(un, thr);
  }
  u = un;
  z = un > thr;  // Eq. (3), strict
}

// Surrogate dz/du at x = u - thr (Sec. III-B).
template <int SG>
__device__ __forceinline__ float surrogate(const ScanArgs& a, float x) {
  const int sg = SG >= 0 ? SG : a.sg;
  if (sg == SG_FAST_SIGMOID) {
    const float d = fmaf(a.sg_a, fabsf(x), 1.0f);
    return __fdividef(1.0f, d * d);
  }
  const float y = a.sg_b * x;
  return __fdividef(a.sg_a, fmaf(y, y, 1.0f));
}

struct BwdLane {
  float du;      // dL/du_{t+1} on entry to step t, dL/du_t on exit
  float di;      // dL/di_{t+1} -> dL/di_t (Synaptic)
  float dbeta, dthr, dalpha;
};

// One reverse step at time t.  u, z, i are u_t, z_t, i_t.  First the
// parameter terms of step t+1 that need the step-t state
// (d u_{t+1}/d beta = u_t or (1-z_t) u_t, the subtract reset's -z_t, and
// d i_{t+1}/d alpha = i_t), then the adjoint of step t.  Returns dL/dI_t.
template <bool SYN, int RESET, int SG>
__device__ __forceinline__ float bwd_step(const ScanArgs& a, float beta, float thr, float alpha,
                                          bool has_next, float u, bool z, float i, float gs,
                                          float extra_u, float extra_i, BwdLane& s) {
  const int reset = RESET >= 0 ? RESET : a.reset;
  if (has_next) {
    s.dbeta = fmaf(s.du, (reset == RESET_ZERO && z) ? 0.0f : u, s.dbeta);
    if (reset == RESET_SUBTRACT && z) s.dthr -= s.du;
    if (SYN) s.dalpha = fmaf(s.di, i, s.dalpha);
    if (!SYN && a.rec && z) s.dalpha += s.du;  // dv: d u_{t+1} / d v = z_t
  }
  const float sgv = surrogate<SG>(a, u - thr);
  float dz = gs;
  if (!a.detach) {
    if (reset == RESET_SUBTRACT) dz = fmaf(-thr, s.du, dz);
    else if (reset == RESET_ZERO) dz = fmaf(-beta * u, s.du, dz);
  }
  if (!SYN && a.rec) dz = fmaf(alpha, s.du, dz);  // the recurrent connection, never detached
  const float decay = (reset == RESET_ZERO && z) ? 0.0f : beta;
  const float du = fmaf(decay, s.du, fmaf(sgv, dz, extra_u));
  s.dthr = fmaf(-sgv, dz, s.dthr);
  s.du = du;
  if (SYN) {
    s.di = fmaf(alpha, s.di, du + extra_i);
    return s.di;
  }
  return du;
}

// Terms of the initial state (step t = -1): u_{-1} = mem0 (or 0),
// z_{-1} = [mem0 > thr] when mem0 is given, else 0.
template <bool SYN>
__device__ __forceinline__ void bwd_initial(const ScanArgs& a, float beta, float thr,
                                            float alpha, bool have_mem0, float u_m1,
                                            float i_m1, BwdLane& s, float& gmem0,
                                            float& gsyn0) {
  const bool z_m1 = have_mem0 && (u_m1 > thr);
  const bool rec = !SYN && a.rec;
  s.dbeta = fmaf(s.du, (a.reset == RESET_ZERO && z_m1) ? 0.0f : u_m1, s.dbeta);
  if (a.reset == RESET_SUBTRACT && z_m1) s.dthr -= s.du;
  if (SYN) s.dalpha = fmaf(s.di, i_m1, s.dalpha);
  if (rec && z_m1) s.dalpha += s.du;
  const float decay = (a.reset == RESET_ZERO && z_m1) ? 0.0f : beta;
  gmem0 = decay * s.du;
  if (have_mem0 && ((!a.detach && a.reset != RESET_NONE) || rec)) {
    const float sgv = surrogate<-1>(a, u_m1 - thr);
    float slope = 0.0f;
    if (!a.detach && a.reset != RESET_NONE) slope = (a.reset == RESET_SUBTRACT) ? -thr : -beta * u_m1;
    if (rec) slope += alpha;
    const float dz = slope * s.du;
    gmem0 = fmaf(sgv, dz, gmem0);
    s.dthr = fmaf(-sgv, dz, s.dthr);
  }
  gsyn0 = SYN ? alpha * s.di : 0.0f;
}

// ---------------------------------------------------------------------------
// Packed pairs of lanes (Blackwell fp32x2: one instruction, two IEEE-rounded
// lane results), used by the staged kernels
// ---------------------------------------------------------------------------

__device__ __forceinline__ float2 f2(float a) { return make_float2(a, a); }
__device__ __forceinline__ float2 add2(float2 a, float2 b) { return __fadd2_rn(a, b); }
__device__ __forceinline__ float2 mul2(float2 a, float2 b) { return __fmul2_rn(a, b); }
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }

// Packed fp32x2 add and multiply, round to nearest: one instruction, two
// correctly rounded lane results.  Measured on sm_103a: a packed multiply
// whose product feeds a packed add is contracted into a packed fused
// multiply-add (about half of all results then differ in the last bit), even
// when both are written in PTX with explicit .rn modifiers, while a scalar
// __fmul_rn product feeding a packed add is not.  So a product that is added
// to something else is formed with scalar __fmul_rn (mul_rn_pair); the packed
// multiply is used only where the product is exact (a spike 0/1 times a
// value), where a fused rounding gives the same result.
__device__ __forceinline__ float2 add2_rn(float2 a, float2 b) { return __fadd2_rn(a, b); }
__device__ __forceinline__ float2 mul_rn_pair(float2 a, float2 b) {
  return make_float2(__fmul_rn(a.x, b.x), __fmul_rn(a.y, b.y));
}
__device__ __forceinline__ float2 mul2_rn(float2 a, float2 b) { return __fmul2_rn(a, b); }

// Eq. (3) as a float: 1.0f where u > thr, else 0.0f (NaN gives 0).
__device__ __forceinline__ float fire(float u, float thr) {
  float d;
  asm("set.gt.f32.f32 %0, %1, %2;" : "=f"(d) : "f"(u), "f"(thr));
  return d;
}
__device__ __forceinline__ float2 fire2(float2 u, float2 negthr) {
  return make_float2(fire(u.x, -negthr.x), fire(u.y, -negthr.y));
}

// Forward step on a pair of lanes, the packed form of fwd_step: Eq. (4) /
// Eqs. (5)-(6) left to right, one correctly rounded operation at a time, so
// it is bit-identical to fwd_step (and to the float32 evaluation of the
// equations).  z holds z_{t-1} on entry and z_t on exit as 0.0f / 1.0f.
//   subtract   u = ((beta*u) + in) + z*(-thr)   z*(-thr) is exact: -thr or -0,
//              and adding -0 leaves every value (signed zeros included) as is;
//              one fused multiply-add, which rounds the same single sum
//   zero       u = (beta*((1-z)*u)) + in        (1-z)*u is u or a zero of u's sign
//   none       u = (beta*u) + in
//   Eq. (7)    u = ((beta*u) + in) + z*vmt      vmt = v - thr, rounded once
// For the Synaptic neuron in = i = (alpha*i) + x first.  `third` is alpha
// (Synaptic) or vmt (recurrent Leaky).
template <bool SYN, int RESET, int REC = 0>
__device__ __forceinline__ void fwd_pair(int reset_rt, float2 beta, float2 negthr, float2 third,
                                         float2 x, float2& u, float2& z, float2& i) {
  const int reset = RESET >= 0 ? RESET : reset_rt;
  float2 in = x;
  if (SYN) {
    i = add2_rn(mul_rn_pair(third, i), x);
    in = i;
  }
  float2 un;
  if (reset == RESET_ZERO) {
    const float2 keep = mul2_rn(make_float2(1.0f - z.x, 1.0f - z.y), u);  // exact
    un = add2_rn(mul_rn_pair(beta, keep), in);
  } else {
    un = add2_rn(mul_rn_pair(beta, u), in);
    // z*(-thr) (or z*vmt) is exact, so the fused z*(-thr) + un rounds once,
    // exactly as the separate add of the exact product
    if (REC > 0) un = fma2(z, third, un);
    else if (reset == RESET_SUBTRACT) un = fma2(z, negthr, un);
  }
  u = un;
  z = fire2(un, negthr);
}

// Approximate reciprocal (one hardware instruction, relative error ~2^-23)
// of a surrogate's denominator (>= 1, or >= 1/a for the arctan form with
// a = alpha/2), so no subnormal occurs.
__device__ __forceinline__ float rcp_ge1(float d) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(d));
  return r;
}

template <int SG>
__device__ __forceinline__ float2 surrogate2(const ScanArgs& a, float2 x) {
  const int sg = SG >= 0 ? SG : a.sg;
  if (sg == SG_FAST_SIGMOID) {
    const float2 d = fma2(f2(a.sg_a), make_float2(fabsf(x.x), fabsf(x.y)), f2(1.0f));
    const float2 d2 = mul2(d, d);
    return make_float2(rcp_ge1(d2.x), rcp_ge1(d2.y));
  }
  const float2 y = mul2(f2(a.sg_b), x);
  const float2 d = fma2(y, y, f2(1.0f));
  return mul2(f2(a.sg_a), make_float2(rcp_ge1(d.x), rcp_ge1(d.y)));
}

// Reverse-pass state of a pair of lanes.  dthr accumulates
// +(sigma'*dz + z_t*du_{t+1}); the threshold gradient is its negation.
struct Bwd2 {
  float2 du, di, dbeta, dthr, dalpha;
};

// One reverse step at time t on a pair of lanes (u, z, i = u_t, z_t, i_t).
// du/di hold dL/du_{t+1}, dL/di_{t+1} on entry (zero at t = T-1, so the
// parameter terms of step t+1 vanish there) and dL/du_t, dL/di_t on exit.
// EXTRA adds eu to dL/du_t and ei to dL/di_t (grad_mem every step,
// grad_mem_final / grad_syn_final at t = T-1).  Returns dL/dI_t.
template <bool SYN, int RESET, int SG, bool EXTRA, bool REC = false>
__device__ __forceinline__ float2 bwd_pair(const ScanArgs& a, float2 beta, float2 negthr,
                                           float2 alpha, float2 u, bool z0, bool z1, float2 i,
                                           float2 gs, float2 eu, float2 ei, Bwd2& s) {
  const int reset = RESET >= 0 ? RESET : a.reset;
  if (reset == RESET_ZERO) {
    s.dbeta = fma2(s.du, make_float2(z0 ? 0.0f : u.x, z1 ? 0.0f : u.y), s.dbeta);
  } else {
    s.dbeta = fma2(s.du, u, s.dbeta);
  }
  if (reset == RESET_SUBTRACT) {  // d u_{t+1} / d thr = -z_t
    if (z0) s.dthr.x += s.du.x;
    if (z1) s.dthr.y += s.du.y;
  }
  if (REC) {  // d u_{t+1} / d v = z_t (Eq. 7)
    if (z0) s.dalpha.x += s.du.x;
    if (z1) s.dalpha.y += s.du.y;
  }
  if (SYN) s.dalpha = fma2(s.di, i, s.dalpha);
  const float2 sg = surrogate2<SG>(a, add2(u, negthr));
  float2 dz = gs;
  if (!a.detach) {
    if (reset == RESET_SUBTRACT) dz = fma2(negthr, s.du, dz);
    else if (reset == RESET_ZERO) dz = fma2(mul2(f2(-1.0f), mul2(beta, u)), s.du, dz);
  }
  if (REC) dz = fma2(alpha, s.du, dz);  // the recurrent connection, never detached
  const float2 p = mul2(sg, dz);
  const float2 decay = reset == RESET_ZERO
                           ? make_float2(z0 ? 0.0f : beta.x, z1 ? 0.0f : beta.y)
                           : beta;
  s.du = fma2(decay, s.du, p);
  if (EXTRA) s.du = add2(s.du, eu);
  s.dthr = add2(s.dthr, p);
  if (SYN) {
    s.di = fma2(alpha, s.di, s.du);
    if (EXTRA) s.di = add2(s.di, ei);
    return s.di;
  }
  return s.du;
}

// ---------------------------------------------------------------------------
// Ring of shared-memory stages
// ---------------------------------------------------------------------------

// Stage index and phase parity of the next item; items are consumed in order.
struct RingPos {
  int s = 0;
  uint32_t ph = 0;
  __device__ __forceinline__ void next(int S) {
    if (++s == S) {
      s = 0;
      ph ^= 1u;
    }
  }
};

// Warp-uniform bounded wait: every lane polls the barrier (so every lane
// acquires the completed phase); the decision to give up is taken by lane 0's
// clock (read every 64 polls) and shared, so the warp never diverges around it.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  bool done = mbar_try_wait(bar, parity);
  if (__all_sync(0xffffffffu, done)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {  // i is warp-uniform
    if (!done) done = mbar_try_wait(bar, parity);
    if (__all_sync(0xffffffffu, done)) return true;
    if ((i & 63u) == 0) {  // the clock every 64 polls
      uint64_t el = globaltimer_ns() - t0;
      el = __shfl_sync(0xffffffffu, el, 0);
      if (el > limit_ns) return false;
    }
  }
}

// The single producer thread: fills stage after stage once the consumers
// have released it, and drains its copies before the CTA may exit.
struct Producer {
  unsigned char* ring;
  uint64_t* full;
  uint64_t* empty;
  int S;
  int stage_bytes;
  RingPos pos;
  bool wrapped = false;  // the ring has been filled once: wait for releases
  int64_t issued = 0;
  bool ok = true;

  // One item in three calls: begin() waits (bounded) for the consumers'
  // release of the stage's previous round and announces the item's total
  // bytes on its full barrier, copy() issues one bulk copy into the stage,
  // end() moves to the next stage.  Items are built in place, with no
  // array of copy descriptors in local memory.
  __device__ __forceinline__ bool begin(uint32_t total, const ScanArgs& a) {
    if (!ok) return false;
    if (wrapped && !mbar_wait_spin(&empty[pos.s], pos.ph ^ 1u, a.wait_ns)) {
      record_status(a.status, kStatusTimeout);
      ok = false;
      return false;
    }
    mbar_arrive_expect_tx(&full[pos.s], total);
    return true;
  }
  __device__ __forceinline__ void copy(uint32_t dst, const void* src, uint32_t bytes) {
    bulk_g2s(ring + (size_t)pos.s * stage_bytes + dst, src, bytes, &full[pos.s]);
  }
  __device__ __forceinline__ void end() {
    ++issued;
    pos.next(S);
    if (pos.s == 0) wrapped = true;
  }

  // Wait (bounded) until the last copy into every stage has landed.
  __device__ __forceinline__ void drain() {
    const int64_t first = issued > S ? issued - S : 0;
    for (int64_t j = first; j < issued; ++j)
      mbar_wait_bounded(&full[j % S], (uint32_t)((j / S) & 1), kDrainNs);
  }
};

template <typename T>
__device__ __forceinline__ const void* row(const void* base, int64_t t, int64_t L, int64_t lane0) {
  return static_cast<const T*>(base) + t * L + lane0;
}

// Barrier block at the start of shared memory: the ring's full/empty pairs
// and the two-slot checkpoint buffer's pairs (recompute backward).
__device__ __forceinline__ void init_ring_barriers(uint64_t* full, uint64_t* empty, int S,
                                                   int consumer_warps) {
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], consumer_warps);
    }
    uint64_t* ck = full + 2 * kMaxStages;
    for (int s = 0; s < 2; ++s) {
      mbar_init(&ck[s], 1);
      mbar_init(&ck[2 + s], consumer_warps);
    }
    fence_barrier_init();
  }
  __syncthreads();
}

// Release a stage: called only after the values read from it were consumed
// (the step's outputs are computed and stored), so every lane's shared-memory
// read has completed before the producer may overwrite the stage.
__device__ __forceinline__ void release_stage(uint64_t* empty, int s, int lid) {
  __syncwarp();
  if (lid == 0) mbar_arrive(&empty[s]);
}

// Lanes per thread of the staged kernels: 8 for the Leaky neuron, 4 for the
// Synaptic one (whose reverse pass carries five adjoints per lane).
template <bool SYN>
constexpr int kLanes = SYN ? 4 : 8;
// The staged backward takes its lanes per thread as VL: kLanes, or 4 for
// the Leaky neuron's store mode on short sequences (half the registers of
// 8, so twice the warps fit an SM: faster at T = 25, slower at T = 500).

template <typename T, int NP>
__device__ __forceinline__ void load_pairs(const T* p, float2 q[NP]) {
  float v[2 * NP];
  loadv<T, 2 * NP>(p, v);
#pragma unroll
  for (int k = 0; k < NP; ++k) q[k] = make_float2(v[2 * k], v[2 * k + 1]);
}

template <typename T, int NP>
__device__ __forceinline__ void store_pairs(T* p, const float2 q[NP]) {
  float v[2 * NP];
#pragma unroll
  for (int k = 0; k < NP; ++k) {
    v[2 * k] = q[k].x;
    v[2 * k + 1] = q[k].y;
  }
  storev<T, 2 * NP>(p, v);
}

template <int NP>
__device__ __forceinline__ void load_pairs_global(const float* p, float2 q[NP]) {
#pragma unroll
  for (int k = 0; k < NP; ++k) q[k] = make_float2(p[2 * k], p[2 * k + 1]);
}

// beta, -thr and alpha of the thread's 2*NP lanes, as pairs
template <bool SYN, int NP>  // SYN: also load the third parameter (alpha, or v)
__device__ __forceinline__ void load_params(const ScanArgs& a, int64_t l, float2 beta[NP],
                                            float2 negthr[NP], float2 alpha[NP]) {
#pragma unroll
  for (int k = 0; k < NP; ++k) {
    const int64_t m = l + 2 * k;
    beta[k] = make_float2(lane_param(a.beta, a.beta_mode, m, a),
                          lane_param(a.beta, a.beta_mode, m + 1, a));
    negthr[k] = make_float2(-lane_param(a.thr, a.thr_mode, m, a),
                            -lane_param(a.thr, a.thr_mode, m + 1, a));
    alpha[k] = SYN ? make_float2(lane_param(a.alpha, a.alpha_mode, m, a),
                                 lane_param(a.alpha, a.alpha_mode, m + 1, a))
                   : f2(0.0f);
  }
}

// Initial state of the thread's lanes: u_{-1} = mem0 (or 0), z_{-1} =
// [mem0 > thr] when mem0 is given (else 0), i_{-1} = syn0 (or 0).
template <bool SYN, int NP>
__device__ __forceinline__ void initial_state(const ScanArgs& a, int64_t l, const float2 negthr[NP],
                                              float2 u[NP], bool z[2 * NP], float2 i[NP]) {
#pragma unroll
  for (int k = 0; k < NP; ++k) {
    if (a.mem0) {
      u[k] = make_float2(a.mem0[l + 2 * k], a.mem0[l + 2 * k + 1]);
      z[2 * k] = u[k].x > -negthr[k].x;
      z[2 * k + 1] = u[k].y > -negthr[k].y;
    } else {
      u[k] = f2(0.0f);
      z[2 * k] = z[2 * k + 1] = false;
    }
    i[k] = (SYN && a.syn0) ? make_float2(a.syn0[l + 2 * k], a.syn0[l + 2 * k + 1]) : f2(0.0f);
  }
}

// ---------------------------------------------------------------------------
// Staged forward
// ---------------------------------------------------------------------------

// Rows (time steps) per ring stage of the staged forward: one wait and one
// release per kFwdRows steps instead of per step.
constexpr int kFwdRows = 8;

template <bool SYN, typename TI, typename TO, int RESET, bool REC = false>
__global__ void __launch_bounds__(kMaxStagedThreads) scan_fwd_staged(const ScanArgs a) {
  constexpr int V = kLanes<SYN>, NP = V / 2, R = kFwdRows;
  extern __shared__ __align__(1024) unsigned char smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem);
  uint64_t* empty = full + kMaxStages;
  unsigned char* ring = smem + kBarrierBytes;
  const int S = a.stages;
  const int cwarps = (int)(blockDim.x >> 5) - 1;
  const int warp = threadIdx.x >> 5, lid = threadIdx.x & 31;
  const int64_t lane0 = (int64_t)blockIdx.x * a.lanes_per_cta;
  const int cta_lanes = (int)min((int64_t)a.lanes_per_cta, a.L - lane0);
  const int row_elems = a.lanes_per_cta;  // a stage holds R rows of the strip
  init_ring_barriers(full, empty, S, cwarps);
  grid_dep_wait();  // the previous kernel on the stream is complete

  if (warp == cwarps) {  // producer warp
    if (lid == 0 && !(a.debug & DEBUG_PRODUCER_IDLE)) {
      Producer p{ring, full, empty, S, a.stage_bytes};
      const uint32_t bytes = (uint32_t)cta_lanes * (uint32_t)sizeof(TI);
      const uint32_t row_bytes = (uint32_t)row_elems * (uint32_t)sizeof(TI);
      const TI* src = static_cast<const TI*>(a.I) + lane0;
      for (int64_t t0 = 0; t0 < a.T; t0 += R) {
        const int nr = (int)min((int64_t)R, a.T - t0);
        if (!p.begin((uint32_t)nr * bytes, a)) break;
        for (int r = 0; r < nr; ++r) p.copy((uint32_t)r * row_bytes, src + (t0 + r) * a.L, bytes);
        p.end();
      }
      p.drain();
    }
    return;
  }

  const int c = threadIdx.x;
  const int64_t l = lane0 + (int64_t)c * V;
  const bool active = c * V < cta_lanes;
  float2 beta[NP], negthr[NP], third[NP], u[NP], z[NP], in[NP];
  if (active) {
    load_params<SYN || REC, NP>(a, l, beta, negthr, third);
    bool zb[V];
    initial_state<SYN, NP>(a, l, negthr, u, zb, in);
#pragma unroll
    for (int k = 0; k < NP; ++k) {
      z[k] = make_float2(zb[2 * k] ? 1.0f : 0.0f, zb[2 * k + 1] ? 1.0f : 0.0f);
      if (REC) third[k] = add2_rn(third[k], negthr[k]);  // v - thr, rounded once
    }
  }
  TO* spk = static_cast<TO*>(a.spk) + l;
  TO* mem = a.mem ? static_cast<TO*>(a.mem) + l : nullptr;
  TO* syn = (SYN && a.syn) ? static_cast<TO*>(a.syn) + l : nullptr;
  float* ck = a.ckpt ? a.ckpt + l : nullptr;
  const int64_t ck_stride = SYN ? 2 * a.L : a.L;
  // spike bits: one byte per thread and step (Leaky, 8 lanes), or one per
  // pair of threads (Synaptic, 4 lanes each: the even thread stores)
  unsigned char* bits = a.bits ? a.bits + lane0 / 8 + (SYN ? c / 2 : c) : nullptr;
  const TI* my = reinterpret_cast<const TI*>(ring) + c * V;
  const int stage_elems = a.stage_bytes / (int)sizeof(TI);
  RingPos pos;
  int kk = a.nseg > 0 ? seg_phase0(a) : 0;  // position inside the current checkpoint segment
  for (int64_t t0 = 0; t0 < a.T; t0 += R) {
    if (!warp_wait(&full[pos.s], pos.ph, a.wait_ns)) {
      if (lid == 0) record_status(a.status, kStatusTimeout);
      break;
    }
    const int nr = (int)min((int64_t)R, a.T - t0);
    unsigned zbits[R];
    if (active) {
      const TI* st = my + pos.s * stage_elems;
#pragma unroll
      for (int r = 0; r < R; ++r) {
        zbits[r] = 0;
        if (r < nr) {
          float2 x[NP];
          load_pairs<TI, NP>(st + r * row_elems, x);
#pragma unroll
          for (int k = 0; k < NP; ++k)
            fwd_pair<SYN, RESET, REC ? 1 : 0>(a.reset, beta[k], negthr[k], third[k], x[k], u[k],
                                              z[k], in[k]);
          if (bits) {
#pragma unroll
            for (int k = 0; k < NP; ++k) {
              zbits[r] |= ((z[k].x != 0.0f) ? 1u : 0u) << (2 * k);
              zbits[r] |= ((z[k].y != 0.0f) ? 1u : 0u) << (2 * k + 1);
            }
          }
          store_pairs<TO, NP>(spk + r * a.L, z);
          if (mem) store_pairs<TO, NP>(mem + r * a.L, u);
          if (SYN && syn) store_pairs<TO, NP>(syn + r * a.L, in);
          if (++kk == a.K) {
            kk = 0;
            if (ck && t0 + r + 1 < a.T) {
              store_pairs<float, NP>(ck, u);
              if (SYN) store_pairs<float, NP>(ck + a.L, in);
              ck += ck_stride;
            }
          }
        }
      }
    }
    if (bits) {
#pragma unroll
      for (int r = 0; r < R; ++r) {
        if (r < nr) {
          if (SYN) {
            const unsigned hi = __shfl_down_sync(0xffffffffu, zbits[r], 1);
            if (active && !(c & 1)) bits[r * a.bits_row] = (unsigned char)(zbits[r] | (hi << 4));
          } else if (active) {
            bits[r * a.bits_row] = (unsigned char)zbits[r];
          }
        }
      }
      bits += R * a.bits_row;
    }
    release_stage(empty, pos.s, lid);
    pos.next(S);
    spk += R * a.L;
    if (mem) mem += R * a.L;
    if (SYN && syn) syn += R * a.L;
  }
  if (active) {
    if (a.mem_final) store_pairs<float, NP>(a.mem_final + l, u);
    if (SYN && a.syn_final) store_pairs<float, NP>(a.syn_final + l, in);
  }
}

// ---------------------------------------------------------------------------
// Staged backward.  Store mode (RECOMP=false): one item per step t = T-1..0
// holding the rows {grad_spk, mem, [spk], [syn], [grad_mem]}.  Recompute
// mode: checkpoint segments from last to first; per segment, items for
// t = t0..t1-1 holding {I, [ckpt u, ckpt i at t0]} replay the forward into a
// per-thread shared-memory buffer, then items t = t1-1..t0 holding
// {grad_spk, [grad_mem]} run the reverse steps.
// ---------------------------------------------------------------------------

// The reverse step on all of a thread's pairs; EXTRA steps (grad_mem given,
// or t = T-1 with grad_mem_final / grad_syn_final) add those gradients.
template <bool SYN, int RESET, int SG, bool EXTRA, int NP, bool REC = false>
__device__ __forceinline__ void bwd_pairs(const ScanArgs& a, const float2 beta[NP],
                                          const float2 negthr[NP], const float2 alpha[NP],
                                          const float2 u[NP], const bool z[2 * NP],
                                          const float2 i[NP], const float2 g[NP],
                                          const float2 eu[NP], const float2 ei[NP], Bwd2 st[NP],
                                          float2 out[NP]) {
#pragma unroll
  for (int k = 0; k < NP; ++k)
    out[k] = bwd_pair<SYN, RESET, SG, EXTRA, REC>(a, beta[k], negthr[k], alpha[k], u[k],
                                                  z[2 * k], z[2 * k + 1], i[k], g[k], eu[k],
                                                  ei[k], st[k]);
}

template <bool SYN, bool RECOMP, typename TI, typename TO, int RESET, int SG, int KC = 0,
          bool REC = false, int VL = kLanes<SYN>>
__global__ void __launch_bounds__(kMaxStagedThreads) scan_bwd_staged(const ScanArgs a) {
  static_assert(VL == kLanes<SYN> || (VL == 4 && !SYN && !RECOMP), "lanes per thread");
  constexpr int V = VL, NP = V / 2;
  extern __shared__ __align__(1024) unsigned char smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem);
  uint64_t* empty = full + kMaxStages;
  unsigned char* ring = smem + kBarrierBytes;
  const int S = a.stages;
  const int cwarps = (int)(blockDim.x >> 5) - 1;
  const int nthr = cwarps * 32;
  const int warp = threadIdx.x >> 5, lid = threadIdx.x & 31;
  const int64_t lane0 = (int64_t)blockIdx.x * a.lanes_per_cta;
  const int cta_lanes = (int)min((int64_t)a.lanes_per_cta, a.L - lane0);
  const int io_stride = a.lanes_per_cta * (int)sizeof(TO);  // byte stride of io tiles
  const bool half_store = !RECOMP && sizeof(TO) != 4;      // z from the spk rows
  const bool use_bits = half_store && a.bits != nullptr;    // ... or from the bit rows
  // the bit row of the strip starts at byte lane0/8, copied from the 16-byte
  // boundary below it: the consumer skips bits_skew bytes
  const int bits_skew = (int)((lane0 / 8) & 15);
  const bool want_syn = SYN && a.part_alpha != nullptr;
  // store-mode tile order: gs, mem, [spk], [syn], [gm]
  const int t_spk = 2, t_syn = 2 + (half_store ? 1 : 0);
  const int t_gm_store = t_syn + ((!RECOMP && want_syn) ? 1 : 0);
  // recompute: two checkpoint slots after the replay buffer, prefetched one
  // segment ahead (each holds the strip's u row, then its i row)
  uint64_t* ck_full = full + 2 * kMaxStages;
  uint64_t* ck_empty = ck_full + 2;
  const int ck_slot_bytes = a.lanes_per_cta * 4 * (SYN ? 2 : 1);
  unsigned char* ck_base = ring + (size_t)S * a.stage_bytes +
                           (RECOMP ? (size_t)nthr * V * 4 * a.K * (SYN ? 2 : 1) : 0);
  init_ring_barriers(full, empty, S, cwarps);
  grid_dep_wait();  // the previous kernel on the stream is complete

  if (warp == cwarps) {
    if (lid == 0 && !(a.debug & DEBUG_PRODUCER_IDLE)) {
      Producer p{ring, full, empty, S, a.stage_bytes};
      const uint32_t bo = (uint32_t)cta_lanes * sizeof(TO);
      const uint32_t bi = (uint32_t)cta_lanes * sizeof(TI);
      const uint32_t bc = (uint32_t)cta_lanes * 4u;
      if (!RECOMP) {
        const uint32_t nb = (uint32_t)(bits_skew + cta_lanes / 8 + 15) & ~15u;  // bit row
        const int n_io = 2 + ((half_store && !use_bits) ? 1 : 0) + (want_syn ? 1 : 0) + (a.gm ? 1 : 0);
        const uint32_t total = (uint32_t)n_io * bo + (use_bits ? nb : 0u);
        for (int64_t t = a.T - 1; t >= 0; --t) {
          if (!p.begin(total, a)) break;
          uint32_t n = 0;
          p.copy(n++ * io_stride, row<TO>(a.gs, t, a.L, lane0), bo);
          p.copy(n++ * io_stride, row<TO>(a.mem_in, t, a.L, lane0), bo);
          if (use_bits)
            p.copy(n++ * io_stride, a.bits + t * a.bits_row + lane0 / 8 - bits_skew, nb);
          else if (half_store)
            p.copy(n++ * io_stride, row<TO>(a.spk_in, t, a.L, lane0), bo);
          if (want_syn) p.copy(n++ * io_stride, row<TO>(a.syn_in, t, a.L, lane0), bo);
          if (a.gm) p.copy(n++ * io_stride, row<TO>(a.gm, t, a.L, lane0), bo);
          p.end();
        }
      } else {
        int64_t ck_n = 0;  // checkpoint loads issued
        for (int k = a.nseg - 1; k >= 0 && p.ok; --k) {
          int64_t t0, t1;
          seg_bounds(a, k, t0, t1);
          if (k > 0) {
            // the segment's starting state: checkpoint rows fp32 [nseg-1][SYN?2:1][L]
            const int slot = (int)(ck_n & 1);
            if (ck_n >= 2 &&
                !mbar_wait_spin(&ck_empty[slot], (uint32_t)(((ck_n >> 1) - 1) & 1), a.wait_ns)) {
              record_status(a.status, kStatusTimeout);
              p.ok = false;
              break;
            }
            const float* cu = a.ckpt + (int64_t)(k - 1) * (SYN ? 2 : 1) * a.L + lane0;
            unsigned char* dst = ck_base + (size_t)slot * ck_slot_bytes;
            mbar_arrive_expect_tx(&ck_full[slot], bc * (SYN ? 2u : 1u));
            bulk_g2s(dst, cu, bc, &ck_full[slot]);
            if (SYN) bulk_g2s(dst + a.lanes_per_cta * 4, cu + a.L, bc, &ck_full[slot]);
            ++ck_n;
          }
          for (int64_t t = t0; t < t1 && p.ok; ++t) {
            if (!p.begin(bi, a)) break;
            p.copy(0, row<TI>(a.I, t, a.L, lane0), bi);
            p.end();
          }
          for (int64_t t = t1 - 1; t >= t0 && p.ok; --t) {
            if (!p.begin(bo * (a.gm ? 2u : 1u), a)) break;
            p.copy(0, row<TO>(a.gs, t, a.L, lane0), bo);
            if (a.gm) p.copy((uint32_t)io_stride, row<TO>(a.gm, t, a.L, lane0), bo);
            p.end();
          }
        }
        for (int64_t j = ck_n > 2 ? ck_n - 2 : 0; j < ck_n; ++j)
          mbar_wait_bounded(&ck_full[j & 1], (uint32_t)((j >> 1) & 1), kDrainNs);
      }
      p.drain();
    }
    return;
  }

  const int c = threadIdx.x;
  const int64_t l = lane0 + (int64_t)c * V;
  const bool active = c * V < cta_lanes;
  float2 beta[NP], negthr[NP], alpha[NP];
  Bwd2 st[NP];
  if (active) load_params<SYN || REC, NP>(a, l, beta, negthr, alpha);
#pragma unroll
  for (int k = 0; k < NP; ++k) st[k] = Bwd2{f2(0.0f), f2(0.0f), f2(0.0f), f2(0.0f), f2(0.0f)};
  const int stage_io_elems = a.stage_bytes / (int)sizeof(TO);
  const int stage_in_elems = a.stage_bytes / (int)sizeof(TI);
  const int tile_io_elems = a.lanes_per_cta;  // elements per io tile
  const TO* ring_o = reinterpret_cast<const TO*>(ring) + c * V;
  const TI* ring_i = reinterpret_cast<const TI*>(ring) + c * V;
  TO* gI = static_cast<TO*>(a.gI) + l + (a.T - 1) * a.L;  // walks backwards
  // per-thread replay buffer: [K][V/4 planes][nthr][4] fp32 for u, then i
  // (each plane holds 4 lanes of every thread: conflict-free 16-byte rows)
  float* seg = reinterpret_cast<float*>(ring + (size_t)S * a.stage_bytes) + c * 4;
  const int seg_row = (V / 4) * nthr * 4;  // floats per replayed step
  const size_t seg_plane = (size_t)a.K * seg_row;
  RingPos pos;
  bool ok = true;

  // one reverse step on the thread's pairs: general (EXTRA) only where needed
  auto reverse = [&](int64_t t, const float2 u[NP], const bool z[V], const float2 i[NP],
                     const float2 g[NP], const float2 gmv[NP], float2 out[NP]) {
    if (a.gm || t == a.T - 1) {
      float2 eu[NP], ei[NP];
#pragma unroll
      for (int k = 0; k < NP; ++k) {
        eu[k] = a.gm ? gmv[k] : f2(0.0f);
        ei[k] = f2(0.0f);
      }
      if (t == a.T - 1) {
        float2 fu[NP], fi[NP];
        if (a.gmf) load_pairs_global<NP>(a.gmf + l, fu);
        if (SYN && a.gsf) load_pairs_global<NP>(a.gsf + l, fi);
#pragma unroll
        for (int k = 0; k < NP; ++k) {
          if (a.gmf) eu[k] = add2(eu[k], fu[k]);
          if (SYN && a.gsf) ei[k] = fi[k];
        }
      }
      bwd_pairs<SYN, RESET, SG, true, NP, REC>(a, beta, negthr, alpha, u, z, i, g, eu, ei, st,
                                               out);
    } else {
      bwd_pairs<SYN, RESET, SG, false, NP, REC>(a, beta, negthr, alpha, u, z, i, g, g, g, st,
                                                out);
    }
  };

  if (!RECOMP) {
    for (int64_t t = a.T - 1; t >= 0; --t) {
      if (!warp_wait(&full[pos.s], pos.ph, a.wait_ns)) {
        if (lid == 0) record_status(a.status, kStatusTimeout);
        ok = false;
        break;
      }
      if (active) {
        const TO* base = ring_o + pos.s * stage_io_elems;
        float2 g[NP], uu[NP], ii[NP], gmv[NP], out[NP];
        bool zz[V];
        load_pairs<TO, NP>(base, g);
        load_pairs<TO, NP>(base + tile_io_elems, uu);
        if (use_bits) {
          const unsigned char* bb = reinterpret_cast<const unsigned char*>(base - c * V) +
                                    t_spk * io_stride + bits_skew + (V == 4 ? c / 2 : c);
          const unsigned zb = V == 4 ? (unsigned)(*bb >> ((c & 1) * 4)) : (unsigned)*bb;
#pragma unroll
          for (int k = 0; k < V; ++k) zz[k] = (zb >> k) & 1u;
        } else if (half_store) {
          float2 sp[NP];
          load_pairs<TO, NP>(base + t_spk * tile_io_elems, sp);
#pragma unroll
          for (int k = 0; k < NP; ++k) {
            zz[2 * k] = sp[k].x != 0.0f;
            zz[2 * k + 1] = sp[k].y != 0.0f;
          }
        } else {
#pragma unroll
          for (int k = 0; k < NP; ++k) {
            zz[2 * k] = uu[k].x > -negthr[k].x;
            zz[2 * k + 1] = uu[k].y > -negthr[k].y;
          }
        }
        if (want_syn) {
          load_pairs<TO, NP>(base + t_syn * tile_io_elems, ii);
        } else {
#pragma unroll
          for (int k = 0; k < NP; ++k) ii[k] = f2(0.0f);
        }
        if (a.gm) load_pairs<TO, NP>(base + t_gm_store * tile_io_elems, gmv);
        reverse(t, uu, zz, ii, g, gmv, out);
        store_pairs<TO, NP>(gI, out);
      }
      release_stage(empty, pos.s, lid);
      pos.next(S);
      gI -= a.L;
    }
  } else {
    int64_t ck_u = 0;  // checkpoints consumed
    float2 u[NP], ii[NP], z[NP], third[NP];
#pragma unroll
    for (int q = 0; q < NP; ++q)  // alpha (Synaptic), or v - thr rounded once (Eq. 7)
      third[q] = REC ? add2_rn(alpha[q], negthr[q]) : alpha[q];
    // Start of segment k: its starting state from the checkpoint slot (k > 0)
    // or the initial state (k = 0).
    auto seg_start = [&](int k) -> bool {
      if (k > 0) {
        if (!warp_wait(&ck_full[ck_u & 1], (uint32_t)((ck_u >> 1) & 1), a.wait_ns)) {
          if (lid == 0) record_status(a.status, kStatusTimeout);
          return false;
        }
        if (active) {
          const float* cb =
              reinterpret_cast<const float*>(ck_base + (size_t)(ck_u & 1) * ck_slot_bytes) + c * V;
          load_pairs<float, NP>(cb, u);
          if (SYN) load_pairs<float, NP>(cb + a.lanes_per_cta, ii);
#pragma unroll
          for (int q = 0; q < NP; ++q) z[q] = fire2(u[q], negthr[q]);
        }
      } else if (active) {
        bool zb[V];
        initial_state<SYN, NP>(a, l, negthr, u, zb, ii);
#pragma unroll
        for (int q = 0; q < NP; ++q)
          z[q] = make_float2(zb[2 * q] ? 1.0f : 0.0f, zb[2 * q + 1] ? 1.0f : 0.0f);
      }
      return true;
    };
    // After the replay consumed the checkpoint values: free the slot.
    auto seg_replayed = [&](int k) {
      if (k > 0) {
        release_stage(ck_empty, (int)(ck_u & 1), lid);
        ++ck_u;
      }
    };
    // One replayed forward step from an I row in the stage at `xin`; the
    // state goes to the replay buffer row `su`.
    auto replay = [&](const TI* xin, float* su) {
      if (!active) return;
      float2 x[NP];
      load_pairs<TI, NP>(xin, x);
#pragma unroll
      for (int q = 0; q < NP; ++q)
        fwd_pair<SYN, RESET, REC ? 1 : 0>(a.reset, beta[q], negthr[q], third[q], x[q], u[q],
                                          z[q], ii[q]);
#pragma unroll
      for (int q = 0; q < V / 4; ++q) {
        *reinterpret_cast<float4*>(su + q * nthr * 4) =
            make_float4(u[2 * q].x, u[2 * q].y, u[2 * q + 1].x, u[2 * q + 1].y);
        if (SYN)
          *reinterpret_cast<float4*>(su + seg_plane + q * nthr * 4) =
              make_float4(ii[2 * q].x, ii[2 * q].y, ii[2 * q + 1].x, ii[2 * q + 1].y);
      }
    };
    // One reverse step at time t: grad rows in the stage at `gin`, the
    // replayed state from buffer row `su`, dL/dI_t to `gout`.
    auto reverse_step = [&](int64_t t, const TO* gin, const float* su, TO* gout) {
      if (!active) return;
      float2 g[NP], gmv[NP], uu[NP], iv[NP], out[NP];
      bool zz[V];
      load_pairs<TO, NP>(gin, g);
      if (a.gm) load_pairs<TO, NP>(gin + tile_io_elems, gmv);
#pragma unroll
      for (int q = 0; q < V / 4; ++q) {
        const float4 uq = *reinterpret_cast<const float4*>(su + q * nthr * 4);
        uu[2 * q] = make_float2(uq.x, uq.y);
        uu[2 * q + 1] = make_float2(uq.z, uq.w);
        if (SYN) {
          const float4 iq = *reinterpret_cast<const float4*>(su + seg_plane + q * nthr * 4);
          iv[2 * q] = make_float2(iq.x, iq.y);
          iv[2 * q + 1] = make_float2(iq.z, iq.w);
        } else {
          iv[2 * q] = f2(0.0f);
          iv[2 * q + 1] = f2(0.0f);
        }
      }
#pragma unroll
      for (int q = 0; q < NP; ++q) {
        zz[2 * q] = uu[q].x > -negthr[q].x;
        zz[2 * q + 1] = uu[q].y > -negthr[q].y;
      }
      reverse(t, uu, zz, iv, g, gmv, out);
      store_pairs<TO, NP>(gout, out);
    };
    auto fail = [&]() {
      if (lid == 0) record_status(a.status, kStatusTimeout);
      ok = false;
    };

    int k = a.nseg - 1;
    if constexpr (KC > 0) {
      // Full segments (all but the first in time) with the ring at exactly
      // KS = KC stages: a segment is two whole ring rounds (KC replay items,
      // then KC reverse items), so every stage index and phase parity below
      // is a compile-time constant and the ring position is unchanged after
      // each segment.
      for (; k >= 1 && ok; --k) {
        int64_t t0, t1;
        seg_bounds(a, k, t0, t1);
        if (!seg_start(k)) {
          ok = false;
          break;
        }
#pragma unroll
        for (int q = 0; q < KC; ++q) {
          if (!warp_wait(&full[q], 0u, a.wait_ns)) {
            fail();
            break;
          }
          replay(ring_i + q * stage_in_elems, seg + q * seg_row);
          release_stage(empty, q, lid);
        }
        if (!ok) break;
        seg_replayed(k);
        TO* gout = static_cast<TO*>(a.gI) + l + t0 * a.L;
#pragma unroll
        for (int q = KC - 1; q >= 0; --q) {
          const int st_idx = KC - 1 - q;  // stage of this reverse item
          if (!warp_wait(&full[st_idx], 1u, a.wait_ns)) {
            fail();
            break;
          }
          reverse_step(t0 + q, ring_o + st_idx * stage_io_elems, seg + q * seg_row,
                       gout + q * a.L);
          release_stage(empty, st_idx, lid);
        }
      }
    }
    // Remaining segments (all of them for run-time K) with the general ring
    // position.
    for (; k >= 0 && ok; --k) {
      int64_t t0, t1;
      seg_bounds(a, k, t0, t1);
      if (!seg_start(k)) {
        ok = false;
        break;
      }
      float* su = seg;
      for (int64_t t = t0; t < t1; ++t) {
        if (!warp_wait(&full[pos.s], pos.ph, a.wait_ns)) {
          fail();
          break;
        }
        replay(ring_i + pos.s * stage_in_elems, su);
        release_stage(empty, pos.s, lid);
        pos.next(S);
        su += seg_row;
      }
      if (!ok) break;
      seg_replayed(k);
      TO* gout = static_cast<TO*>(a.gI) + l + t0 * a.L;
      for (int64_t t = t1 - 1; t >= t0; --t) {
        su -= seg_row;
        if (!warp_wait(&full[pos.s], pos.ph, a.wait_ns)) {
          fail();
          break;
        }
        reverse_step(t, ring_o + pos.s * stage_io_elems, su, gout + (t - t0) * a.L);
        release_stage(empty, pos.s, lid);
        pos.next(S);
      }
    }
  }
  if (!ok || !active) return;
  float gm0[V], gs0[V], db[V], dt[V], da[V];
#pragma unroll
  for (int v = 0; v < V; ++v) {
    const Bwd2& q = st[v / 2];
    const bool hi = v & 1;
    BwdLane sl{hi ? q.du.y : q.du.x, hi ? q.di.y : q.di.x, hi ? q.dbeta.y : q.dbeta.x,
               -(hi ? q.dthr.y : q.dthr.x), hi ? q.dalpha.y : q.dalpha.x};
    const float b = hi ? beta[v / 2].y : beta[v / 2].x;
    const float th = -(hi ? negthr[v / 2].y : negthr[v / 2].x);
    const float al = hi ? alpha[v / 2].y : alpha[v / 2].x;
    if (a.T == 0) {
      gm0[v] = a.gmf ? a.gmf[l + v] : 0.0f;
      gs0[v] = (SYN && a.gsf) ? a.gsf[l + v] : 0.0f;
    } else {
      const float m0 = a.mem0 ? a.mem0[l + v] : 0.0f;
      const float s0 = (SYN && a.syn0) ? a.syn0[l + v] : 0.0f;
      bwd_initial<SYN>(a, b, th, al, a.mem0 != nullptr, m0, s0, sl, gm0[v], gs0[v]);
    }
    db[v] = sl.dbeta;
    dt[v] = sl.dthr;
    da[v] = sl.dalpha;
  }
  if (a.gmem0) storev<float, V>(a.gmem0 + l, gm0);
  if (SYN && a.gsyn0) storev<float, V>(a.gsyn0 + l, gs0);
  if (a.part_beta) storev<float, V>(a.part_beta + l, db);
  if (a.part_thr) storev<float, V>(a.part_thr + l, dt);
  if ((SYN || REC) && a.part_alpha) storev<float, V>(a.part_alpha + l, da);
}

// ---------------------------------------------------------------------------
// Plain kernels: one lane per thread, direct loads, any shape, run-time modes.
// ---------------------------------------------------------------------------

template <bool SYN, typename TI, typename TO>
__global__ void __launch_bounds__(256) scan_fwd_plain(const ScanArgs a) {
  grid_dep_wait();
  const int64_t l = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (l >= a.L) return;
  const float beta = lane_param(a.beta, a.beta_mode, l, a);
  const float thr = lane_param(a.thr, a.thr_mode, l, a);
  const float alpha = (SYN || a.rec) ? lane_param(a.alpha, a.alpha_mode, l, a) : 0.0f;
  float u = a.mem0 ? a.mem0[l] : 0.0f;
  bool z = a.mem0 ? (u > thr) : false;
  float i = (SYN && a.syn0) ? a.syn0[l] : 0.0f;
  const TI* I = static_cast<const TI*>(a.I);
  TO* spk = static_cast<TO*>(a.spk);
  TO* mem = static_cast<TO*>(a.mem);
  TO* syn = static_cast<TO*>(a.syn);
  const int64_t ckpt_stride = SYN ? 2 * a.L : a.L;
  int kk = a.nseg > 0 ? seg_phase0(a) : 0;
  float* cp = a.ckpt ? a.ckpt + l : nullptr;
  for (int64_t t = 0; t < a.T; ++t) {
    const int64_t off = t * a.L + l;
    fwd_step<SYN, -1, -1>(a.reset, beta, thr, alpha, Elem<TI>::load1(I + off), u, z, i,
                          a.rec != 0);
    Elem<TO>::store1(spk + off, z ? 1.0f : 0.0f);
    if (mem) Elem<TO>::store1(mem + off, u);
    if (SYN && syn) Elem<TO>::store1(syn + off, i);
    if (++kk == a.K) {
      kk = 0;
      if (cp && t + 1 < a.T) {
        *cp = u;
        if (SYN) cp[a.L] = i;
        cp += ckpt_stride;
      }
    }
  }
  if (a.mem_final) a.mem_final[l] = u;
  if (SYN && a.syn_final) a.syn_final[l] = i;
}

template <bool SYN, bool RECOMP, typename TI, typename TO>
__global__ void __launch_bounds__(128) scan_bwd_plain(const ScanArgs a) {
  extern __shared__ __align__(16) float segbuf[];  // [K][blockDim] u, then i
  grid_dep_wait();
  const int64_t l = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (l >= a.L) return;
  const float beta = lane_param(a.beta, a.beta_mode, l, a);
  const float thr = lane_param(a.thr, a.thr_mode, l, a);
  const float alpha = (SYN || a.rec) ? lane_param(a.alpha, a.alpha_mode, l, a) : 0.0f;
  const bool have_mem0 = a.mem0 != nullptr;
  const float m0 = have_mem0 ? a.mem0[l] : 0.0f;
  const float s0 = (SYN && a.syn0) ? a.syn0[l] : 0.0f;
  const float ex_u = a.gmf ? a.gmf[l] : 0.0f;
  const float ex_i = (SYN && a.gsf) ? a.gsf[l] : 0.0f;
  const bool half_store = !RECOMP && sizeof(TO) != 4;
  const bool want_syn = SYN && a.part_alpha != nullptr;
  const TO* gs = static_cast<const TO*>(a.gs);
  const TO* gm = static_cast<const TO*>(a.gm);
  TO* gI = static_cast<TO*>(a.gI);
  BwdLane st{0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
  if (!RECOMP) {
    const TO* mem = static_cast<const TO*>(a.mem_in);
    const TO* spk = static_cast<const TO*>(a.spk_in);
    const TO* syn = static_cast<const TO*>(a.syn_in);
    for (int64_t t = a.T - 1; t >= 0; --t) {
      const int64_t off = t * a.L + l;
      const float u = Elem<TO>::load1(mem + off);
      const bool z = half_store ? (Elem<TO>::load1(spk + off) != 0.0f) : (u > thr);
      const float i = want_syn ? Elem<TO>::load1(syn + off) : 0.0f;
      const bool last = (t == a.T - 1);
      const float eu = (gm ? Elem<TO>::load1(gm + off) : 0.0f) + (last ? ex_u : 0.0f);
      Elem<TO>::store1(gI + off, bwd_step<SYN, -1, -1>(a, beta, thr, alpha, !last, u, z, i,
                                                       Elem<TO>::load1(gs + off), eu,
                                                       last ? ex_i : 0.0f, st));
    }
  } else {
    const TI* I = static_cast<const TI*>(a.I);
    float* su = segbuf + threadIdx.x;
    float* si = segbuf + (size_t)a.K * blockDim.x + threadIdx.x;
    for (int k = a.nseg - 1; k >= 0; --k) {
      int64_t t0, t1;
      seg_bounds(a, k, t0, t1);
      float u, i;
      bool z;
      if (k > 0) {
        const float* cp = a.ckpt + (int64_t)(k - 1) * (SYN ? 2 : 1) * a.L + l;
        u = cp[0];
        i = SYN ? cp[a.L] : 0.0f;
        z = u > thr;
      } else {
        u = m0;
        i = s0;
        z = have_mem0 && (m0 > thr);
      }
      for (int64_t t = t0; t < t1; ++t) {
        fwd_step<SYN, -1, -1>(a.reset, beta, thr, alpha, Elem<TI>::load1(I + t * a.L + l), u,
                              z, i, a.rec != 0);
        su[(t - t0) * blockDim.x] = u;
        if (SYN) si[(t - t0) * blockDim.x] = i;
      }
      for (int64_t t = t1 - 1; t >= t0; --t) {
        const int64_t off = t * a.L + l;
        const float uu = su[(t - t0) * blockDim.x];
        const float iv = SYN ? si[(t - t0) * blockDim.x] : 0.0f;
        const bool last = (t == a.T - 1);
        const float eu = (gm ? Elem<TO>::load1(gm + off) : 0.0f) + (last ? ex_u : 0.0f);
        Elem<TO>::store1(gI + off, bwd_step<SYN, -1, -1>(a, beta, thr, alpha, !last, uu,
                                                         uu > thr, iv, Elem<TO>::load1(gs + off),
                                                         eu, last ? ex_i : 0.0f, st));
      }
    }
  }
  float gm0, gs0;
  if (a.T == 0) {
    gm0 = ex_u;
    gs0 = ex_i;
  } else {
    bwd_initial<SYN>(a, beta, thr, alpha, have_mem0, m0, s0, st, gm0, gs0);
  }
  if (a.gmem0) a.gmem0[l] = gm0;
  if (SYN && a.gsyn0) a.gsyn0[l] = gs0;
  if (a.part_beta) a.part_beta[l] = st.dbeta;
  if (a.part_thr) a.part_thr[l] = st.dthr;
  if ((SYN || a.rec) && a.part_alpha) a.part_alpha[l] = st.dalpha;
}

}  // namespace snn
