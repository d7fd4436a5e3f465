// Fused temporal-scan kernels for the Leaky (Eq. 4) and Synaptic (Eqs. 5-6)
// neurons of arXiv 2211.10725, forward and BPTT (Sec. II-A/B, III-B).
//
// Layout: every [T, B, N] tensor is t-major, so the L = B*N lanes of one step
// are contiguous.  A lane is independent of every other lane and sequential
// in t: each thread owns VEC=4 consecutive lanes and keeps their state (u, i,
// z and, backward, the adjoints) in registers for the whole scan.
//
// Staged kernels (the fast path): a CTA owns a contiguous strip of lanes.
// One producer thread streams the strip's row of every input tensor, step by
// step, into a ring of shared-memory stages with 1-D bulk copies (TMA,
// cp.async.bulk) completing on an mbarrier per stage; the consumer warps wait
// on the stage, read their lanes, release the stage on a second mbarrier and
// write outputs with vector stores.  The ring depth, not the thread count,
// supplies the bytes in flight that HBM needs.
//
// Plain kernels: one lane per thread, direct loads; taken for shapes whose
// rows are not 16-byte multiples.  Both use the same per-lane step code, so
// they give bit-identical forward results.
#pragma once

#include "snn_device.cuh"

namespace snn {

enum { RESET_SUBTRACT = 0, RESET_ZERO = 1, RESET_NONE = 2 };
enum { SG_FAST_SIGMOID = 0, SG_ATAN = 1 };
enum { PM_SCALAR = 0, PM_PER_NEURON = 1, PM_PER_CHANNEL = 2 };
constexpr uint32_t DEBUG_PRODUCER_IDLE = 1u;
constexpr int VEC = 4;                 // lanes per thread in the staged kernels
constexpr int kBarrierBytes = 1024;    // room for up to 64 stages x 2 mbarriers
constexpr int kMaxStages = 64;
constexpr uint64_t kDrainNs = 1000000000ull;

struct ScanArgs {
  int64_t T, L, N, C, HW;
  int K;      // checkpoint interval (recompute); T in store mode
  int nseg;   // ceil(T / K)
  int reset, detach, sg;
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

// One forward step, Eq. (4) / Eqs. (5)-(6), evaluated left to right as the
// equations are written, one rounded fp32 operation at a time (no FMA), so
// the forward and the backward's recomputation agree bit for bit.
template <bool SYN>
__device__ __forceinline__ void fwd_step(int reset, float beta, float thr, float alpha, float x,
                                         float& u, bool& z, float& i) {
  float in = x;
  if (SYN) {
    i = __fadd_rn(__fmul_rn(alpha, i), x);
    in = i;
  }
  float un;
  if (reset == RESET_ZERO) {
    un = __fadd_rn(__fmul_rn(beta, z ? 0.0f : u), in);
  } else {
    un = __fadd_rn(__fmul_rn(beta, u), in);
    if (reset == RESET_SUBTRACT && z) un = __fsub_rn(un, thr);
  }
  u = un;
  z = un > thr;  // Eq. (3), strict
}

// Surrogate dz/du at x = u - thr (Sec. III-B).
__device__ __forceinline__ float surrogate(const ScanArgs& a, float x) {
  if (a.sg == SG_FAST_SIGMOID) {
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
template <bool SYN>
__device__ __forceinline__ float bwd_step(const ScanArgs& a, float beta, float thr, float alpha,
                                          bool has_next, float u, bool z, float i, float gs,
                                          float extra_u, float extra_i, BwdLane& s) {
  if (has_next) {
    s.dbeta = fmaf(s.du, (a.reset == RESET_ZERO && z) ? 0.0f : u, s.dbeta);
    if (a.reset == RESET_SUBTRACT && z) s.dthr -= s.du;
    if (SYN) s.dalpha = fmaf(s.di, i, s.dalpha);
  }
  const float sgv = surrogate(a, u - thr);
  float dz = gs;
  if (!a.detach) {
    if (a.reset == RESET_SUBTRACT) dz = fmaf(-thr, s.du, dz);
    else if (a.reset == RESET_ZERO) dz = fmaf(-beta * u, s.du, dz);
  }
  const float decay = (a.reset == RESET_ZERO && z) ? 0.0f : beta;
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
  s.dbeta = fmaf(s.du, (a.reset == RESET_ZERO && z_m1) ? 0.0f : u_m1, s.dbeta);
  if (a.reset == RESET_SUBTRACT && z_m1) s.dthr -= s.du;
  if (SYN) s.dalpha = fmaf(s.di, i_m1, s.dalpha);
  const float decay = (a.reset == RESET_ZERO && z_m1) ? 0.0f : beta;
  gmem0 = decay * s.du;
  if (have_mem0 && !a.detach && a.reset != RESET_NONE) {
    const float sgv = surrogate(a, u_m1 - thr);
    const float slope = (a.reset == RESET_SUBTRACT) ? -thr : -beta * u_m1;
    const float dz = slope * s.du;
    gmem0 = fmaf(sgv, dz, gmem0);
    s.dthr = fmaf(-sgv, dz, s.dthr);
  }
  gsyn0 = SYN ? alpha * s.di : 0.0f;
}

// Warp-uniform bounded wait: every lane polls the barrier (so every lane
// acquires the completed phase); the decision to give up is taken by lane 0's
// clock and shared, so the warp never diverges around it.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  bool done = mbar_try_wait(bar, parity);
  if (__all_sync(0xffffffffu, done)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    if (!done) done = mbar_try_wait(bar, parity);
    if (__all_sync(0xffffffffu, done)) return true;
    uint64_t el = globaltimer_ns() - t0;
    el = __shfl_sync(0xffffffffu, el, 0);
    if (el > limit_ns) return false;
  }
}

// ---------------------------------------------------------------------------
// Producer: streams item j's tiles into stage j % S.
// ---------------------------------------------------------------------------

struct Tile {
  const void* src;  // global address of the strip's row (16-byte aligned)
  uint32_t bytes;   // multiple of 16
  uint32_t dst;     // byte offset inside the stage (multiple of 16)
};

struct Producer {
  unsigned char* ring;
  uint64_t* full;
  uint64_t* empty;
  int S;
  int stage_bytes;
  int64_t issued = 0;
  bool ok = true;

  // Issue the next item into stage issued % S once the consumers released it.
  __device__ __forceinline__ void issue(const Tile* tiles, int n, const ScanArgs& a) {
    if (!ok) return;
    const int64_t j = issued;
    const int s = (int)(j % S);
    if (j >= S &&
        !mbar_wait_bounded(&empty[s], (uint32_t)(((j / S) - 1) & 1), a.wait_ns)) {
      record_status(a.status, kStatusTimeout);
      ok = false;
      return;
    }
    uint32_t total = 0;
    for (int k = 0; k < n; ++k) total += tiles[k].bytes;
    mbar_arrive_expect_tx(&full[s], total);
    unsigned char* dst = ring + (size_t)s * stage_bytes;
    for (int k = 0; k < n; ++k) bulk_g2s(dst + tiles[k].dst, tiles[k].src, tiles[k].bytes, &full[s]);
    issued = j + 1;
  }

  // Wait until every copy this thread issued has landed (bounded), so the
  // CTA's shared memory outlives all of them.
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

__device__ __forceinline__ void init_ring_barriers(uint64_t* full, uint64_t* empty, int S,
                                                   int consumer_warps) {
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], consumer_warps);
    }
    fence_barrier_init();
  }
  __syncthreads();
}

// ---------------------------------------------------------------------------
// Staged forward
// ---------------------------------------------------------------------------

template <bool SYN, typename TI, typename TO>
__global__ void __launch_bounds__(1024) scan_fwd_staged(const ScanArgs a) {
  extern __shared__ __align__(1024) unsigned char smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem);
  uint64_t* empty = full + kMaxStages;
  unsigned char* ring = smem + kBarrierBytes;
  const int S = a.stages;
  const int cwarps = (int)(blockDim.x >> 5) - 1;
  const int warp = threadIdx.x >> 5, lid = threadIdx.x & 31;
  const int64_t lane0 = (int64_t)blockIdx.x * a.lanes_per_cta;
  const int cta_lanes = (int)min((int64_t)a.lanes_per_cta, a.L - lane0);
  init_ring_barriers(full, empty, S, cwarps);

  if (warp == cwarps) {  // producer warp
    if (lid == 0 && !(a.debug & DEBUG_PRODUCER_IDLE)) {
      Producer p{ring, full, empty, S, a.stage_bytes};
      const uint32_t bytes = (uint32_t)cta_lanes * sizeof(TI);
      for (int64_t t = 0; t < a.T && p.ok; ++t) {
        const Tile tile{row<TI>(a.I, t, a.L, lane0), bytes, 0};
        p.issue(&tile, 1, a);
      }
      p.drain();
    }
    return;
  }

  const int c = threadIdx.x;
  const int64_t l = lane0 + (int64_t)c * VEC;
  const bool active = c * VEC < cta_lanes;
  float beta[VEC], thr[VEC], alpha[VEC], u[VEC], in[VEC];
  bool z[VEC];
  if (active) {
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      beta[v] = lane_param(a.beta, a.beta_mode, l + v, a);
      thr[v] = lane_param(a.thr, a.thr_mode, l + v, a);
      alpha[v] = SYN ? lane_param(a.alpha, a.alpha_mode, l + v, a) : 0.0f;
      u[v] = a.mem0 ? a.mem0[l + v] : 0.0f;
      z[v] = a.mem0 ? (u[v] > thr[v]) : false;
      in[v] = (SYN && a.syn0) ? a.syn0[l + v] : 0.0f;
    }
  }
  TO* spk = static_cast<TO*>(a.spk);
  TO* mem = static_cast<TO*>(a.mem);
  TO* syn = static_cast<TO*>(a.syn);
  const int64_t ckpt_stride = SYN ? 2 * a.L : a.L;
  int kk = 0;  // position inside the current checkpoint segment
  for (int64_t t = 0; t < a.T; ++t) {
    const int s = (int)(t % S);
    if (!warp_wait(&full[s], (uint32_t)((t / S) & 1), a.wait_ns)) {
      if (lid == 0) record_status(a.status, kStatusTimeout);
      break;
    }
    float x[VEC];
    if (active) Elem<TI>::load4(reinterpret_cast<const TI*>(ring + (size_t)s * a.stage_bytes) + c * VEC, x);
    if (active) {
      float zf[VEC];
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        fwd_step<SYN>(a.reset, beta[v], thr[v], alpha[v], x[v], u[v], z[v], in[v]);
        zf[v] = z[v] ? 1.0f : 0.0f;
      }
      const int64_t off = t * a.L + l;
      Elem<TO>::store4(spk + off, zf);
      if (mem) Elem<TO>::store4(mem + off, u);
      if (SYN && syn) Elem<TO>::store4(syn + off, in);
      if (++kk == a.K) {
        kk = 0;
        if (a.ckpt && t + 1 < a.T) {
          float* cp = a.ckpt + (t / a.K) * ckpt_stride + l;
          Elem<float>::store4(cp, u);
          if (SYN) Elem<float>::store4(cp + a.L, in);
        }
      }
    }
    // Release the stage only after its values were consumed: the stores
    // above depend on them, so every lane's shared-memory read has completed
    // before the producer may refill the stage with a bulk copy.
    __syncwarp();
    if (lid == 0) mbar_arrive(&empty[s]);
  }
  if (active) {
    if (a.mem_final) Elem<float>::store4(a.mem_final + l, u);
    if (SYN && a.syn_final) Elem<float>::store4(a.syn_final + l, in);
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

template <bool SYN, bool RECOMP, typename TI, typename TO>
__global__ void __launch_bounds__(1024) scan_bwd_staged(const ScanArgs a) {
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
  const int io_stride = a.lanes_per_cta * (int)sizeof(TO);   // tile stride of io tiles
  const int in_stride = a.lanes_per_cta * (int)sizeof(TI);
  const bool half_store = !RECOMP && sizeof(TO) != 4;       // z from the spk rows
  const bool want_syn = SYN && a.part_alpha != nullptr;
  // store-mode tile order: gs, mem, [spk], [syn], [gm]
  const int t_spk = 2, t_syn = 2 + (half_store ? 1 : 0);
  const int t_gm_store = t_syn + ((!RECOMP && want_syn) ? 1 : 0);
  const int ck_off = (in_stride + 15) & ~15;  // recompute: checkpoint tiles after I
  init_ring_barriers(full, empty, S, cwarps);

  if (warp == cwarps) {
    if (lid == 0 && !(a.debug & DEBUG_PRODUCER_IDLE)) {
      Producer p{ring, full, empty, S, a.stage_bytes};
      const uint32_t bo = (uint32_t)cta_lanes * sizeof(TO);
      const uint32_t bi = (uint32_t)cta_lanes * sizeof(TI);
      const uint32_t bc = (uint32_t)cta_lanes * 4u;
      Tile tiles[5];
      if (!RECOMP) {
        for (int64_t t = a.T - 1; t >= 0 && p.ok; --t) {
          int n = 0;
          tiles[n] = Tile{row<TO>(a.gs, t, a.L, lane0), bo, (uint32_t)(n * io_stride)}; ++n;
          tiles[n] = Tile{row<TO>(a.mem_in, t, a.L, lane0), bo, (uint32_t)(n * io_stride)}; ++n;
          if (half_store) { tiles[n] = Tile{row<TO>(a.spk_in, t, a.L, lane0), bo, (uint32_t)(n * io_stride)}; ++n; }
          if (want_syn) { tiles[n] = Tile{row<TO>(a.syn_in, t, a.L, lane0), bo, (uint32_t)(n * io_stride)}; ++n; }
          if (a.gm) { tiles[n] = Tile{row<TO>(a.gm, t, a.L, lane0), bo, (uint32_t)(n * io_stride)}; ++n; }
          p.issue(tiles, n, a);
        }
      } else {
        for (int k = a.nseg - 1; k >= 0 && p.ok; --k) {
          const int64_t t0 = (int64_t)k * a.K, t1 = min(a.T, t0 + a.K);
          for (int64_t t = t0; t < t1 && p.ok; ++t) {
            int n = 0;
            tiles[n++] = Tile{row<TI>(a.I, t, a.L, lane0), bi, 0};
            if (t == t0 && k > 0) {
              // the segment's starting state rides with its first input row;
              // checkpoint rows are fp32 [nseg-1][SYN ? 2 : 1][L]
              const float* cu = a.ckpt + (int64_t)(k - 1) * (SYN ? 2 : 1) * a.L + lane0;
              tiles[n++] = Tile{cu, bc, (uint32_t)ck_off};
              if (SYN) tiles[n++] = Tile{cu + a.L, bc, (uint32_t)(ck_off + a.lanes_per_cta * 4)};
            }
            p.issue(tiles, n, a);
          }
          for (int64_t t = t1 - 1; t >= t0 && p.ok; --t) {
            int n = 0;
            tiles[n++] = Tile{row<TO>(a.gs, t, a.L, lane0), bo, 0};
            if (a.gm) tiles[n++] = Tile{row<TO>(a.gm, t, a.L, lane0), bo, (uint32_t)io_stride};
            p.issue(tiles, n, a);
          }
        }
      }
      p.drain();
    }
    return;
  }

  const int c = threadIdx.x;
  const int64_t l = lane0 + (int64_t)c * VEC;
  const bool active = c * VEC < cta_lanes;
  float beta[VEC], thr[VEC], alpha[VEC], m0[VEC], s0[VEC], ex_u[VEC], ex_i[VEC];
  BwdLane st[VEC];
  const bool have_mem0 = a.mem0 != nullptr;
  if (active) {
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      beta[v] = lane_param(a.beta, a.beta_mode, l + v, a);
      thr[v] = lane_param(a.thr, a.thr_mode, l + v, a);
      alpha[v] = SYN ? lane_param(a.alpha, a.alpha_mode, l + v, a) : 0.0f;
      m0[v] = have_mem0 ? a.mem0[l + v] : 0.0f;
      s0[v] = (SYN && a.syn0) ? a.syn0[l + v] : 0.0f;
      ex_u[v] = a.gmf ? a.gmf[l + v] : 0.0f;
      ex_i[v] = (SYN && a.gsf) ? a.gsf[l + v] : 0.0f;
      st[v] = BwdLane{0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
    }
  }
  TO* gI = static_cast<TO*>(a.gI);
  // per-thread replay buffer for one checkpoint segment: [K][nthr][VEC] fp32
  // (u), followed by the same for i (Synaptic)
  float* seg = reinterpret_cast<float*>(ring + (size_t)S * a.stage_bytes);
  const size_t seg_plane = (size_t)a.K * nthr * VEC;
  bool ok = true;
  int64_t j = 0;  // item counter, mirrors the producer's

  auto wait_item = [&](int64_t jj, const unsigned char*& base) -> bool {
    const int s = (int)(jj % S);
    if (!warp_wait(&full[s], (uint32_t)((jj / S) & 1), a.wait_ns)) {
      if (lid == 0) record_status(a.status, kStatusTimeout);
      return false;
    }
    base = ring + (size_t)s * a.stage_bytes;
    return true;
  };
  // Called only once the values read from item jj's stage have been consumed
  // (outputs computed and stored), so the reads have completed before the
  // producer may overwrite the stage.
  auto release_item = [&](int64_t jj) {
    __syncwarp();
    if (lid == 0) mbar_arrive(&empty[(int)(jj % S)]);
  };

  if (!RECOMP) {
    for (int64_t t = a.T - 1; t >= 0; --t, ++j) {
      const unsigned char* base;
      if (!wait_item(j, base)) { ok = false; break; }
      float g[VEC], uu[VEC], zz[VEC], ii[VEC], gmv[VEC];
      if (active) {
        Elem<TO>::load4(reinterpret_cast<const TO*>(base) + c * VEC, g);
        Elem<TO>::load4(reinterpret_cast<const TO*>(base + io_stride) + c * VEC, uu);
        if (half_store) Elem<TO>::load4(reinterpret_cast<const TO*>(base + t_spk * io_stride) + c * VEC, zz);
        if (want_syn) Elem<TO>::load4(reinterpret_cast<const TO*>(base + t_syn * io_stride) + c * VEC, ii);
        if (a.gm) Elem<TO>::load4(reinterpret_cast<const TO*>(base + t_gm_store * io_stride) + c * VEC, gmv);
      }
      if (active) {
        float out[VEC];
        const bool last = (t == a.T - 1);
#pragma unroll
        for (int v = 0; v < VEC; ++v) {
          const bool zv = half_store ? (zz[v] != 0.0f) : (uu[v] > thr[v]);
          const float eu = (a.gm ? gmv[v] : 0.0f) + (last ? ex_u[v] : 0.0f);
          out[v] = bwd_step<SYN>(a, beta[v], thr[v], alpha[v], !last, uu[v], zv,
                                 want_syn ? ii[v] : 0.0f, g[v], eu, last ? ex_i[v] : 0.0f, st[v]);
        }
        Elem<TO>::store4(gI + t * a.L + l, out);
      }
      release_item(j);  // after the values read from the stage were consumed
    }
  } else {
    for (int k = a.nseg - 1; k >= 0 && ok; --k) {
      const int64_t t0 = (int64_t)k * a.K, t1 = min(a.T, t0 + a.K);
      float u[VEC], ii[VEC];
      bool z[VEC];
      // replay the forward over the segment
      for (int64_t t = t0; t < t1; ++t, ++j) {
        const unsigned char* base;
        if (!wait_item(j, base)) { ok = false; break; }
        float x[VEC];
        if (active) {
          Elem<TI>::load4(reinterpret_cast<const TI*>(base) + c * VEC, x);
          if (t == t0) {
            if (k > 0) {
              Elem<float>::load4(reinterpret_cast<const float*>(base + ck_off) + c * VEC, u);
              if (SYN)
                Elem<float>::load4(reinterpret_cast<const float*>(base + ck_off + a.lanes_per_cta * 4) + c * VEC, ii);
#pragma unroll
              for (int v = 0; v < VEC; ++v) z[v] = u[v] > thr[v];
            } else {
#pragma unroll
              for (int v = 0; v < VEC; ++v) {
                u[v] = m0[v];
                z[v] = have_mem0 && (m0[v] > thr[v]);
                ii[v] = s0[v];
              }
            }
          }
        }
        if (active) {
#pragma unroll
          for (int v = 0; v < VEC; ++v)
            fwd_step<SYN>(a.reset, beta[v], thr[v], alpha[v], x[v], u[v], z[v], ii[v]);
          float* su = seg + ((size_t)(t - t0) * nthr + c) * VEC;
          Elem<float>::store4(su, u);
          if (SYN) Elem<float>::store4(su + seg_plane, ii);
        }
        release_item(j);
      }
      if (!ok) break;
      // reverse steps over the segment
      for (int64_t t = t1 - 1; t >= t0; --t, ++j) {
        const unsigned char* base;
        if (!wait_item(j, base)) { ok = false; break; }
        float g[VEC], gmv[VEC];
        if (active) {
          Elem<TO>::load4(reinterpret_cast<const TO*>(base) + c * VEC, g);
          if (a.gm) Elem<TO>::load4(reinterpret_cast<const TO*>(base + io_stride) + c * VEC, gmv);
        }
        if (active) {
          const float* su = seg + ((size_t)(t - t0) * nthr + c) * VEC;
          float uu[VEC], iv[VEC], out[VEC];
          Elem<float>::load4(su, uu);
          if (SYN) Elem<float>::load4(su + seg_plane, iv);
          const bool last = (t == a.T - 1);
#pragma unroll
          for (int v = 0; v < VEC; ++v) {
            const float eu = (a.gm ? gmv[v] : 0.0f) + (last ? ex_u[v] : 0.0f);
            out[v] = bwd_step<SYN>(a, beta[v], thr[v], alpha[v], !last, uu[v], uu[v] > thr[v],
                                   SYN ? iv[v] : 0.0f, g[v], eu, last ? ex_i[v] : 0.0f, st[v]);
          }
          Elem<TO>::store4(gI + t * a.L + l, out);
        }
        release_item(j);
      }
    }
  }
  if (!ok || !active) return;
  float gm0[VEC], gs0[VEC], db[VEC], dt[VEC], da[VEC];
#pragma unroll
  for (int v = 0; v < VEC; ++v) {
    if (a.T == 0) {
      gm0[v] = ex_u[v];
      gs0[v] = ex_i[v];
    } else {
      bwd_initial<SYN>(a, beta[v], thr[v], alpha[v], have_mem0, m0[v], s0[v], st[v], gm0[v], gs0[v]);
    }
    db[v] = st[v].dbeta;
    dt[v] = st[v].dthr;
    da[v] = st[v].dalpha;
  }
  if (a.gmem0) Elem<float>::store4(a.gmem0 + l, gm0);
  if (SYN && a.gsyn0) Elem<float>::store4(a.gsyn0 + l, gs0);
  if (a.part_beta) Elem<float>::store4(a.part_beta + l, db);
  if (a.part_thr) Elem<float>::store4(a.part_thr + l, dt);
  if (SYN && a.part_alpha) Elem<float>::store4(a.part_alpha + l, da);
}

// ---------------------------------------------------------------------------
// Plain kernels: one lane per thread, direct loads, any shape.
// ---------------------------------------------------------------------------

template <bool SYN, typename TI, typename TO>
__global__ void __launch_bounds__(256) scan_fwd_plain(const ScanArgs a) {
  const int64_t l = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (l >= a.L) return;
  const float beta = lane_param(a.beta, a.beta_mode, l, a);
  const float thr = lane_param(a.thr, a.thr_mode, l, a);
  const float alpha = SYN ? lane_param(a.alpha, a.alpha_mode, l, a) : 0.0f;
  float u = a.mem0 ? a.mem0[l] : 0.0f;
  bool z = a.mem0 ? (u > thr) : false;
  float i = (SYN && a.syn0) ? a.syn0[l] : 0.0f;
  const TI* I = static_cast<const TI*>(a.I);
  TO* spk = static_cast<TO*>(a.spk);
  TO* mem = static_cast<TO*>(a.mem);
  TO* syn = static_cast<TO*>(a.syn);
  const int64_t ckpt_stride = SYN ? 2 * a.L : a.L;
  int kk = 0;
  for (int64_t t = 0; t < a.T; ++t) {
    const int64_t off = t * a.L + l;
    fwd_step<SYN>(a.reset, beta, thr, alpha, Elem<TI>::load1(I + off), u, z, i);
    Elem<TO>::store1(spk + off, z ? 1.0f : 0.0f);
    if (mem) Elem<TO>::store1(mem + off, u);
    if (SYN && syn) Elem<TO>::store1(syn + off, i);
    if (++kk == a.K) {
      kk = 0;
      if (a.ckpt && t + 1 < a.T) {
        float* cp = a.ckpt + (t / a.K) * ckpt_stride + l;
        *cp = u;
        if (SYN) cp[a.L] = i;
      }
    }
  }
  if (a.mem_final) a.mem_final[l] = u;
  if (SYN && a.syn_final) a.syn_final[l] = i;
}

template <bool SYN, bool RECOMP, typename TI, typename TO>
__global__ void __launch_bounds__(128) scan_bwd_plain(const ScanArgs a) {
  extern __shared__ __align__(16) float segbuf[];  // [K][blockDim] u, then i
  const int64_t l = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (l >= a.L) return;
  const float beta = lane_param(a.beta, a.beta_mode, l, a);
  const float thr = lane_param(a.thr, a.thr_mode, l, a);
  const float alpha = SYN ? lane_param(a.alpha, a.alpha_mode, l, a) : 0.0f;
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
      Elem<TO>::store1(gI + off, bwd_step<SYN>(a, beta, thr, alpha, !last, u, z, i,
                                               Elem<TO>::load1(gs + off), eu,
                                               last ? ex_i : 0.0f, st));
    }
  } else {
    const TI* I = static_cast<const TI*>(a.I);
    float* su = segbuf + threadIdx.x;
    float* si = segbuf + (size_t)a.K * blockDim.x + threadIdx.x;
    for (int k = a.nseg - 1; k >= 0; --k) {
      const int64_t t0 = (int64_t)k * a.K, t1 = min(a.T, t0 + a.K);
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
        fwd_step<SYN>(a.reset, beta, thr, alpha, Elem<TI>::load1(I + t * a.L + l), u, z, i);
        su[(t - t0) * blockDim.x] = u;
        if (SYN) si[(t - t0) * blockDim.x] = i;
      }
      for (int64_t t = t1 - 1; t >= t0; --t) {
        const int64_t off = t * a.L + l;
        const float uu = su[(t - t0) * blockDim.x];
        const float iv = SYN ? si[(t - t0) * blockDim.x] : 0.0f;
        const bool last = (t == a.T - 1);
        const float eu = (gm ? Elem<TO>::load1(gm + off) : 0.0f) + (last ? ex_u : 0.0f);
        Elem<TO>::store1(gI + off, bwd_step<SYN>(a, beta, thr, alpha, !last, uu, uu > thr, iv,
                                                 Elem<TO>::load1(gs + off), eu,
                                                 last ? ex_i : 0.0f, st));
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
  if (SYN && a.part_alpha) a.part_alpha[l] = st.dalpha;
}

}  // namespace snn
