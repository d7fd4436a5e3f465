// Recompute-variant BPTT of the Leaky neuron (Eq. 4, and Eq. 7 with REC)
// with the replayed segment held in registers.
//
// The forward stored u (fp32) at the end of every checkpoint segment of KC
// steps (segments aligned to the end of the sequence, so only the first can
// be shorter).  The reverse pass walks the segments from last to first.  For
// each segment it
//   1. replays Eq. (4) from the segment's starting state over the segment's
//      rows of I, bit for bit as the forward evaluated it (fwd_pair), and
//      keeps the KC fp32 membrane values of each lane in registers;
//   2. runs the KC reverse steps of the BPTT recurrence (bwd_pair_seg) over the
//      segment's rows of dL/dspk, writing dL/dI.
// (A per-step dL/dmem input takes scan_bwd_staged.)
// A CTA owns a strip of lanes; one producer thread streams, per segment,
// replay items {checkpoint row, rows of I} and gradient items {rows of
// grad_spk} of up to kSegItemRows steps each into a ring of shared-memory
// stages with 1-D bulk copies (one per row), so a consumer warp waits and
// releases once per item rather than per step, and the ring keeps several
// items of loads in flight.  Each consumer thread owns kSegLanes consecutive
// lanes.
//
// Against the shared-memory replay buffer of scan_bwd_staged, the trace
// costs no shared memory and no load or store instructions, so the ring
// takes all of the shared memory.  KC = 16 would halve the checkpoint bytes
// of KC = 8, but at 128 registers a thread it runs slower (0.32 against
// 0.29 ms on the 524,288-lane, T = 500 workload); KC = 8 is the default.
#pragma once

#include "scan_kernels.cuh"

namespace snn {

// Lanes per consumer thread: the trace is KC x kSegLanes fp32 registers.
// Measured slower: 8 lanes at KC = 8 (the trace spills past 128 registers),
// 2 lanes at KC = 16 or 32 (more steps' overhead per lane, and three waves).
template <int KC>
constexpr int kSegLanes = 4;

// One reverse step at time t on a pair of lanes (u = u_t, z = z_t as 0/1
// floats), the compact form of bwd_pair for the fully unrolled segment loop:
// the extra gradient eu (grad_mem_final at t = T-1; zero otherwise) is
// always added, so that one copy of the step serves every t.
// s.du holds dL/du_{t+1} on entry and dL/du_t on exit; s.dthr accumulates
// the negated threshold gradient.  Returns dL/dI_t.
//
// The arctan surrogate is evaluated as 1 / (1/a + (c u - c thr)^2) with
// c = b / sqrt(a) (a = alpha/2, b = pi alpha/2): the same function as
// a / (1 + (b (u - thr))^2) in two packed operations and the reciprocal.
// sgt holds -c*thr of the pair's lanes, sgc = c and sgi = 1/a.
template <int RESET, int SG, bool REC>
__device__ __forceinline__ float2 bwd_pair_seg(const ScanArgs& a, float2 beta, float2 negthr,
                                               float2 sgt, float sgc, float sgi, float2 v,
                                               float2 u, float2 z, float2 gs, float2 eu,
                                               Bwd2& s) {
  const float2 omz = make_float2(1.0f - z.x, 1.0f - z.y);
  // parameter terms of step t+1 that need the step-t state
  if (RESET == RESET_ZERO) s.dbeta = fma2(s.du, mul2(omz, u), s.dbeta);  // (1-z_t) u_t
  else s.dbeta = fma2(s.du, u, s.dbeta);
  if (RESET == RESET_SUBTRACT) s.dthr = fma2(z, s.du, s.dthr);  // d u_{t+1}/d thr = -z_t
  if (REC) s.dalpha = fma2(z, s.du, s.dalpha);                   // d u_{t+1}/d v = z_t
  float2 sg;
  if (SG == SG_ATAN) {
    const float2 y = fma2(f2(sgc), u, sgt);
    const float2 d = fma2(y, y, f2(sgi));
    sg = make_float2(rcp_ge1(d.x), rcp_ge1(d.y));
  } else {
    sg = surrogate2<SG>(a, add2(u, negthr));
  }
  float2 dz = gs;
  if (!a.detach) {
    if (RESET == RESET_SUBTRACT) dz = fma2(negthr, s.du, dz);
    else if (RESET == RESET_ZERO) dz = fma2(mul2(f2(-1.0f), mul2(beta, u)), s.du, dz);
  }
  if (REC) dz = fma2(v, s.du, dz);  // the recurrent connection, never detached
  const float2 p = mul2(sg, dz);
  const float2 decay = RESET == RESET_ZERO ? mul2(beta, omz) : beta;
  s.du = add2(fma2(decay, s.du, p), eu);
  s.dthr = add2(s.dthr, p);
  return s.du;
}

// Rows per ring item of the register-segment BPTT: a segment of KC steps is
// streamed as KC / kSegItemRows replay items and as many gradient items
// (whole segments up to 16 steps: 8-row items measured slower at KC = 16).
constexpr int kSegItemRows = 16;

template <typename TI, typename TO, int RESET, int SG, int KC, bool REC>
__global__ void __launch_bounds__(kMaxStagedThreads) scan_bwd_seg(const ScanArgs a) {
  constexpr int V = kSegLanes<KC>, NP = V / 2;
  constexpr int RH = KC < kSegItemRows ? KC : kSegItemRows, NH = KC / RH;
  extern __shared__ __align__(1024) unsigned char smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem);
  uint64_t* empty = full + kMaxStages;
  unsigned char* ring = smem + kBarrierBytes;
  const int S = a.stages;
  const int cwarps = (int)(blockDim.x >> 5) - 1;
  const int warp = threadIdx.x >> 5, lid = threadIdx.x & 31;
  const int64_t lane0 = (int64_t)blockIdx.x * a.lanes_per_cta;
  const int cta_lanes = (int)min((int64_t)a.lanes_per_cta, a.L - lane0);
  // stage layout: replay item = [checkpoint row fp32 (first item of a
  // segment)][RH rows of I]; gradient item = [RH rows of grad_spk]
  const int lpc = a.lanes_per_cta;
  const uint32_t ck_bytes = (uint32_t)lpc * 4u;
  const uint32_t in_row = (uint32_t)lpc * (uint32_t)sizeof(TI);
  const uint32_t io_row = (uint32_t)lpc * (uint32_t)sizeof(TO);
  init_ring_barriers(full, empty, S, cwarps);
  grid_dep_wait();  // the previous kernel on the stream is complete

  if (warp == cwarps) {
    if (lid == 0 && !(a.debug & DEBUG_PRODUCER_IDLE)) {
      Producer p{ring, full, empty, S, a.stage_bytes};
      const uint32_t bi = (uint32_t)cta_lanes * (uint32_t)sizeof(TI);
      const uint32_t bo = (uint32_t)cta_lanes * (uint32_t)sizeof(TO);
      const uint32_t bc = (uint32_t)cta_lanes * 4u;
      for (int k = a.nseg - 1; k >= 0; --k) {
        int64_t t0, t1;
        seg_bounds(a, k, t0, t1);
        const int Kk = (int)(t1 - t0);
        bool go = true;
        for (int h = 0; h < NH && go; ++h) {  // replay items, in time order
          const int r0 = h * RH, nr = min(RH, Kk - r0);
          if (nr <= 0) break;
          const bool ck = (h == 0 && k > 0);
          if (!(go = p.begin((ck ? bc : 0u) + (uint32_t)nr * bi, a))) break;
          if (ck)  // the segment's starting state, checkpoint rows fp32 [nseg-1][L]
            p.copy(0, a.ckpt + (int64_t)(k - 1) * a.L + lane0, bc);
          for (int r = 0; r < nr; ++r)
            p.copy(ck_bytes + (uint32_t)r * in_row, row<TI>(a.I, t0 + r0 + r, a.L, lane0), bi);
          p.end();
        }
        for (int h = NH - 1; h >= 0 && go; --h) {  // gradient items, last half first
          const int r0 = h * RH, nr = min(RH, Kk - r0);
          if (nr <= 0) continue;
          if (!(go = p.begin((uint32_t)nr * bo, a))) break;
          for (int r = 0; r < nr; ++r)
            p.copy((uint32_t)r * io_row, row<TO>(a.gs, t0 + r0 + r, a.L, lane0), bo);
          p.end();
        }
        if (!go) break;
      }
      p.drain();
    }
    return;
  }

  const int c = threadIdx.x;
  RingPos pos;
  bool ok = true;
  const int64_t l = lane0 + (int64_t)c * V;
  const bool active = c * V < cta_lanes;
  float2 beta[NP], negthr[NP], alpha[NP], third[NP];
  Bwd2 st[NP];
  if (active) load_params<REC, NP>(a, l, beta, negthr, alpha);
#pragma unroll
  for (int q = 0; q < NP; ++q) {
    st[q] = Bwd2{f2(0.0f), f2(0.0f), f2(0.0f), f2(0.0f), f2(0.0f)};
    third[q] = REC ? add2_rn(alpha[q], negthr[q]) : f2(0.0f);  // v - thr, rounded once
  }
  const float2 zero2 = f2(0.0f);
  // arctan surrogate constants (see bwd_pair_seg)
  const float sgc = SG == SG_ATAN ? a.sg_b * rsqrtf(a.sg_a) : 0.0f;
  const float sgi = SG == SG_ATAN ? 1.0f / a.sg_a : 0.0f;
  float2 sgt[NP];
#pragma unroll
  for (int q = 0; q < NP; ++q) sgt[q] = mul2(negthr[q], f2(sgc));
  float2 gmf[NP];  // dL/du_{T-1} through the returned final state
#pragma unroll
  for (int q = 0; q < NP; ++q) gmf[q] = zero2;
  if (active && a.gmf) load_pairs_global<NP>(a.gmf + l, gmf);
  for (int k = a.nseg - 1; k >= 0; --k) {
    int64_t t0, t1;
    seg_bounds(a, k, t0, t1);
    const int Kk = (int)(t1 - t0);
    float2 tr[KC][NP];  // the replayed u_t of the segment, t = t0 + j

    // 1. replay Eq. (4) from the segment's starting state, item by item
    float2 u[NP], z[NP];
#pragma unroll
    for (int h = 0; h < NH; ++h) {
      if (h * RH >= Kk) break;
      if (!warp_wait(&full[pos.s], pos.ph, a.wait_ns)) {
        if (lid == 0) record_status(a.status, kStatusTimeout);
        ok = false;
        break;
      }
      if (active) {
        const unsigned char* stage = ring + (size_t)pos.s * a.stage_bytes;
        if (h == 0) {
          if (k > 0) {
            load_pairs<float, NP>(reinterpret_cast<const float*>(stage) + c * V, u);
#pragma unroll
            for (int q = 0; q < NP; ++q) z[q] = fire2(u[q], negthr[q]);
          } else {
            bool zb[V];
            float2 idummy[NP];
            initial_state<false, NP>(a, l, negthr, u, zb, idummy);
#pragma unroll
            for (int q = 0; q < NP; ++q)
              z[q] = make_float2(zb[2 * q] ? 1.0f : 0.0f, zb[2 * q + 1] ? 1.0f : 0.0f);
          }
        }
        const TI* xin = reinterpret_cast<const TI*>(stage + ck_bytes) + c * V;
#pragma unroll
        for (int r = 0; r < RH; ++r) {
          const int j = h * RH + r;
          if (j < Kk) {
            float2 x[NP], idummy = zero2;
            load_pairs<TI, NP>(xin + r * lpc, x);
#pragma unroll
            for (int q = 0; q < NP; ++q) {
              fwd_pair<false, RESET, REC ? 1 : 0>(a.reset, beta[q], negthr[q], third[q], x[q],
                                                  u[q], z[q], idummy);
              tr[j][q] = u[q];
            }
          }
        }
      }
      release_stage(empty, pos.s, lid);
      pos.next(S);
    }
    if (!ok) break;

    // 2. the segment's reverse steps, last item first
    TO* gout = static_cast<TO*>(a.gI) + l + t0 * a.L;
    const bool last_seg = (k == a.nseg - 1);
#pragma unroll
    for (int h = NH - 1; h >= 0; --h) {
      if (h * RH >= Kk) continue;
      if (!warp_wait(&full[pos.s], pos.ph, a.wait_ns)) {
        if (lid == 0) record_status(a.status, kStatusTimeout);
        ok = false;
        break;
      }
      if (active) {
        const TO* gin = reinterpret_cast<const TO*>(ring + (size_t)pos.s * a.stage_bytes) + c * V;
#pragma unroll
        for (int r = RH - 1; r >= 0; --r) {
          const int j = h * RH + r;
          if (j < Kk) {
            float2 g[NP], eu[NP], out[NP];
            load_pairs<TO, NP>(gin + r * lpc, g);
#pragma unroll
            for (int q = 0; q < NP; ++q) eu[q] = zero2;
            if (last_seg && j == Kk - 1) {  // t = T-1: the final state's gradient
#pragma unroll
              for (int q = 0; q < NP; ++q) eu[q] = add2(eu[q], gmf[q]);
            }
#pragma unroll
            for (int q = 0; q < NP; ++q)
              out[q] = bwd_pair_seg<RESET, SG, REC>(
                  a, beta[q], negthr[q], sgt[q], sgc, sgi, alpha[q], tr[j][q],
                  fire2(tr[j][q], negthr[q]), g[q], eu[q], st[q]);
            store_pairs<TO, NP>(gout + j * a.L, out);
          }
        }
      }
      release_stage(empty, pos.s, lid);
      pos.next(S);
    }
    if (!ok) break;
  }
  if (!ok || !active) return;
  float gm0[V], db[V], dt[V], da[V];
#pragma unroll
  for (int v = 0; v < V; ++v) {
    const Bwd2& q = st[v / 2];
    const bool hi = v & 1;
    BwdLane sl{hi ? q.du.y : q.du.x, 0.0f, hi ? q.dbeta.y : q.dbeta.x,
               -(hi ? q.dthr.y : q.dthr.x), hi ? q.dalpha.y : q.dalpha.x};
    const float b = hi ? beta[v / 2].y : beta[v / 2].x;
    const float th = -(hi ? negthr[v / 2].y : negthr[v / 2].x);
    const float al = hi ? alpha[v / 2].y : alpha[v / 2].x;
    if (a.T == 0) {
      gm0[v] = a.gmf ? a.gmf[l + v] : 0.0f;
    } else {
      float gs0;
      const float m0 = a.mem0 ? a.mem0[l + v] : 0.0f;
      bwd_initial<false>(a, b, th, al, a.mem0 != nullptr, m0, 0.0f, sl, gm0[v], gs0);
    }
    db[v] = sl.dbeta;
    dt[v] = sl.dthr;
    da[v] = sl.dalpha;
  }
  if (a.gmem0) storev<float, V>(a.gmem0 + l, gm0);
  if (a.part_beta) storev<float, V>(a.part_beta + l, db);
  if (a.part_thr) storev<float, V>(a.part_thr + l, dt);
  if (REC && a.part_alpha) storev<float, V>(a.part_alpha + l, da);
}

}  // namespace snn
