// env_lbf.cuh -- Level-Based Foraging on the device (one thread per env).
//
// Rules (the workload's statement; the paper fixes none, Sec. 4 Table): two agents with levels in
// 1..max_level, n_food foods with levels in 1..(sum of agent levels); actions
// {noop, N, S, W, E, load}; a food is eaten when the summed levels of the 4-adjacent
// loading agents reach its level, each loader receiving food_level*agent_level /
// (loader_level_sum * total_food_level).  Moves resolve on the pre-step state.
#pragma once
#include "aht_common.cuh"

namespace aht {

struct EnvLbf {
  static constexpr bool kTurnBased = false;
  static constexpr int kNumActions = 6;
  struct State {
    uint8_t ax[2], ay[2];
    uint8_t al[2], F, eaten;  // eaten: bit k set when food k is gone (absent foods too)
    uint8_t fx[4], fy[4], fl[4];  // slot 3 of fx / fy: agent 1's position at the episode start
    uint32_t ep_t;
    float ret;
  };
  static constexpr int kWords = sizeof(State) / 4;

  __device__ static void reset(const DevEnv& d, Key key, uint32_t env, uint32_t step, State& s) {
    DrawSeq r(key, env, step, kStreamReset);
    s.al[0] = (uint8_t)(1 + uniform_int(r.next(), (uint32_t)d.max_level));
    s.al[1] = (uint8_t)(1 + uniform_int(r.next(), (uint32_t)d.max_level));
    const uint32_t lsum = s.al[0] + s.al[1];
    uint32_t F = 0;
#pragma unroll
    for (int k = 0; k < 3; ++k) {  // fixed trip count: the state stays in registers
      if (k < d.n_food) {
        s.fl[k] = (uint8_t)(1 + uniform_int(r.next(), lsum));
        F += s.fl[k];
      }
    }
    s.F = (uint8_t)F;
    // n_food + 2 steps of a Fisher-Yates shuffle of the cell indices (identity at the
    // start).  Step i swaps positions i and j >= i; position i is final afterwards and
    // never read again, so only the values written to the j's need remembering: wpos[m],
    // wval[m] for step m (a later write to the same position wins).  Fixed-size loops keep
    // everything in registers.
    const int cells = d.width * d.height;
    const int n_obj = d.n_food + 2;
    int wpos[5], wval[5], placed[5];
    int c0 = 0, c1 = 0;  // the agents' cells, placed[n_food] and placed[n_food + 1]
#pragma unroll
    for (int i = 0; i < 5; ++i) {
      if (i < n_obj) {
        const int j = i + (int)uniform_int(r.next(), (uint32_t)(cells - i));
        int vi = i, vj = j;
#pragma unroll
        for (int m = 0; m < i; ++m) {
          if (wpos[m] == i) vi = wval[m];
          if (wpos[m] == j) vj = wval[m];
        }
        placed[i] = vj;  // position i now holds the old value at j
        wpos[i] = j;     // and position j the old value at i
        wval[i] = vi;
        if (i == n_obj - 2) c0 = vj;  // taken as they are placed: a runtime index into
        if (i == n_obj - 1) c1 = vj;  // placed[] would move it out of registers
      } else {
        placed[i] = 0;
        wpos[i] = -1;
        wval[i] = 0;
      }
    }
    // cell -> (x, y): one division for the grid's reciprocal, then y = floor(c * m / 2^32)
    // with m = ceil(2^32 / width), exact for c, width < 2^16
    const uint32_t wd = (uint32_t)d.width, m = 0xFFFFFFFFu / wd + 1u;
    auto cell_y = [&](int c) { return __umulhi((uint32_t)c, m); };
    s.eaten = 0;
#pragma unroll
    for (int k = 0; k < 3; ++k) {
      if (k < d.n_food) {
        const uint32_t y = cell_y(placed[k]);
        s.fx[k] = (uint8_t)((uint32_t)placed[k] - y * wd);
        s.fy[k] = (uint8_t)y;
      } else {
        s.fx[k] = s.fy[k] = s.fl[k] = 0;
        s.eaten |= (uint8_t)(1u << k);
      }
    }
    s.fl[3] = 0;
    const uint32_t y0 = cell_y(c0), y1 = cell_y(c1);
    s.ax[0] = (uint8_t)((uint32_t)c0 - y0 * wd);
    s.ay[0] = (uint8_t)y0;
    s.ax[1] = (uint8_t)((uint32_t)c1 - y1 * wd);
    s.ay[1] = (uint8_t)y1;
    s.fx[3] = s.ax[1];  // the start position a Sequential teammate plans from
    s.fy[3] = s.ay[1];
    s.ep_t = 0;
    s.ret = 0.0f;
  }

  // Loops run over all three food slots: absent foods are marked eaten at reset, so the
  // fixed trip counts keep the state in registers when the caller holds a copy.
  __device__ static int step(const DevEnv& d, State& s, int a0, int a1, float& r0, float& r1,
                             float& team) {
    r0 = 0.0f;
    r1 = 0.0f;
    uint32_t newly = 0;
    const int ax0 = s.ax[0], ay0 = s.ay[0], ax1 = s.ax[1], ay1 = s.ay[1];
    if (a0 == 5 || a1 == 5) {
#pragma unroll
      for (int k = 0; k < 3; ++k) {
        if ((s.eaten >> k) & 1u) continue;
        const int fx = s.fx[k], fy = s.fy[k], fl = s.fl[k];
        const bool l0 = a0 == 5 && abs(ax0 - fx) + abs(ay0 - fy) == 1;
        const bool l1 = a1 == 5 && abs(ax1 - fx) + abs(ay1 - fy) == 1;
        const int lsum = (l0 ? s.al[0] : 0) + (l1 ? s.al[1] : 0);
        if (lsum > 0 && lsum >= fl) {
          newly |= 1u << k;
          const float den = (float)(lsum * (int)s.F);
          if (l0) r0 = __fadd_rn(r0, __fdiv_rn((float)(fl * s.al[0]), den));
          if (l1) r1 = __fadd_rn(r1, __fdiv_rn((float)(fl * s.al[1]), den));
        }
      }
    }
    int tx[2], ty[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int a = i == 0 ? a0 : a1;
      const int cx = i == 0 ? ax0 : ax1, cy = i == 0 ? ay0 : ay1;
      const int dx = (a == 4) - (a == 3), dy = (a == 2) - (a == 1);
      const int x = cx + dx, y = cy + dy;
      bool ok = (dx | dy) != 0 && x >= 0 && x < d.width && y >= 0 && y < d.height;
#pragma unroll
      for (int k = 0; k < 3; ++k)
        if (!((s.eaten >> k) & 1u) && s.fx[k] == x && s.fy[k] == y) ok = false;
      if ((ax0 == x && ay0 == y) || (ax1 == x && ay1 == y)) ok = false;
      tx[i] = ok ? x : cx;
      ty[i] = ok ? y : cy;
    }
    if (!(tx[0] == tx[1] && ty[0] == ty[1])) {
      s.ax[0] = (uint8_t)tx[0];
      s.ay[0] = (uint8_t)ty[0];
      s.ax[1] = (uint8_t)tx[1];
      s.ay[1] = (uint8_t)ty[1];
    }
    s.eaten |= (uint8_t)newly;
    s.ep_t += 1;
    team = __fadd_rn(r0, r1);
    s.ret = __fadd_rn(s.ret, team);
    return (s.eaten == 7u || (int)s.ep_t == d.episode_len) ? 1 : 0;
  }

  // Level-scaled one-hot per cell: channel 0 own level, 1 other's level, 2 food level,
  // 3 = 1 for an empty cell.  One 32-bit word per cell (channel c in byte c).
  __device__ static void obs(const DevEnv& d, const State& s, int seat, uint8_t* row) {
    uint32_t* w = reinterpret_cast<uint32_t*>(row);
    const int cells = d.width * d.height;
    for (int c = 0; c < cells; ++c) w[c] = 0x01000000u;
    for (int k = 0; k < d.n_food; ++k)
      if (!((s.eaten >> k) & 1u)) w[s.fy[k] * d.width + s.fx[k]] = (uint32_t)s.fl[k] << 16;
    const int o = 1 - seat;
    w[s.ay[o] * d.width + s.ax[o]] = (uint32_t)s.al[o] << 8;
    w[s.ay[seat] * d.width + s.ax[seat]] = (uint32_t)s.al[seat];
  }

  // The observation as changes to the all-empty pattern (every cell word 0x01000000):
  // slot i (foods 0-2, the other agent, the agent itself) is the cell's two changed
  // features, +value in its channel and -1 in channel 3, as entries (feature << 8) |
  // (delta & 0xFF) in e[2i], e[2i + 1].  Returns the mask of the entries in use (eaten
  // foods have none).  The rules keep occupied cells distinct, so this equals obs().
  __device__ static uint32_t sparse_obs(const DevEnv& d, const State& s, int seat, uint32_t (&e)[10]) {
    auto cell = [&](int i, int x, int y, int ch, int v) {
      const uint32_t c = (uint32_t)(y * d.width + x);
      e[2 * i] = ((4u * c + (uint32_t)ch) << 8) | (uint32_t)(v & 0xFF);
      e[2 * i + 1] = ((4u * c + 3u) << 8) | 0xFFu;
    };
    uint32_t mask = 0x3C0u;
#pragma unroll
    for (int k = 0; k < 3; ++k) {
      cell(k, s.fx[k], s.fy[k], 2, s.fl[k]);
      if (!((s.eaten >> k) & 1u)) mask |= 3u << (2 * k);
    }
    cell(3, s.ax[1 - seat], s.ay[1 - seat], 1, s.al[1 - seat]);
    cell(4, s.ax[seat], s.ay[seat], 0, s.al[seat]);
    return mask;
  }

  // The other seat's view of one cell word of the observation: channels 0 (the observing
  // agent's level) and 1 (the other agent's level) trade places; the food and empty
  // channels do not depend on the seat.
  __device__ static uint32_t other_seat_word(uint32_t w) { return __byte_perm(w, 0u, 0x3201); }

  // Words [w0, w1) of the same row (w1 <= cells): one cell per word.
  __device__ static void obs_words(const DevEnv& d, const State& s, int seat, uint32_t* w, int w0,
                                   int w1) {
    for (int c = w0; c < w1; ++c) w[c] = 0x01000000u;
    auto put = [&](int x, int y, uint32_t v) {
      const int c = y * d.width + x;
      if (c >= w0 && c < w1) w[c] = v;
    };
#pragma unroll
    for (int k = 0; k < 3; ++k)  // absent foods are marked eaten
      if (!((s.eaten >> k) & 1u)) put(s.fx[k], s.fy[k], (uint32_t)s.fl[k] << 16);
    // the agents by selection, not by a runtime index (which would move the state copy
    // out of registers)
    const bool s1 = seat != 0;
    put(s1 ? s.ax[0] : s.ax[1], s1 ? s.ay[0] : s.ay[1], (uint32_t)(s1 ? s.al[0] : s.al[1]) << 8);
    put(s1 ? s.ax[1] : s.ax[0], s1 ? s.ay[1] : s.ay[0], (uint32_t)(s1 ? s.al[1] : s.al[0]));
  }

  // Rule-based teammate k in seat 1 (the LBF heuristic suite: Greedy criteria 0..4,
  // Sequential orderings 5..10, Entitled 11): the cell to go for, then load when there,
  // else a step along the axis with the larger remaining distance (ties: x), else along
  // the other axis, when the cell is on the grid and free of uneaten food and of agent 0.
  // Greedy and Sequential go for a food and load when 4-adjacent to it; Entitled takes
  // the lowest-index uneaten food's pair of squares (its first two neighbours W, E, N, S
  // on the grid and free of uneaten food) and waits until agent 0 stands on one of them,
  // then goes for the other and loads there.
  __device__ __noinline__ static int heuristic(const DevEnv& d, const State& s, int k) {
    const int x = s.ax[1], y = s.ay[1], ox = s.ax[0], oy = s.ay[0];
    auto food_at = [&](int cx, int cy) {
#pragma unroll
      for (int f = 0; f < 3; ++f)
        if (!((s.eaten >> f) & 1u) && s.fx[f] == cx && s.fy[f] == cy) return true;
      return false;
    };
    auto free_cell = [&](int cx, int cy) {
      if (cx < 0 || cx >= d.width || cy < 0 || cy >= d.height) return false;
      return !food_at(cx, cy) && !(ox == cx && oy == cy);
    };
    auto step_to = [&](int tx, int ty) {
      const int dx = tx - x, dy = ty - y;
      const int sx = dx > 0 ? 1 : -1, sy = dy > 0 ? 1 : -1;
      const bool xmove = dx != 0 && free_cell(x + sx, y);
      const bool ymove = dy != 0 && free_cell(x, y + sy);
      const int x_act = dx > 0 ? 4 : 3, y_act = dy > 0 ? 2 : 1;
      if (abs(dx) >= abs(dy)) return xmove ? x_act : (ymove ? y_act : 0);
      return ymove ? y_act : (xmove ? x_act : 0);
    };
    if (k == 11) {
      int f = 0;
      while (f < 3 && ((s.eaten >> f) & 1u)) ++f;
      if (f == 3) return 0;
      const int cx = s.fx[f], cy = s.fy[f];
      int px[2], py[2], n = 0;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int nx = cx + (q == 0 ? -1 : q == 1 ? 1 : 0);
        const int ny = cy + (q == 2 ? -1 : q == 3 ? 1 : 0);
        if (n < 2 && nx >= 0 && nx < d.width && ny >= 0 && ny < d.height && !food_at(nx, ny)) {
          px[n] = nx;
          py[n] = ny;
          ++n;
        }
      }
      if (n < 2) return 0;
      int q;
      if (ox == px[0] && oy == py[0]) q = 1;
      else if (ox == px[1] && oy == py[1]) q = 0;
      else return 0;
      if (x == px[q] && y == py[q]) return 5;
      return step_to(px[q], py[q]);
    }
    int target = -1, best = 0;
#pragma unroll
    for (int f = 0; f < 3; ++f) {
      if ((s.eaten >> f) & 1u) continue;  // absent foods are marked eaten
      const int fx = s.fx[f], fy = s.fy[f];
      const int d_me = abs(x - fx) + abs(y - fy), d_tm = abs(ox - fx) + abs(oy - fy);
      const int d_start = abs((int)s.fx[3] - fx) + abs((int)s.fy[3] - fy);
      const int rm = fy * d.width + fx, cm = fx * d.height + fy;
      int key;
      switch (k) {
        case 0: key = d_me; break;
        case 1: key = d_tm; break;
        case 2: key = d_me + d_tm; break;
        case 3: key = s.fl[f]; break;
        case 4: key = -(int)s.fl[f]; break;
        case 5: key = rm; break;
        case 6: key = -rm; break;
        case 7: key = cm; break;
        case 8: key = -cm; break;
        case 9: key = d_start; break;
        default: key = -d_start; break;
      }
      if (target < 0 || key < best) {
        target = f;
        best = key;
      }
    }
    if (target < 0) return 0;
    if (abs((int)s.fx[target] - x) + abs((int)s.fy[target] - y) == 1) return 5;
    return step_to(s.fx[target], s.fy[target]);
  }

  __device__ static uint32_t legal(const State&) { return 0x3Fu; }
  __device__ static int actor(const State&) { return -1; }
  __device__ static float ret(const State& s) { return s.ret; }
};

}  // namespace aht
