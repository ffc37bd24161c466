// env_overcooked.cuh -- the 5x4 Overcooked-style kitchen on the device (one thread per env).
//
// Layout (x right, y down):  row 0 "#O#P#", row 1 "#...#", row 2 "D...S", row 3 "##O##"
// (# counter, O onion dispenser, P pot, D dish dispenser, S serving cell, . floor).
// Actions {noop, N, S, E, W, interact}; a full pot (3 onions) cooks for cook_time steps;
// a served soup pays soup_reward to the team.  A move sets the facing and enters floor
// only (equal targets or a swap: both stay); interact acts on the faced cell, agent 0
// first; a pot cooking at the start of a step counts down at its end; episodes have a
// fixed length and a shared reward only.
#pragma once
#include "aht_common.cuh"

namespace aht {

// Cell types: 0 floor, 1 counter, 2 onion dispenser, 3 pot, 4 dish dispenser, 5 serving;
// cell c = y * 5 + x of the layout above.
__host__ __device__ constexpr int kitchen_type(int c) {
  return (c == 1 || c == 17) ? 2
         : c == 3            ? 3
         : c == 10           ? 4
         : c == 14           ? 5
         : (c == 6 || c == 7 || c == 8 || c == 11 || c == 12 || c == 13) ? 0
                                                                          : 1;
}
// the same table in constant memory, for cells indexed at run time
__constant__ uint8_t kKitchenCell[20] = {
    kitchen_type(0),  kitchen_type(1),  kitchen_type(2),  kitchen_type(3),  kitchen_type(4),
    kitchen_type(5),  kitchen_type(6),  kitchen_type(7),  kitchen_type(8),  kitchen_type(9),
    kitchen_type(10), kitchen_type(11), kitchen_type(12), kitchen_type(13), kitchen_type(14),
    kitchen_type(15), kitchen_type(16), kitchen_type(17), kitchen_type(18), kitchen_type(19)};

// The observation bits that depend only on the layout (each cell's type channel) and on
// the urgency flag (channel 25 of every cell), as 32-bit words (bit k % 32 of word k / 32).
constexpr int kOcObsBits = 20 * 26;
constexpr int kOcObsWords = (kOcObsBits + 31) / 32;
struct OcObsMasks {
  uint32_t layout[kOcObsWords], urgent[kOcObsWords];
};
__host__ __device__ constexpr int oc_type_channel(int t) {
  return t == 1 ? 10 : t == 2 ? 12 : t == 3 ? 11 : t == 4 ? 13 : t == 5 ? 14 : -1;
}
__host__ __device__ constexpr OcObsMasks oc_obs_masks() {
  OcObsMasks m{};
  for (int c = 0; c < 20; ++c) {
    const int ch = oc_type_channel(kitchen_type(c));
    if (ch >= 0) m.layout[(c * 26 + ch) >> 5] |= 1u << ((c * 26 + ch) & 31);
    m.urgent[(c * 26 + 25) >> 5] |= 1u << ((c * 26 + 25) & 31);
  }
  return m;
}

struct EnvOvercooked {
  static constexpr bool kTurnBased = false;
  static constexpr int kNumActions = 6;
  enum : uint8_t { kNone = 0, kOnion = 1, kDish = 2, kSoup = 3 };
  struct State {
    uint8_t ax[2], ay[2];
    uint8_t face[2], held[2];  // face 0 N, 1 S, 2 E, 3 W
    uint8_t pot_n, pot_timer, pad0, pad1;
    uint8_t item[20];          // item lying on each cell (counters only)
    uint32_t ep_t;
    float ret;
  };
  static constexpr int kWords = sizeof(State) / 4;

  __device__ static int cell(int x, int y) {
    return (x < 0 || x >= 5 || y < 0 || y >= 4) ? -1 : kKitchenCell[y * 5 + x];
  }
  __device__ static void facing(int f, int& dx, int& dy) {
    dx = (f == 2) - (f == 3);
    dy = (f == 1) - (f == 0);
  }

  __device__ static void reset(const DevEnv&, Key, uint32_t, uint32_t, State& s) {
    s.ax[0] = 1; s.ay[0] = 1;
    s.ax[1] = 3; s.ay[1] = 2;
    s.face[0] = s.face[1] = 0;
    s.held[0] = s.held[1] = kNone;
    s.pot_n = 0;
    s.pot_timer = 0;
    s.pad0 = s.pad1 = 0;
    for (int c = 0; c < 20; ++c) s.item[c] = kNone;
    s.ep_t = 0;
    s.ret = 0.0f;
  }

  __device__ static int step(const DevEnv& d, State& s, int a0, int a1, float& r0, float& r1,
                             float& team) {
    const bool was_cooking = s.pot_n == 3 && s.pot_timer > 0;
    const int act[2] = {a0, a1};
    int px[2], py[2];
    for (int i = 0; i < 2; ++i) {
      px[i] = s.ax[i];
      py[i] = s.ay[i];
      if (act[i] >= 1 && act[i] <= 4) {
        s.face[i] = (uint8_t)(act[i] - 1);
        int dx, dy;
        facing(s.face[i], dx, dy);
        if (cell(s.ax[i] + dx, s.ay[i] + dy) == 0) {
          px[i] = s.ax[i] + dx;
          py[i] = s.ay[i] + dy;
        }
      }
    }
    const bool collide = (px[0] == px[1] && py[0] == py[1]) ||
                         (px[0] == s.ax[1] && py[0] == s.ay[1] && px[1] == s.ax[0] && py[1] == s.ay[0]);
    if (!collide) {
      for (int i = 0; i < 2; ++i) {
        s.ax[i] = (uint8_t)px[i];
        s.ay[i] = (uint8_t)py[i];
      }
    }
    float reward = 0.0f;
    for (int i = 0; i < 2; ++i) {
      if (act[i] != 5) continue;
      int dx, dy;
      facing(s.face[i], dx, dy);
      const int cx = s.ax[i] + dx, cy = s.ay[i] + dy;
      const int c = cell(cx, cy);
      uint8_t h = s.held[i];
      if (c == 2) {
        if (h == kNone) h = kOnion;
      } else if (c == 4) {
        if (h == kNone) h = kDish;
      } else if (c == 3) {
        if (h == kOnion && s.pot_n < 3) {
          h = kNone;
          s.pot_n += 1;
          if (s.pot_n == 3) s.pot_timer = (uint8_t)d.cook_time;
        } else if (h == kDish && s.pot_n == 3 && s.pot_timer == 0) {
          h = kSoup;
          s.pot_n = 0;
          s.pot_timer = 0;
        }
      } else if (c == 5) {
        if (h == kSoup) {
          h = kNone;
          reward = __fadd_rn(reward, (float)d.soup_reward);
        }
      } else if (c == 1) {
        uint8_t& it = s.item[cy * 5 + cx];
        if (h != kNone && it == kNone) {
          it = h;
          h = kNone;
        } else if (h == kNone && it != kNone) {
          h = it;
          it = kNone;
        }
      }
      s.held[i] = h;
    }
    if (was_cooking && s.pot_timer > 0) s.pot_timer -= 1;
    s.ep_t += 1;
    r0 = reward;
    r1 = reward;
    team = reward;
    s.ret = __fadd_rn(s.ret, reward);
    return (int)s.ep_t == d.episode_len ? 1 : 0;
  }

  // 26 binary channels per cell, index (y*5 + x)*26 + c.
  __device__ static bool urgent(const DevEnv& d, const State& s) { return d.episode_len - (int)s.ep_t <= 40; }
  // the channels that change with the state: items on counters, the pot, the agents
  template <class Row>
  __device__ static void obs_state_bits(const State& s, int seat, Row& row) {
#pragma unroll
    for (int c = 0; c < 20; ++c) {
      const int o = c * 26;
      const int t = kitchen_type(c);
      if (t == 1) {
        if (s.item[c] != kNone) row.set(o + 14 + s.item[c], 1);
      } else if (t == 3) {
        if (s.pot_n >= 1) row.set(o + 17 + s.pot_n, 1);
        if (s.pot_n == 3) row.set(o + (s.pot_timer > 0 ? 21 : 22), 1);
      }
    }
    for (int who = 0; who < 2; ++who) {
      const int i = who == 0 ? seat : 1 - seat;
      const int o = (s.ay[i] * 5 + s.ax[i]) * 26;
      row.set(o + who, 1);
      row.set(o + 2 + 4 * who + s.face[i], 1);
      if (s.held[i] != kNone) {
        row.set(o + 23 + who, 1);
        row.set(o + 14 + s.held[i], 1);
      }
    }
  }
  template <class Row>
  __device__ static void obs_into(const DevEnv& d, const State& s, int seat, Row& row) {
    row.clear();
    const bool urg = urgent(d, s);
    for (int c = 0; c < 20; ++c) {
      const int ch = oc_type_channel(kKitchenCell[c]);
      if (ch >= 0) row.set(c * 26 + ch, 1);
      if (urg) row.set(c * 26 + 25, 1);
    }
    obs_state_bits(s, seat, row);
  }
  // The same bits into a word row (the streamed cross-play kernel): the layout and urgency
  // channels as whole words, then the state's channels bit by bit.
  __device__ static void obs_into(const DevEnv& d, const State& s, int seat, ObsBits& row) {
    constexpr OcObsMasks M = oc_obs_masks();
    const uint32_t u = urgent(d, s) ? 0xFFFFFFFFu : 0u;
#pragma unroll
    for (int i = 0; i < kOcObsWords; ++i) row.w[i] = M.layout[i] | (M.urgent[i] & u);
    for (int i = kOcObsWords; i < row.words; ++i) row.w[i] = 0u;
    obs_state_bits(s, seat, row);
  }
  __device__ static void obs(const DevEnv& d, const State& s, int seat, uint8_t* row) {
    ObsBytes w{row, 130};
    obs_into(d, s, seat, w);
  }

  __device__ static uint32_t legal(const State&) { return 0x3Fu; }
  __device__ static int actor(const State&) { return -1; }
  __device__ static float ret(const State& s) { return s.ret; }
};

}  // namespace aht
