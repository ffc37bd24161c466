// aht_oracle.cpp -- plain, slow CPU oracle (TEST INFRASTRUCTURE ONLY; see aht_oracle.h).
//
// Written to be read against the paper and the readings stated in aht_oracle.h, not to be fast:
// one env at a time, plain loops, fp64 for every policy, sampling and GAE quantity,
// fp32 exactly where the method's own rewards and returns are fp32.  Built with
// -ffp-contract=off so no multiply-add is fused on any host.
#include "aht_oracle.h"

#include <algorithm>
#include <cmath>
#include <cstring>
#include <limits>
#include <thread>
#include <vector>

// ======================================================================================
// Philox4x32-10, from Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy as
// 1, 2, 3" (SC'11): ten rounds of two 32x32->64 multiplies, with the key bumped by the
// Weyl constants between rounds.
// ======================================================================================
namespace {
const uint32_t kPhiloxM0 = 0xD2511F53u, kPhiloxM1 = 0xCD9E8D57u;
const uint32_t kWeyl0 = 0x9E3779B9u, kWeyl1 = 0xBB67AE85u;

// The draws of one (env, step, stream) tuple, taken in order.
struct DrawSeq {
  uint64_t seed;
  uint32_t env, step, stream, n = 0;
  DrawSeq(uint64_t s, uint32_t e, uint32_t t, uint32_t st) : seed(s), env(e), step(t), stream(st) {}
  uint32_t next() { return orc_draw(seed, env, step, stream, n++); }
};
}  // namespace

extern "C" void orc_philox4x32_10(uint32_t k0, uint32_t k1, const uint32_t ctr[4],
                                  uint32_t out[4]) {
  uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += kWeyl0;
      k1 += kWeyl1;
    }
    uint64_t p0 = (uint64_t)kPhiloxM0 * x0;
    uint64_t p1 = (uint64_t)kPhiloxM1 * x2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t y0 = hi1 ^ x1 ^ k0;
    uint32_t y1 = lo1;
    uint32_t y2 = hi0 ^ x3 ^ k1;
    uint32_t y3 = lo0;
    x0 = y0; x1 = y1; x2 = y2; x3 = y3;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

extern "C" uint32_t orc_draw(uint64_t seed, uint32_t env, uint32_t step, uint32_t stream,
                             uint32_t n) {
  uint32_t ctr[4] = {env, step, stream, n / 4u};
  uint32_t out[4];
  orc_philox4x32_10((uint32_t)(seed & 0xffffffffu), (uint32_t)(seed >> 32), ctr, out);
  return out[n % 4u];
}

extern "C" uint32_t orc_uniform_int(uint32_t x, uint32_t n) {
  return (uint32_t)(((uint64_t)x * (uint64_t)n) >> 32);
}

extern "C" double orc_u01(uint32_t x) { return (double)(x >> 8) * (1.0 / 16777216.0); }

// ======================================================================================
// Environment descriptions
// ======================================================================================
extern "C" int32_t orc_obs_dim(const orc_env_desc* d) {
  switch (d->kind) {
    case ORC_LBF: return d->width * d->height * 4;
    case ORC_OVERCOOKED: return 5 * 4 * 26;
    case ORC_HANABI: return 660;
    case ORC_MINI_HANABI: return 156;
  }
  return -1;
}

extern "C" int32_t orc_n_actions(const orc_env_desc* d) {
  switch (d->kind) {
    case ORC_LBF: return 6;
    case ORC_OVERCOOKED: return 6;
    case ORC_HANABI: return 20;
    case ORC_MINI_HANABI: return 10;
  }
  return -1;
}

extern "C" int32_t orc_check_desc(const orc_env_desc* d) {
  if (d->kind == ORC_LBF) {
    if (d->width < 3 || d->width > 12 || d->height < 3 || d->height > 12) return -1;
    if (d->n_food < 1 || d->n_food > ORC_LBF_MAX_FOOD) return -2;
    if (d->max_agent_level < 1 || d->max_agent_level > 9) return -3;
    if (d->episode_len < 1) return -4;
    return 0;
  }
  if (d->kind == ORC_OVERCOOKED) {
    if (d->width != 5 || d->height != 4) return -1;
    if (d->episode_len < 1 || d->cook_time < 0 || d->cook_time > 255) return -4;
    return 0;
  }
  if (d->kind == ORC_HANABI || d->kind == ORC_MINI_HANABI) {
    if (d->episode_len != 0) return -4;
    return 0;
  }
  return -5;
}

// ======================================================================================
// Level-Based Foraging.  Grid cell (x, y) has index y*W + x; N is y-1, S is y+1,
// W is x-1, E is x+1.  Actions: 0 noop, 1 N, 2 S, 3 W, 4 E, 5 load.
// ======================================================================================
namespace {
const int kLbfLoad = 5;
void lbf_delta(int a, int* dx, int* dy) {
  *dx = 0; *dy = 0;
  if (a == 1) *dy = -1;
  if (a == 2) *dy = 1;
  if (a == 3) *dx = -1;
  if (a == 4) *dx = 1;
}
}  // namespace

extern "C" void orc_lbf_reset(const orc_env_desc* d, uint64_t seed, uint32_t env,
                              uint32_t step, orc_lbf_state* s) {
  std::memset(s, 0, sizeof(*s));
  DrawSeq draws(seed, env, step, ORC_STREAM_RESET);
  // Levels first: two agents, then each food in index order.
  s->al[0] = 1 + (int)orc_uniform_int(draws.next(), (uint32_t)d->max_agent_level);
  s->al[1] = 1 + (int)orc_uniform_int(draws.next(), (uint32_t)d->max_agent_level);
  int level_sum = s->al[0] + s->al[1];
  s->F = 0;
  for (int k = 0; k < d->n_food; ++k) {
    s->fl[k] = 1 + (int)orc_uniform_int(draws.next(), (uint32_t)level_sum);
    s->F += s->fl[k];
  }
  // Positions: the first n_food + 2 steps of a Fisher-Yates shuffle of all cells.
  int cells = d->width * d->height;
  std::vector<int> perm(cells);
  for (int c = 0; c < cells; ++c) perm[c] = c;
  for (int i = 0; i < d->n_food + 2; ++i) {
    int j = i + (int)orc_uniform_int(draws.next(), (uint32_t)(cells - i));
    std::swap(perm[i], perm[j]);
  }
  for (int k = 0; k < d->n_food; ++k) {
    s->fx[k] = perm[k] % d->width;
    s->fy[k] = perm[k] / d->width;
    s->eaten[k] = 0;
  }
  for (int k = d->n_food; k < ORC_LBF_MAX_FOOD; ++k) s->eaten[k] = 1;  // absent foods
  for (int i = 0; i < 2; ++i) {
    s->ax[i] = perm[d->n_food + i] % d->width;
    s->ay[i] = perm[d->n_food + i] / d->width;
    s->ix[i] = s->ax[i];
    s->iy[i] = s->ay[i];
  }
  s->ep_t = 0;
  s->done = 0;
  s->ret = 0.0f;
}

extern "C" int32_t orc_lbf_step(const orc_env_desc* d, orc_lbf_state* s, int32_t a0,
                                int32_t a1, float r[2], float* team) {
  const int act[2] = {a0, a1};
  r[0] = 0.0f;
  r[1] = 0.0f;
  // Loading, on the positions before the step.
  int eaten_now[ORC_LBF_MAX_FOOD] = {0, 0, 0};
  for (int k = 0; k < d->n_food; ++k) {
    if (s->eaten[k]) continue;
    int loader_sum = 0;
    bool loader[2] = {false, false};
    for (int i = 0; i < 2; ++i) {
      int dist = std::abs(s->ax[i] - s->fx[k]) + std::abs(s->ay[i] - s->fy[k]);
      if (act[i] == kLbfLoad && dist == 1) {
        loader[i] = true;
        loader_sum += s->al[i];
      }
    }
    if (loader_sum > 0 && loader_sum >= s->fl[k]) {
      eaten_now[k] = 1;
      for (int i = 0; i < 2; ++i) {
        if (!loader[i]) continue;
        float num = (float)(s->fl[k] * s->al[i]);
        float den = (float)(loader_sum * s->F);
        r[i] = r[i] + num / den;
      }
    }
  }
  // Movement, on the state before the step.
  int tx[2], ty[2];
  for (int i = 0; i < 2; ++i) {
    int dx, dy;
    lbf_delta(act[i], &dx, &dy);
    tx[i] = s->ax[i] + dx;
    ty[i] = s->ay[i] + dy;
    bool valid = (dx != 0 || dy != 0);
    if (tx[i] < 0 || tx[i] >= d->width || ty[i] < 0 || ty[i] >= d->height) valid = false;
    for (int k = 0; k < d->n_food && valid; ++k)
      if (!s->eaten[k] && s->fx[k] == tx[i] && s->fy[k] == ty[i]) valid = false;
    for (int j = 0; j < 2 && valid; ++j)
      if (s->ax[j] == tx[i] && s->ay[j] == ty[i]) valid = false;
    if (!valid) {
      tx[i] = s->ax[i];
      ty[i] = s->ay[i];
    }
  }
  if (tx[0] == tx[1] && ty[0] == ty[1]) {
    for (int i = 0; i < 2; ++i) {
      tx[i] = s->ax[i];
      ty[i] = s->ay[i];
    }
  }
  for (int i = 0; i < 2; ++i) {
    s->ax[i] = tx[i];
    s->ay[i] = ty[i];
  }
  for (int k = 0; k < d->n_food; ++k)
    if (eaten_now[k]) s->eaten[k] = 1;
  s->ep_t += 1;
  bool all_eaten = true;
  for (int k = 0; k < d->n_food; ++k)
    if (!s->eaten[k]) all_eaten = false;
  s->done = (all_eaten || s->ep_t == d->episode_len) ? 1 : 0;
  *team = r[0] + r[1];
  s->ret = s->ret + *team;
  return s->done;
}

extern "C" int32_t orc_lbf_heuristic(const orc_env_desc* d, const orc_lbf_state* s, int32_t seat,
                                     int32_t k) {
  const int me = seat, other = 1 - seat;
  auto dist = [&](int x, int y, int f) { return std::abs(x - s->fx[f]) + std::abs(y - s->fy[f]); };
  auto free_cell = [&](int cx, int cy) {
    if (cx < 0 || cx >= d->width || cy < 0 || cy >= d->height) return false;
    for (int f = 0; f < d->n_food; ++f)
      if (!s->eaten[f] && s->fx[f] == cx && s->fy[f] == cy) return false;
    return !(s->ax[other] == cx && s->ay[other] == cy);
  };
  // one step from (x, y) toward (tx, ty): the axis with the larger distance first (ties:
  // x), the other axis if that cell is not free; noop if neither is
  auto step_toward = [&](int x, int y, int tx, int ty) {
    const int dx = tx - x, dy = ty - y;
    const int x_act = dx > 0 ? 4 : 3, y_act = dy > 0 ? 2 : 1;
    const int sx = dx > 0 ? 1 : -1, sy = dy > 0 ? 1 : -1;
    const bool x_first = std::abs(dx) >= std::abs(dy);
    for (int c = 0; c < 2; ++c) {
      const bool along_x = (c == 0) == x_first;
      if (along_x && dx != 0 && free_cell(x + sx, y)) return x_act;
      if (!along_x && dy != 0 && free_cell(x, y + sy)) return y_act;
    }
    return 0;
  };
  if (k == 11) {  // Entitled
    int f = 0;
    while (f < d->n_food && s->eaten[f]) ++f;
    if (f >= d->n_food) return 0;
    const int nx[4] = {s->fx[f] - 1, s->fx[f] + 1, s->fx[f], s->fx[f]};
    const int ny[4] = {s->fy[f], s->fy[f], s->fy[f] - 1, s->fy[f] + 1};
    int pair[2], n = 0;
    for (int q = 0; q < 4 && n < 2; ++q) {
      bool ok = nx[q] >= 0 && nx[q] < d->width && ny[q] >= 0 && ny[q] < d->height;
      for (int g = 0; ok && g < d->n_food; ++g)
        if (!s->eaten[g] && s->fx[g] == nx[q] && s->fy[g] == ny[q]) ok = false;
      if (ok) pair[n++] = q;
    }
    if (n < 2) return 0;
    int mine = -1;
    for (int q = 0; q < 2; ++q)
      if (s->ax[other] == nx[pair[q]] && s->ay[other] == ny[pair[q]]) mine = pair[1 - q];
    if (mine < 0) return 0;  // wait for the other agent to take one square
    if (s->ax[me] == nx[mine] && s->ay[me] == ny[mine]) return kLbfLoad;
    return step_toward(s->ax[me], s->ay[me], nx[mine], ny[mine]);
  }
  // the food to go for
  int target = -1;
  long best = 0;
  for (int f = 0; f < d->n_food; ++f) {
    if (s->eaten[f]) continue;
    long key = 0;
    switch (k) {
      case 0: key = dist(s->ax[me], s->ay[me], f); break;
      case 1: key = dist(s->ax[other], s->ay[other], f); break;
      case 2: key = dist(s->ax[me], s->ay[me], f) + dist(s->ax[other], s->ay[other], f); break;
      case 3: key = s->fl[f]; break;
      case 4: key = -s->fl[f]; break;
      case 5: key = s->fy[f] * d->width + s->fx[f]; break;
      case 6: key = -(s->fy[f] * d->width + s->fx[f]); break;
      case 7: key = s->fx[f] * d->height + s->fy[f]; break;
      case 8: key = -(s->fx[f] * d->height + s->fy[f]); break;
      case 9: key = dist(s->ix[me], s->iy[me], f); break;
      case 10: key = -dist(s->ix[me], s->iy[me], f); break;
      default: return 0;
    }
    if (target < 0 || key < best) {  // strict: the lower food index wins ties
      target = f;
      best = key;
    }
  }
  if (target < 0) return 0;
  const int x = s->ax[me], y = s->ay[me];
  if (dist(x, y, target) == 1) return kLbfLoad;
  return step_toward(x, y, s->fx[target], s->fy[target]);
}

extern "C" void orc_lbf_obs(const orc_env_desc* d, const orc_lbf_state* s, int32_t seat,
                            uint8_t* out) {
  const int other = 1 - seat;
  for (int y = 0; y < d->height; ++y) {
    for (int x = 0; x < d->width; ++x) {
      uint8_t* cell = out + (y * d->width + x) * 4;
      cell[0] = cell[1] = cell[2] = cell[3] = 0;
      int food = -1;
      for (int k = 0; k < d->n_food; ++k)
        if (!s->eaten[k] && s->fx[k] == x && s->fy[k] == y) food = k;
      if (s->ax[seat] == x && s->ay[seat] == y)
        cell[0] = (uint8_t)s->al[seat];
      else if (s->ax[other] == x && s->ay[other] == y)
        cell[1] = (uint8_t)s->al[other];
      else if (food >= 0)
        cell[2] = (uint8_t)s->fl[food];
      else
        cell[3] = 1;
    }
  }
}

// ======================================================================================
// Overcooked-style kitchen.  Fixed 5x4 layout (x right, y down):
//   y0: # O # P #
//   y1: # . . . #
//   y2: D . . . S
//   y3: # # O # #
// Actions: 0 noop, 1 N, 2 S, 3 E, 4 W, 5 interact.  Facing 0 N, 1 S, 2 E, 3 W.
// ======================================================================================
namespace {
const char* kKitchen[4] = {"#O#P#", "#...#", "D...S", "##O##"};
void oc_dir(int face, int* dx, int* dy) {
  *dx = 0; *dy = 0;
  if (face == 0) *dy = -1;
  if (face == 1) *dy = 1;
  if (face == 2) *dx = 1;
  if (face == 3) *dx = -1;
}
}  // namespace

extern "C" int32_t orc_oc_cell(int32_t x, int32_t y) {
  if (x < 0 || x >= 5 || y < 0 || y >= 4) return -1;
  switch (kKitchen[y][x]) {
    case '.': return ORC_OC_FLOOR;
    case '#': return ORC_OC_COUNTER;
    case 'O': return ORC_OC_ONION_D;
    case 'P': return ORC_OC_POT;
    case 'D': return ORC_OC_DISH_D;
    case 'S': return ORC_OC_SERVE;
  }
  return -1;
}

extern "C" void orc_oc_reset(const orc_env_desc* d, orc_oc_state* s) {
  (void)d;
  std::memset(s, 0, sizeof(*s));
  s->ax[0] = 1; s->ay[0] = 1;
  s->ax[1] = 3; s->ay[1] = 2;
  s->face[0] = s->face[1] = 0;
  s->held[0] = s->held[1] = ORC_OC_NONE;
  s->pot_n = 0;
  s->pot_timer = 0;
  s->ep_t = 0;
  s->done = 0;
  s->ret = 0.0f;
}

extern "C" int32_t orc_oc_step(const orc_env_desc* d, orc_oc_state* s, int32_t a0,
                               int32_t a1, float r[2], float* team) {
  const int act[2] = {a0, a1};
  const bool cooking_at_start = (s->pot_n == 3 && s->pot_timer > 0);
  // Movement: a move sets facing; the agent proposes the adjacent cell if it is floor.
  int px[2], py[2];
  for (int i = 0; i < 2; ++i) {
    px[i] = s->ax[i];
    py[i] = s->ay[i];
    if (act[i] >= 1 && act[i] <= 4) {
      s->face[i] = act[i] - 1;
      int dx, dy;
      oc_dir(s->face[i], &dx, &dy);
      if (orc_oc_cell(s->ax[i] + dx, s->ay[i] + dy) == ORC_OC_FLOOR) {
        px[i] = s->ax[i] + dx;
        py[i] = s->ay[i] + dy;
      }
    }
  }
  bool same = (px[0] == px[1] && py[0] == py[1]);
  bool swap = (px[0] == s->ax[1] && py[0] == s->ay[1] && px[1] == s->ax[0] && py[1] == s->ay[0]);
  if (!same && !swap) {
    for (int i = 0; i < 2; ++i) {
      s->ax[i] = px[i];
      s->ay[i] = py[i];
    }
  }
  // Interact on the faced cell, agent 0 first.
  float reward = 0.0f;
  for (int i = 0; i < 2; ++i) {
    if (act[i] != 5) continue;
    int dx, dy;
    oc_dir(s->face[i], &dx, &dy);
    int cx = s->ax[i] + dx, cy = s->ay[i] + dy;
    int cell = orc_oc_cell(cx, cy);
    int& held = s->held[i];
    switch (cell) {
      case ORC_OC_ONION_D:
        if (held == ORC_OC_NONE) held = ORC_OC_ONION;
        break;
      case ORC_OC_DISH_D:
        if (held == ORC_OC_NONE) held = ORC_OC_DISH;
        break;
      case ORC_OC_POT:
        if (held == ORC_OC_ONION && s->pot_n < 3) {
          s->pot_n += 1;
          held = ORC_OC_NONE;
          if (s->pot_n == 3) s->pot_timer = d->cook_time;
        } else if (held == ORC_OC_DISH && s->pot_n == 3 && s->pot_timer == 0) {
          held = ORC_OC_SOUP;
          s->pot_n = 0;
          s->pot_timer = 0;
        }
        break;
      case ORC_OC_SERVE:
        if (held == ORC_OC_SOUP) {
          held = ORC_OC_NONE;
          reward = reward + (float)d->soup_reward;
        }
        break;
      case ORC_OC_COUNTER: {
        int& item = s->counter_item[cy * 5 + cx];
        if (held != ORC_OC_NONE && item == ORC_OC_NONE) {
          item = held;
          held = ORC_OC_NONE;
        } else if (held == ORC_OC_NONE && item != ORC_OC_NONE) {
          held = item;
          item = ORC_OC_NONE;
        }
        break;
      }
      default:
        break;
    }
  }
  if (cooking_at_start && s->pot_timer > 0) s->pot_timer -= 1;
  s->ep_t += 1;
  s->done = (s->ep_t == d->episode_len) ? 1 : 0;
  r[0] = reward;
  r[1] = reward;
  *team = reward;
  s->ret = s->ret + reward;
  return s->done;
}

extern "C" void orc_oc_obs(const orc_env_desc* d, const orc_oc_state* s, int32_t seat,
                           uint8_t* out) {
  const int C = 26;
  std::memset(out, 0, 5 * 4 * C);
  const int other = 1 - seat;
  for (int y = 0; y < 4; ++y) {
    for (int x = 0; x < 5; ++x) {
      uint8_t* o = out + (y * 5 + x) * C;
      int cell = orc_oc_cell(x, y);
      if (cell == ORC_OC_COUNTER) {
        o[10] = 1;
        int item = s->counter_item[y * 5 + x];
        if (item != ORC_OC_NONE) o[14 + item] = 1;
      }
      if (cell == ORC_OC_POT) {
        o[11] = 1;
        if (s->pot_n >= 1) o[17 + s->pot_n] = 1;
        if (s->pot_n == 3 && s->pot_timer > 0) o[21] = 1;
        if (s->pot_n == 3 && s->pot_timer == 0) o[22] = 1;
      }
      if (cell == ORC_OC_ONION_D) o[12] = 1;
      if (cell == ORC_OC_DISH_D) o[13] = 1;
      if (cell == ORC_OC_SERVE) o[14] = 1;
      if (d->episode_len - s->ep_t <= 40) o[25] = 1;
    }
  }
  uint8_t* me = out + (s->ay[seat] * 5 + s->ax[seat]) * C;
  me[0] = 1;
  me[2 + s->face[seat]] = 1;
  if (s->held[seat] != ORC_OC_NONE) {
    me[23] = 1;
    me[14 + s->held[seat]] = 1;
  }
  uint8_t* you = out + (s->ay[other] * 5 + s->ax[other]) * C;
  you[1] = 1;
  you[6 + s->face[other]] = 1;
  if (s->held[other] != ORC_OC_NONE) {
    you[24] = 1;
    you[14 + s->held[other]] = 1;
  }
}

// ======================================================================================
// Hanabi, 2 players.  Card type = colour*5 + (rank-1).  Actions: 0-4 play slot,
// 5-9 discard slot, 10-14 hint colour, 15-19 hint rank (to the partner).
// ======================================================================================
namespace {
const int kRankOfCopy[10] = {1, 1, 1, 2, 2, 3, 3, 4, 4, 5};
const int kDiscardBase[5] = {0, 3, 5, 7, 9};  // thermometer offset per rank (copies 3,2,2,2,1)
uint32_t colour_mask(int c) { return 0x1Fu << (5 * c); }
uint32_t rank_mask(int r) {  // r in 1..5
  uint32_t m = 0;
  for (int c = 0; c < 5; ++c) m |= 1u << (5 * c + r - 1);
  return m;
}
const uint32_t kAllCards = (1u << 25) - 1;

void hb_remove_slot(orc_hanabi_state* s, int seat, int slot) {
  for (int k = slot; k < s->n_hand[seat] - 1; ++k) {
    s->hand[seat][k] = s->hand[seat][k + 1];
    s->know[seat][k] = s->know[seat][k + 1];
    s->hint_col[seat][k] = s->hint_col[seat][k + 1];
    s->hint_rank[seat][k] = s->hint_rank[seat][k + 1];
  }
  int last = s->n_hand[seat] - 1;
  s->hand[seat][last] = -1;
  s->know[seat][last] = 0;
  s->hint_col[seat][last] = 0;
  s->hint_rank[seat][last] = 0;
  s->n_hand[seat] -= 1;
}

void hb_draw(orc_hanabi_state* s, int seat) {
  if (s->ptr >= 50) return;
  int k = s->n_hand[seat];
  s->hand[seat][k] = s->deck[s->ptr];
  s->know[seat][k] = kAllCards;
  s->hint_col[seat][k] = 0;
  s->hint_rank[seat][k] = 0;
  s->n_hand[seat] += 1;
  s->ptr += 1;
  if (s->ptr == 50) s->fr = 2;
}
}  // namespace

extern "C" void orc_hanabi_reset(uint64_t seed, uint32_t env, uint32_t step,
                                 orc_hanabi_state* s) {
  std::memset(s, 0, sizeof(*s));
  for (int c = 0; c < 5; ++c)
    for (int i = 0; i < 10; ++i) s->deck[c * 10 + i] = c * 5 + (kRankOfCopy[i] - 1);
  DrawSeq draws(seed, env, step, ORC_STREAM_RESET);
  for (int i = 49; i >= 1; --i) {
    int j = (int)orc_uniform_int(draws.next(), (uint32_t)(i + 1));
    std::swap(s->deck[i], s->deck[j]);
  }
  for (int seat = 0; seat < 2; ++seat) {
    for (int k = 0; k < 5; ++k) {
      s->hand[seat][k] = s->deck[seat * 5 + k];
      s->know[seat][k] = kAllCards;
      s->hint_col[seat][k] = 0;
      s->hint_rank[seat][k] = 0;
    }
    s->n_hand[seat] = 5;
  }
  s->ptr = 10;
  s->info = 8;
  s->lives = 3;
  s->score = 0;
  s->fr = -1;
  s->turn = 0;
  s->la_valid = 0;
  s->done = 0;
  s->ret = 0.0f;
}

extern "C" void orc_hanabi_legal(const orc_hanabi_state* s, uint8_t legal[20]) {
  const int me = s->turn % 2, partner = 1 - me;
  for (int k = 0; k < 5; ++k) {
    legal[k] = (k < s->n_hand[me]) ? 1 : 0;
    legal[5 + k] = (k < s->n_hand[me] && s->info < 8) ? 1 : 0;
  }
  for (int v = 0; v < 5; ++v) {
    bool col = false, rank = false;
    for (int k = 0; k < s->n_hand[partner]; ++k) {
      int card = s->hand[partner][k];
      if (card / 5 == v) col = true;
      if (card % 5 == v) rank = true;
    }
    legal[10 + v] = (s->info > 0 && col) ? 1 : 0;
    legal[15 + v] = (s->info > 0 && rank) ? 1 : 0;
  }
}

extern "C" int32_t orc_hanabi_step(orc_hanabi_state* s, int32_t a, float* team) {
  uint8_t legal[20];
  orc_hanabi_legal(s, legal);
  if (a < 0 || a >= 20 || !legal[a]) return -1;
  const int me = s->turn % 2, partner = 1 - me;
  const int fr_start = s->fr;
  const int score_before = s->score;
  float reward = 0.0f;
  s->la_valid = 1;
  s->la_actor = me;
  s->la_colour = -1;
  s->la_rank = 0;
  s->la_slot = -1;
  s->la_card = -1;
  s->la_hinted = 0;
  s->la_success = 0;
  s->la_bomb = 0;
  if (a < 10) {
    const int slot = a % 5;
    const int card = s->hand[me][slot];
    const int c = card / 5, rank = card % 5 + 1;
    s->la_type = (a < 5) ? 0 : 1;
    s->la_colour = c;
    s->la_rank = rank;
    s->la_slot = slot;
    s->la_card = card;
    hb_remove_slot(s, me, slot);
    if (a < 5) {
      if (s->fw[c] == rank - 1) {
        s->fw[c] = rank;
        s->score += 1;
        reward = 1.0f;
        if (rank == 5 && s->info < 8) s->info += 1;
        s->la_success = 1;
      } else {
        s->lives -= 1;
        s->disc[card] += 1;
        s->la_bomb = 1;
      }
    } else {
      s->disc[card] += 1;
      s->info += 1;
    }
    hb_draw(s, me);
  } else {
    const bool by_colour = (a < 15);
    const int v = (a - 10) % 5;
    const uint32_t m = by_colour ? colour_mask(v) : rank_mask(v + 1);
    s->info -= 1;
    s->la_type = by_colour ? 2 : 3;
    if (by_colour) s->la_colour = v; else s->la_rank = v + 1;
    for (int k = 0; k < s->n_hand[partner]; ++k) {
      const int card = s->hand[partner][k];
      const bool match = by_colour ? (card / 5 == v) : (card % 5 == v);
      if (match) {
        s->know[partner][k] &= m;
        if (by_colour) s->hint_col[partner][k] |= 1u << v;
        else s->hint_rank[partner][k] |= 1u << v;
        s->la_hinted |= 1 << k;
      } else {
        s->know[partner][k] &= ~m;
      }
    }
  }
  s->turn += 1;
  int done = 0;
  if (s->lives == 0) {
    done = 1;
    reward = -(float)score_before;
  } else if (s->score == 25) {
    done = 1;
  } else if (fr_start >= 1) {
    s->fr = fr_start - 1;
    if (s->fr == 0) done = 1;
  }
  s->done = done;
  *team = reward;
  s->ret = s->ret + reward;
  return done;
}

extern "C" void orc_hanabi_obs(const orc_hanabi_state* s, int32_t seat, uint8_t* out) {
  std::memset(out, 0, 660);
  const int me = seat, partner = 1 - seat;
  int o = 0;
  for (int k = 0; k < 5; ++k)  // partner hand
    if (k < s->n_hand[partner]) out[o + k * 25 + s->hand[partner][k]] = 1;
  o += 125;
  for (int k = 0; k < 5; ++k)  // own knowledge
    for (int b = 0; b < 25; ++b)
      if (k < s->n_hand[me] && ((s->know[me][k] >> b) & 1u)) out[o + k * 25 + b] = 1;
  o += 125;
  for (int k = 0; k < 5; ++k)  // partner knowledge
    for (int b = 0; b < 25; ++b)
      if (k < s->n_hand[partner] && ((s->know[partner][k] >> b) & 1u)) out[o + k * 25 + b] = 1;
  o += 125;
  for (int c = 0; c < 5; ++c)  // fireworks
    if (s->fw[c] >= 1) out[o + c * 5 + s->fw[c] - 1] = 1;
  o += 25;
  for (int i = 0; i < s->info; ++i) out[o + i] = 1;
  o += 8;
  for (int i = 0; i < s->lives; ++i) out[o + i] = 1;
  o += 3;
  for (int i = 0; i < 50 - s->ptr; ++i) out[o + i] = 1;
  o += 40;
  for (int c = 0; c < 5; ++c)  // discard thermometers
    for (int r = 1; r <= 5; ++r)
      for (int i = 0; i < s->disc[c * 5 + r - 1]; ++i) out[o + c * 10 + kDiscardBase[r - 1] + i] = 1;
  o += 50;
  if (s->la_valid) {  // last action, 53 bits
    out[o + (s->la_actor == me ? 0 : 1)] = 1;
    out[o + 2 + s->la_type] = 1;
    if (s->la_colour >= 0) out[o + 6 + s->la_colour] = 1;
    if (s->la_rank >= 1) out[o + 11 + s->la_rank - 1] = 1;
    if (s->la_slot >= 0) out[o + 16 + s->la_slot] = 1;
    if (s->la_card >= 0) out[o + 21 + s->la_card] = 1;
    for (int k = 0; k < 5; ++k)
      if ((s->la_hinted >> k) & 1) out[o + 46 + k] = 1;
    if (s->la_success) out[o + 51] = 1;
    if (s->la_bomb) out[o + 52] = 1;
  }
  o += 53;
  for (int pass = 0; pass < 2; ++pass) {  // explicit hints: own, then partner
    const int who = pass == 0 ? me : partner;
    for (int k = 0; k < 5; ++k)
      for (int b = 0; b < 5; ++b) {
        if ((s->hint_col[who][k] >> b) & 1u) out[o + k * 10 + b] = 1;
        if ((s->hint_rank[who][k] >> b) & 1u) out[o + k * 10 + 5 + b] = 1;
      }
    o += 50;
  }
  for (int k = 0; k < 5; ++k)
    if (k < s->n_hand[me]) out[o + k] = 1;
  o += 5;
  if (s->fr >= 0) out[o] = 1;
  o += 1;
}

// ======================================================================================
// Mini Hanabi, 2 players: 3 colours x ranks (1,1,1,2,2,3), 2-card hands, 3 info and 1
// life tokens.  Card type = colour*3 + (rank-1).  Actions: 0-1 play slot, 2-3 discard
// slot, 4-6 hint colour, 7-9 hint rank (to the partner).
// ======================================================================================
namespace {
const int kMhRankOfCopy[6] = {1, 1, 1, 2, 2, 3};
const int kMhDiscardBase[3] = {0, 3, 5};  // thermometer offset per rank (copies 3, 2, 1)
const uint32_t kMhAllCards = (1u << 9) - 1;
uint32_t mh_colour_mask(int c) { return 0x7u << (3 * c); }
uint32_t mh_rank_mask(int r) {  // r in 1..3
  uint32_t m = 0;
  for (int c = 0; c < 3; ++c) m |= 1u << (3 * c + r - 1);
  return m;
}

void mh_remove_slot(orc_mhanabi_state* s, int seat, int slot) {
  for (int k = slot; k < s->n_hand[seat] - 1; ++k) {
    s->hand[seat][k] = s->hand[seat][k + 1];
    s->know[seat][k] = s->know[seat][k + 1];
    s->hint_col[seat][k] = s->hint_col[seat][k + 1];
    s->hint_rank[seat][k] = s->hint_rank[seat][k + 1];
  }
  const int last = s->n_hand[seat] - 1;
  s->hand[seat][last] = -1;
  s->know[seat][last] = 0;
  s->hint_col[seat][last] = 0;
  s->hint_rank[seat][last] = 0;
  s->n_hand[seat] -= 1;
}

void mh_draw(orc_mhanabi_state* s, int seat) {
  if (s->ptr >= 18) return;
  const int k = s->n_hand[seat];
  s->hand[seat][k] = s->deck[s->ptr];
  s->know[seat][k] = kMhAllCards;
  s->hint_col[seat][k] = 0;
  s->hint_rank[seat][k] = 0;
  s->n_hand[seat] += 1;
  s->ptr += 1;
  if (s->ptr == 18) s->fr = 2;
}
}  // namespace

extern "C" void orc_mhanabi_reset(uint64_t seed, uint32_t env, uint32_t step,
                                  orc_mhanabi_state* s) {
  std::memset(s, 0, sizeof(*s));
  for (int c = 0; c < 3; ++c)
    for (int i = 0; i < 6; ++i) s->deck[c * 6 + i] = c * 3 + (kMhRankOfCopy[i] - 1);
  DrawSeq draws(seed, env, step, ORC_STREAM_RESET);
  for (int i = 17; i >= 1; --i) {
    const int j = (int)orc_uniform_int(draws.next(), (uint32_t)(i + 1));
    std::swap(s->deck[i], s->deck[j]);
  }
  for (int seat = 0; seat < 2; ++seat) {
    for (int k = 0; k < 2; ++k) {
      s->hand[seat][k] = s->deck[seat * 2 + k];
      s->know[seat][k] = kMhAllCards;
    }
    s->n_hand[seat] = 2;
  }
  s->ptr = 4;
  s->info = 3;
  s->lives = 1;
  s->fr = -1;
}

extern "C" void orc_mhanabi_legal(const orc_mhanabi_state* s, uint8_t legal[10]) {
  const int me = s->turn % 2, partner = 1 - me;
  for (int k = 0; k < 2; ++k) {
    legal[k] = (k < s->n_hand[me]) ? 1 : 0;
    legal[2 + k] = (k < s->n_hand[me] && s->info < 3) ? 1 : 0;
  }
  for (int v = 0; v < 3; ++v) {
    bool col = false, rank = false;
    for (int k = 0; k < s->n_hand[partner]; ++k) {
      const int card = s->hand[partner][k];
      if (card / 3 == v) col = true;
      if (card % 3 == v) rank = true;
    }
    legal[4 + v] = (s->info > 0 && col) ? 1 : 0;
    legal[7 + v] = (s->info > 0 && rank) ? 1 : 0;
  }
}

extern "C" int32_t orc_mhanabi_step(orc_mhanabi_state* s, int32_t a, float* team) {
  uint8_t legal[10];
  orc_mhanabi_legal(s, legal);
  if (a < 0 || a >= 10 || !legal[a]) return -1;
  const int me = s->turn % 2, partner = 1 - me;
  const int fr_start = s->fr;
  const int score_before = s->score;
  float reward = 0.0f;
  s->la_valid = 1;
  s->la_actor = me;
  s->la_colour = -1;
  s->la_rank = 0;
  s->la_slot = -1;
  s->la_card = -1;
  s->la_hinted = 0;
  s->la_success = 0;
  s->la_bomb = 0;
  if (a < 4) {
    const int slot = a % 2;
    const int card = s->hand[me][slot];
    const int c = card / 3, rank = card % 3 + 1;
    s->la_type = (a < 2) ? 0 : 1;
    s->la_colour = c;
    s->la_rank = rank;
    s->la_slot = slot;
    s->la_card = card;
    mh_remove_slot(s, me, slot);
    if (a < 2) {
      if (s->fw[c] == rank - 1) {
        s->fw[c] = rank;
        s->score += 1;
        reward = 1.0f;
        if (rank == 3 && s->info < 3) s->info += 1;
        s->la_success = 1;
      } else {
        s->lives -= 1;
        s->disc[card] += 1;
        s->la_bomb = 1;
      }
    } else {
      s->disc[card] += 1;
      s->info += 1;
    }
    mh_draw(s, me);
  } else {
    const bool by_colour = (a < 7);
    const int v = (a - 4) % 3;
    const uint32_t m = by_colour ? mh_colour_mask(v) : mh_rank_mask(v + 1);
    s->info -= 1;
    s->la_type = by_colour ? 2 : 3;
    if (by_colour) s->la_colour = v; else s->la_rank = v + 1;
    for (int k = 0; k < s->n_hand[partner]; ++k) {
      const int card = s->hand[partner][k];
      const bool match = by_colour ? (card / 3 == v) : (card % 3 == v);
      if (match) {
        s->know[partner][k] &= m;
        if (by_colour) s->hint_col[partner][k] |= 1u << v;
        else s->hint_rank[partner][k] |= 1u << v;
        s->la_hinted |= 1 << k;
      } else {
        s->know[partner][k] &= ~m;
      }
    }
  }
  s->turn += 1;
  int done = 0;
  if (s->lives == 0) {
    done = 1;
    reward = -(float)score_before;
  } else if (s->score == 9) {
    done = 1;
  } else if (fr_start >= 1) {
    s->fr = fr_start - 1;
    if (s->fr == 0) done = 1;
  }
  s->done = done;
  *team = reward;
  s->ret = s->ret + reward;
  return done;
}

// 153 bits: partner hand 18, own knowledge 18, partner knowledge 18, fireworks 9, info 3,
// lives 1, deck 14, discards 18, last action 27, explicit hints 12 + 12, slots 2, final 1;
// then 3 zero features (156: observation rows stay 4-byte multiples).
extern "C" void orc_mhanabi_obs(const orc_mhanabi_state* s, int32_t seat, uint8_t* out) {
  std::memset(out, 0, 156);
  const int me = seat, partner = 1 - seat;
  int o = 0;
  for (int k = 0; k < 2; ++k)
    if (k < s->n_hand[partner]) out[o + k * 9 + s->hand[partner][k]] = 1;
  o += 18;
  for (int k = 0; k < 2; ++k)
    for (int b = 0; b < 9; ++b)
      if (k < s->n_hand[me] && ((s->know[me][k] >> b) & 1u)) out[o + k * 9 + b] = 1;
  o += 18;
  for (int k = 0; k < 2; ++k)
    for (int b = 0; b < 9; ++b)
      if (k < s->n_hand[partner] && ((s->know[partner][k] >> b) & 1u)) out[o + k * 9 + b] = 1;
  o += 18;
  for (int c = 0; c < 3; ++c)
    if (s->fw[c] >= 1) out[o + c * 3 + s->fw[c] - 1] = 1;
  o += 9;
  for (int i = 0; i < s->info; ++i) out[o + i] = 1;
  o += 3;
  for (int i = 0; i < s->lives; ++i) out[o + i] = 1;
  o += 1;
  for (int i = 0; i < 18 - s->ptr; ++i) out[o + i] = 1;
  o += 14;
  for (int c = 0; c < 3; ++c)
    for (int r = 1; r <= 3; ++r)
      for (int i = 0; i < s->disc[c * 3 + r - 1]; ++i) out[o + c * 6 + kMhDiscardBase[r - 1] + i] = 1;
  o += 18;
  if (s->la_valid) {  // last action, 27 bits
    out[o + (s->la_actor == me ? 0 : 1)] = 1;
    out[o + 2 + s->la_type] = 1;
    if (s->la_colour >= 0) out[o + 6 + s->la_colour] = 1;
    if (s->la_rank >= 1) out[o + 9 + s->la_rank - 1] = 1;
    if (s->la_slot >= 0) out[o + 12 + s->la_slot] = 1;
    if (s->la_card >= 0) out[o + 14 + s->la_card] = 1;
    for (int k = 0; k < 2; ++k)
      if ((s->la_hinted >> k) & 1) out[o + 23 + k] = 1;
    if (s->la_success) out[o + 25] = 1;
    if (s->la_bomb) out[o + 26] = 1;
  }
  o += 27;
  for (int pass = 0; pass < 2; ++pass) {  // explicit hints: own, then partner
    const int who = pass == 0 ? me : partner;
    for (int k = 0; k < 2; ++k)
      for (int b = 0; b < 3; ++b) {
        if ((s->hint_col[who][k] >> b) & 1u) out[o + k * 6 + b] = 1;
        if ((s->hint_rank[who][k] >> b) & 1u) out[o + k * 6 + 3 + b] = 1;
      }
    o += 12;
  }
  for (int k = 0; k < 2; ++k)
    if (k < s->n_hand[me]) out[o + k] = 1;
  o += 2;
  if (s->fr >= 0) out[o] = 1;
  o += 1;
}

// ======================================================================================
// Generic env dispatch over orc_state blobs.
// ======================================================================================
namespace {
static_assert(sizeof(orc_lbf_state) <= ORC_STATE_BYTES, "state blob too small");
static_assert(sizeof(orc_oc_state) <= ORC_STATE_BYTES, "state blob too small");
static_assert(sizeof(orc_hanabi_state) <= ORC_STATE_BYTES, "state blob too small");
static_assert(sizeof(orc_mhanabi_state) <= ORC_STATE_BYTES, "state blob too small");

bool turn_based(const orc_env_desc* d) { return d->kind == ORC_HANABI || d->kind == ORC_MINI_HANABI; }

void env_reset(const orc_env_desc* d, uint64_t seed, uint32_t env, uint32_t step, orc_state* st) {
  std::memset(st, 0, sizeof(*st));
  if (d->kind == ORC_LBF) orc_lbf_reset(d, seed, env, step, (orc_lbf_state*)st);
  if (d->kind == ORC_OVERCOOKED) orc_oc_reset(d, (orc_oc_state*)st);
  if (d->kind == ORC_HANABI) orc_hanabi_reset(seed, env, step, (orc_hanabi_state*)st);
  if (d->kind == ORC_MINI_HANABI) orc_mhanabi_reset(seed, env, step, (orc_mhanabi_state*)st);
}

void env_obs(const orc_env_desc* d, const orc_state* st, int seat, uint8_t* out) {
  if (d->kind == ORC_LBF) orc_lbf_obs(d, (const orc_lbf_state*)st, seat, out);
  if (d->kind == ORC_OVERCOOKED) orc_oc_obs(d, (const orc_oc_state*)st, seat, out);
  if (d->kind == ORC_HANABI) orc_hanabi_obs((const orc_hanabi_state*)st, seat, out);
  if (d->kind == ORC_MINI_HANABI) orc_mhanabi_obs((const orc_mhanabi_state*)st, seat, out);
}

// Returns done, or -1 for an illegal action.
int env_step(const orc_env_desc* d, orc_state* st, int a0, int a1, float r[2], float* team) {
  if (d->kind == ORC_LBF) return orc_lbf_step(d, (orc_lbf_state*)st, a0, a1, r, team);
  if (d->kind == ORC_OVERCOOKED) return orc_oc_step(d, (orc_oc_state*)st, a0, a1, r, team);
  if (d->kind == ORC_MINI_HANABI) {
    orc_mhanabi_state* m = (orc_mhanabi_state*)st;
    const int done = orc_mhanabi_step(m, (m->turn % 2 == 0) ? a0 : a1, team);
    r[0] = r[1] = *team;
    if (done == 0 && m->turn >= 100) return -2;
    return done;
  }
  orc_hanabi_state* h = (orc_hanabi_state*)st;
  int a = (h->turn % 2 == 0) ? a0 : a1;
  int done = orc_hanabi_step(h, a, team);
  r[0] = r[1] = *team;
  if (done == 0 && h->turn >= 100) return -2;  // length bound (<= 97 turns) violated
  return done;
}

int acting_seat(const orc_env_desc* d, const orc_state* st) {
  if (!turn_based(d)) return -1;
  if (d->kind == ORC_MINI_HANABI) return ((const orc_mhanabi_state*)st)->turn % 2;
  return ((const orc_hanabi_state*)st)->turn % 2;
}

void env_legal(const orc_env_desc* d, const orc_state* st, uint8_t* legal) {
  if (d->kind == ORC_HANABI) {
    orc_hanabi_legal((const orc_hanabi_state*)st, legal);
    return;
  }
  if (d->kind == ORC_MINI_HANABI) {
    orc_mhanabi_legal((const orc_mhanabi_state*)st, legal);
    return;
  }
  for (int k = 0; k < orc_n_actions(d); ++k) legal[k] = 1;
}

template <class F>
void parallel_for(int64_t n, int32_t n_threads, F f) {
  if (n_threads <= 1 || n < 2) {
    for (int64_t i = 0; i < n; ++i) f(i);
    return;
  }
  std::vector<std::thread> pool;
  int64_t chunk = (n + n_threads - 1) / n_threads;
  for (int32_t t = 0; t < n_threads; ++t) {
    int64_t lo = t * chunk, hi = std::min<int64_t>(n, lo + chunk);
    if (lo >= hi) break;
    pool.emplace_back([=, &f]() {
      for (int64_t i = lo; i < hi; ++i) f(i);
    });
  }
  for (auto& th : pool) th.join();
}
}  // namespace

extern "C" int32_t orc_reset_all(const orc_env_desc* d, uint64_t seed, int64_t n_envs,
                                 int64_t step, orc_state* states) {
  if (orc_check_desc(d) != 0) return -1;
  for (int64_t e = 0; e < n_envs; ++e) env_reset(d, seed, (uint32_t)e, (uint32_t)step, &states[e]);
  return 0;
}

extern "C" int32_t orc_reset_envs(const orc_env_desc* d, uint64_t seed, const int64_t* ids,
                                  int64_t n, int64_t step, orc_state* states) {
  if (orc_check_desc(d) != 0) return -1;
  for (int64_t i = 0; i < n; ++i) env_reset(d, seed, (uint32_t)ids[i], (uint32_t)step, &states[i]);
  return 0;
}

extern "C" int32_t orc_step_forced(const orc_env_desc* d, uint64_t seed, int64_t n_envs,
                                   int64_t step, orc_state* states, const uint8_t* actions,
                                   float* rewards2, float* team, uint8_t* dones, uint8_t* obs2) {
  if (orc_check_desc(d) != 0) return -1;
  const int od = orc_obs_dim(d);
  int status = 0;
  for (int64_t e = 0; e < n_envs; ++e) {
    float r[2], tr;
    int done = env_step(d, &states[e], actions[e * 2], actions[e * 2 + 1], r, &tr);
    if (done < 0) {
      status = -2;
      r[0] = r[1] = tr = 0.0f;
      done = 0;
    }
    if (done) env_reset(d, seed, (uint32_t)e, (uint32_t)(step + 1), &states[e]);
    if (rewards2) { rewards2[e * 2] = r[0]; rewards2[e * 2 + 1] = r[1]; }
    if (team) team[e] = tr;
    if (dones) dones[e] = (uint8_t)done;
    if (obs2) {
      env_obs(d, &states[e], 0, obs2 + (e * 2 + 0) * od);
      env_obs(d, &states[e], 1, obs2 + (e * 2 + 1) * od);
    }
  }
  return status;
}

// ======================================================================================
// Policy MLP (Sec. 3 decentralised policy; tanh hidden layers), fp64.
// ======================================================================================
extern "C" void orc_mlp_forward(const orc_mlp* p, const double* x, double* z) {
  std::vector<double> h0(p->h0), h1(p->h1);
  for (int j = 0; j < p->h0; ++j) {
    double acc = p->b1[j];
    for (int k = 0; k < p->obs_dim; ++k) acc += p->W1[(int64_t)j * p->obs_dim + k] * x[k];
    h0[j] = std::tanh(acc);
  }
  for (int j = 0; j < p->h1; ++j) {
    double acc = p->b2[j];
    for (int k = 0; k < p->h0; ++k) acc += p->W2[(int64_t)j * p->h0 + k] * h0[k];
    h1[j] = std::tanh(acc);
  }
  for (int j = 0; j < p->n_out; ++j) {
    double acc = p->b3[j];
    for (int k = 0; k < p->h1; ++k) acc += p->W3[(int64_t)j * p->h1 + k] * h1[k];
    z[j] = acc;
  }
}

extern "C" void orc_sample(const double* z, const uint8_t* legal, int32_t K, double u,
                           int32_t* a, double* logp, double* margin) {
  double m = -INFINITY;
  for (int k = 0; k < K; ++k)
    if (legal[k]) m = std::max(m, z[k]);
  std::vector<double> S(K);
  double run = 0.0;
  for (int k = 0; k < K; ++k) {
    if (legal[k]) run += std::exp(z[k] - m);
    S[k] = run;
  }
  const double Z = S[K - 1];
  int chosen = -1;
  for (int k = 0; k < K; ++k) {
    if (u * Z < S[k]) {
      chosen = k;
      break;
    }
  }
  if (chosen < 0)
    for (int k = K - 1; k >= 0; --k)
      if (legal[k]) { chosen = k; break; }
  double mg = 2.0;
  for (int k = 0; k < K; ++k) mg = std::min(mg, std::fabs(u - S[k] / Z));
  *a = chosen;
  *logp = z[chosen] - m - std::log(Z);
  *margin = mg;
}

extern "C" double orc_logp(const double* z, const uint8_t* legal, int32_t K, int32_t a) {
  double m = -INFINITY;
  for (int k = 0; k < K; ++k)
    if (legal[k]) m = std::max(m, z[k]);
  double Z = 0.0;
  for (int k = 0; k < K; ++k)
    if (legal[k]) Z += std::exp(z[k] - m);
  return z[a] - m - std::log(Z);
}

extern "C" void orc_policy_outputs(const orc_mlp* p, const uint8_t* obs, int64_t n,
                                   double* out) {
  std::vector<double> x(p->obs_dim);
  for (int64_t i = 0; i < n; ++i) {
    for (int k = 0; k < p->obs_dim; ++k) x[k] = (double)obs[i * p->obs_dim + k];
    orc_mlp_forward(p, x.data(), out + i * p->n_out);
  }
}

// ======================================================================================
// GAE (PPO, App. C), fp64.
// ======================================================================================
extern "C" void orc_gae(const float* r, const float* v, const uint8_t* d, const float* v_last,
                        int64_t n_envs, int32_t T, double gamma, double lambda, double* adv,
                        double* targets) {
  for (int64_t e = 0; e < n_envs; ++e) {
    double next_v = (double)v_last[e];
    double next_a = 0.0;
    for (int t = T - 1; t >= 0; --t) {
      const int64_t i = (int64_t)t * n_envs + e;
      const double nonterminal = d[i] ? 0.0 : 1.0;
      const double delta = (double)r[i] + gamma * nonterminal * next_v - (double)v[i];
      const double a = delta + gamma * lambda * nonterminal * next_a;
      adv[i] = a;
      if (targets) targets[i] = a + (double)v[i];
      next_a = a;
      next_v = (double)v[i];
    }
  }
}

// ======================================================================================
// Cross-play matrix consumers (App. B "Upper bound estimation"; Sec. 3 J_AHT; App. A
// ROTATE regret and BRDiv objective), fp64.
// ======================================================================================
extern "C" void orc_xp_stats(const float* xp, int32_t n_ego, int32_t n_tm, double* upper,
                             double* norm, double* regret, double* j_aht, double* j_norm,
                             double* max_regret, int32_t* worst, double* brdiv) {
  // the bound of teammate m rises to any XP score of its column above the recorded value
  for (int m = 0; m < n_tm; ++m)
    for (int e = 0; e < n_ego; ++e)
      if ((double)xp[(int64_t)e * n_tm + m] > upper[m]) upper[m] = (double)xp[(int64_t)e * n_tm + m];
  std::vector<double> off_row(n_ego, 0.0);
  for (int e = 0; e < n_ego; ++e) {
    double sum = 0.0, sum_norm = 0.0, best = 0.0;
    int arg = 0;
    for (int m = 0; m < n_tm; ++m) {
      const double x = (double)xp[(int64_t)e * n_tm + m];
      const double u = upper[m];
      const double nr = u > 0.0 ? x / u : std::numeric_limits<double>::quiet_NaN();
      const double rg = u - x;
      if (norm) norm[(int64_t)e * n_tm + m] = nr;
      if (regret) regret[(int64_t)e * n_tm + m] = rg;
      sum += x;
      sum_norm += nr;
      if (m == 0 || rg > best) {
        best = rg;
        arg = m;
      }
      if (m != e) off_row[e] += x;
    }
    if (j_aht) j_aht[e] = sum / n_tm;
    if (j_norm) j_norm[e] = sum_norm / n_tm;
    if (max_regret) max_regret[e] = best;
    if (worst) worst[e] = arg;
  }
  if (brdiv && n_ego == n_tm) {
    const int n = n_ego;
    double diag = 0.0, off = 0.0;
    for (int i = 0; i < n; ++i) diag += (double)xp[(int64_t)i * n + i];
    for (int i = 0; i < n; ++i) off += off_row[i];
    *brdiv = diag / n - (n > 1 ? off / ((double)n * (n - 1)) : 0.0);
  }
}

// ======================================================================================
// Rollout drivers.
// ======================================================================================
namespace {
std::vector<double> obs_to_double(const uint8_t* o, int n) {
  std::vector<double> x(n);
  for (int k = 0; k < n; ++k) x[k] = (double)o[k];
  return x;
}
}  // namespace

extern "C" int32_t orc_rollout(const orc_env_desc* d, const orc_mlp* pols, int32_t n_pols,
                               orc_rollout_io* io) {
  if (orc_check_desc(d) != 0) return -1;
  if (turn_based(d)) return -3;  // PPO collection is for simultaneous-move games
  if (io->ego_id < 0 || io->ego_id >= n_pols || io->pool_size < 1) return -4;
  if (io->resample && !io->ep_step) return -4;
  const int min_id = d->kind == ORC_LBF ? -ORC_LBF_N_HEURISTICS : 0;  // heuristic teammates
  for (int k = 0; k < io->pool_size; ++k)
    if (io->pool[k] < min_id || io->pool[k] >= n_pols) return -4;
  const int od = orc_obs_dim(d), K = orc_n_actions(d);
  const int64_t N = io->n_envs;
  const int T = io->T;
  const orc_mlp* ego = &pols[io->ego_id];
  const bool has_value = ego->n_out > K;
  std::vector<int> status(N, 0);
  parallel_for(N, io->n_threads, [&](int64_t e) {
    const uint32_t env = (uint32_t)(io->env_ids ? io->env_ids[e] : e);
    // Teammate (Sec. 3): per call, one uniform pool draw per env at the call's first
    // step (counter (env, step0, stream 3)), kept for the whole call; per episode, the
    // draw of the step the current episode began (counter (env, s, stream 5)).
    auto episode_teammate = [&](uint32_t s) {
      const uint32_t x = orc_draw(io->seed, env, s, ORC_STREAM_EPISODE_TEAMMATE, 0);
      return io->pool[orc_uniform_int(x, (uint32_t)io->pool_size)];
    };
    const uint32_t x = orc_draw(io->seed, env, (uint32_t)io->step0, ORC_STREAM_TEAMMATE, 0);
    int tm_id = io->resample ? episode_teammate(io->ep_step[e])
                             : io->pool[orc_uniform_int(x, (uint32_t)io->pool_size)];
    if (io->teammate) io->teammate[e] = tm_id;
    const orc_mlp* tm = tm_id >= 0 ? &pols[tm_id] : nullptr;  // null: a heuristic teammate
    orc_state* st = &io->states[e];
    std::vector<uint8_t> o0(od), o1(od), legal(K, 1);
    int max_out = 1;
    for (int k = 0; k < io->pool_size; ++k)
      if (io->pool[k] >= 0) max_out = std::max(max_out, pols[io->pool[k]].n_out);
    std::vector<double> z0(ego->n_out), z1(max_out);
    for (int t = 0; t < T; ++t) {
      const uint32_t gt = (uint32_t)(io->step0 + t);
      const int64_t i = (int64_t)t * N + e;
      if (io->teammates_t) io->teammates_t[i] = tm_id;
      env_obs(d, st, 0, o0.data());
      env_obs(d, st, 1, o1.data());
      if (io->obs) std::memcpy(io->obs + i * od, o0.data(), od);
      if (io->obs_tm) std::memcpy(io->obs_tm + i * od, o1.data(), od);
      orc_mlp_forward(ego, obs_to_double(o0.data(), od).data(), z0.data());
      int own[2];
      double lp[2], mg[2];
      orc_sample(z0.data(), legal.data(), K, orc_u01(orc_draw(io->seed, env, gt, ORC_STREAM_ACT0, 0)),
                 &own[0], &lp[0], &mg[0]);
      if (tm) {
        orc_mlp_forward(tm, obs_to_double(o1.data(), od).data(), z1.data());
        orc_sample(z1.data(), legal.data(), K, orc_u01(orc_draw(io->seed, env, gt, ORC_STREAM_ACT1, 0)),
                   &own[1], &lp[1], &mg[1]);
      } else {
        own[1] = orc_lbf_heuristic(d, (const orc_lbf_state*)st, 1, -1 - tm_id);
        lp[1] = 0.0;
        mg[1] = 2.0;  // no draw: never flagged
      }
      int act[2] = {own[0], own[1]};
      if (io->forced) {
        act[0] = io->forced[i * 2];
        act[1] = io->forced[i * 2 + 1];
      }
      if (io->actions) { io->actions[i * 2] = (uint8_t)act[0]; io->actions[i * 2 + 1] = (uint8_t)act[1]; }
      if (io->own_actions) { io->own_actions[i * 2] = (uint8_t)own[0]; io->own_actions[i * 2 + 1] = (uint8_t)own[1]; }
      if (io->margin) { io->margin[i * 2] = mg[0]; io->margin[i * 2 + 1] = mg[1]; }
      if (io->logits) std::memcpy(io->logits + i * ego->n_out, z0.data(), sizeof(double) * ego->n_out);
      if (io->logp) io->logp[i] = orc_logp(z0.data(), legal.data(), K, act[0]);
      if (io->values) io->values[i] = has_value ? z0[K] : 0.0;
      if (io->logp_tm) io->logp_tm[i] = tm ? orc_logp(z1.data(), legal.data(), K, act[1]) : 0.0;
      if (io->values_tm) io->values_tm[i] = tm && tm->n_out > K ? z1[K] : 0.0;
      float r[2], team;
      int done = env_step(d, st, act[0], act[1], r, &team);
      if (done < 0) { status[e] = -2; done = 0; team = 0.0f; }
      if (io->rewards) io->rewards[i] = team;
      if (io->dones) io->dones[i] = (uint8_t)done;
      if (done) {
        env_reset(d, io->seed, env, gt + 1, st);
        if (io->ep_step) io->ep_step[e] = gt + 1;
        if (io->resample) {  // the next episode's teammate
          tm_id = episode_teammate(gt + 1);
          tm = tm_id >= 0 ? &pols[tm_id] : nullptr;
        }
      }
    }
    if (io->last_value) {
      env_obs(d, st, 0, o0.data());
      orc_mlp_forward(ego, obs_to_double(o0.data(), od).data(), z0.data());
      io->last_value[e] = has_value ? z0[K] : 0.0;
    }
    if (io->last_value_tm) {
      double v = 0.0;
      if (tm && tm->n_out > K) {
        env_obs(d, st, 1, o1.data());
        orc_mlp_forward(tm, obs_to_double(o1.data(), od).data(), z1.data());
        v = z1[K];
      }
      io->last_value_tm[e] = v;
    }
  });
  for (int64_t e = 0; e < N; ++e)
    if (status[e]) return status[e];
  return 0;
}

extern "C" int32_t orc_xplay(const orc_env_desc* d, const orc_mlp* pols, int32_t n_pols,
                             orc_xplay_io* io) {
  if (orc_check_desc(d) != 0) return -1;
  for (int i = 0; i < io->n_ego; ++i)
    if (io->ego_ids[i] < 0 || io->ego_ids[i] >= n_pols) return -4;
  const int min_id = d->kind == ORC_LBF ? -ORC_LBF_N_HEURISTICS : 0;  // heuristic teammates
  for (int j = 0; j < io->n_tm; ++j)
    if (io->tm_ids[j] < min_id || io->tm_ids[j] >= n_pols) return -4;
  const int od = orc_obs_dim(d), K = orc_n_actions(d);
  const int P = io->envs_per_pair;
  const int64_t n_all = (int64_t)io->n_ego * io->n_tm * P;
  const int64_t N = io->env_ids ? io->n_sel : n_all;  // rows
  for (int64_t r = 0; io->env_ids && r < N; ++r)
    if (io->env_ids[r] < 0 || io->env_ids[r] >= n_all) return -4;
  std::vector<float> returns(N, 0.0f);
  std::vector<int> status(N, 0);
  parallel_for(N, io->n_threads, [&](int64_t e) {
    const int64_t g = io->env_ids ? io->env_ids[e] : e;  // global env index
    const uint32_t env = (uint32_t)g;
    const int64_t pair = g / P;
    const int tm_id = io->tm_ids[pair % io->n_tm];
    const orc_mlp* pol[2] = {&pols[io->ego_ids[pair / io->n_tm]], tm_id >= 0 ? &pols[tm_id] : nullptr};
    orc_state st;
    env_reset(d, io->seed, env, (uint32_t)io->step0, &st);
    std::vector<uint8_t> o(od), legal(K);
    std::vector<double> z(std::max(pol[0]->n_out, pol[1] ? pol[1]->n_out : 1));
    int steps = 0;
    bool done = false;
    for (int s = 0; s < io->max_steps; ++s) {
      const int64_t i = (int64_t)s * N + e;
      if (io->actions) { io->actions[i * 2] = 255; io->actions[i * 2 + 1] = 255; }
      if (io->own_actions) { io->own_actions[i * 2] = 255; io->own_actions[i * 2 + 1] = 255; }
      if (io->margin) { io->margin[i * 2] = 2.0; io->margin[i * 2 + 1] = 2.0; }
      if (done) continue;
      const uint32_t gt = (uint32_t)(io->step0 + s);
      const int actor = acting_seat(d, &st);
      int act[2] = {0, 0};
      for (int seat = 0; seat < 2; ++seat) {
        if (actor >= 0 && seat != actor) continue;
        if (!pol[seat]) {  // heuristic teammate: its rule, no draw
          act[seat] = io->forced ? io->forced[i * 2 + seat]
                                 : orc_lbf_heuristic(d, (const orc_lbf_state*)&st, seat, -1 - tm_id);
          if (io->actions) io->actions[i * 2 + seat] = (uint8_t)act[seat];
          if (io->own_actions)
            io->own_actions[i * 2 + seat] = (uint8_t)orc_lbf_heuristic(d, (const orc_lbf_state*)&st, seat, -1 - tm_id);
          continue;
        }
        env_obs(d, &st, seat, o.data());
        env_legal(d, &st, legal.data());
        orc_mlp_forward(pol[seat], obs_to_double(o.data(), od).data(), z.data());
        if (io->logits)
          for (int k = 0; k < pol[seat]->n_out && k < io->logit_stride; ++k)
            io->logits[(i * 2 + seat) * io->logit_stride + k] = z[k];
        int own;
        double lp, mg;
        orc_sample(z.data(), legal.data(), K,
                   orc_u01(orc_draw(io->seed, env, gt, (uint32_t)(ORC_STREAM_ACT0 + seat), 0)), &own, &lp, &mg);
        act[seat] = io->forced ? io->forced[i * 2 + seat] : own;
        if (io->actions) io->actions[i * 2 + seat] = (uint8_t)act[seat];
        if (io->own_actions) io->own_actions[i * 2 + seat] = (uint8_t)own;
        if (io->margin) io->margin[i * 2 + seat] = mg;
      }
      float r[2], team;
      int dn = env_step(d, &st, act[0], act[1], r, &team);
      if (dn < 0) { status[e] = dn; done = true; continue; }
      steps += 1;
      done = dn != 0;
    }
    if (!done && turn_based(d)) status[e] = -2;  // Hanabi must terminate within the cap
    float ret = 0.0f;
    if (d->kind == ORC_LBF) ret = ((orc_lbf_state*)&st)->ret;
    if (d->kind == ORC_OVERCOOKED) ret = ((orc_oc_state*)&st)->ret;
    if (d->kind == ORC_HANABI) ret = ((orc_hanabi_state*)&st)->ret;
    if (d->kind == ORC_MINI_HANABI) ret = ((orc_mhanabi_state*)&st)->ret;
    returns[e] = ret;
    if (io->returns) io->returns[e] = ret;
    if (io->steps) io->steps[e] = steps;
  });
  if (io->matrix && !io->env_ids) {
    for (int64_t pair = 0; pair < (int64_t)io->n_ego * io->n_tm; ++pair) {
      double acc = 0.0;
      for (int k = 0; k < P; ++k) acc += (double)returns[pair * P + k];
      io->matrix[pair] = (float)(acc / (double)P);
    }
  }
  for (int64_t e = 0; e < N; ++e)
    if (status[e]) return status[e];
  return 0;
}
